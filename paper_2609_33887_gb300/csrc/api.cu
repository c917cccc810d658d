// Host side of the C ABI declared in include/bdcommit.h: argument checks,
// the workspace plan, TMA descriptors and the launch sequence of one commit
// step on the caller's stream.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <mutex>

#include "bdcommit.h"
#include "checks.h"
#include "kernels.h"
#include "trace.h"

namespace {

using bd::BandPlan;

constexpr int MAX_DEVICES = 64;
constexpr int64_t MAX_POSITIONS = int64_t(1) << 24;
constexpr int64_t MAX_VOCAB = int64_t(1) << 30;
constexpr int64_t MAX_DIM = int64_t(1) << 20;

struct DevCtx {
  bool ready = false;
  int sm_count = 0;
  int pairs = 0;               // CTA pairs of the pair kernel that fit on the device at once
  int quads = 0;               // ... clusters of two pairs
  uint32_t* status = nullptr;  // device status word (bd::DEV_* bits)
  void* ws = nullptr;          // library-owned workspace
  size_t ws_bytes = 0;
};

std::mutex g_mu;
DevCtx g_dev[MAX_DEVICES];
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

int device_ctx(DevCtx** out, int* dev_out = nullptr) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return BD_ERR_CUDA;
  if (dev < 0 || dev >= MAX_DEVICES) return BD_ERR_DEVICE;
  std::lock_guard<std::mutex> lk(g_mu);
  DevCtx& c = g_dev[dev];
  if (!c.ready) {
    int maj = 0, mnr = 0, sms = 0;
    if (cudaDeviceGetAttribute(&maj, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&mnr, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return BD_ERR_CUDA;
    if (maj != 10 || mnr != 3) return BD_ERR_DEVICE;  // the kernels are built for sm_103a only
    if (g_encode == nullptr) {
      cudaDriverEntryPointQueryResult q;
      void* fn = nullptr;
      if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
              cudaSuccess ||
          q != cudaDriverEntryPointSuccess || fn == nullptr)
        return BD_ERR_CUDA;
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    int pairs = 0, quads = 0;
    if (bd::lmhead_pair_max_clusters(sms, 1, &pairs) != cudaSuccess) return BD_ERR_CUDA;
    if (bd::lmhead_pair_max_clusters(sms, 2, &quads) != cudaSuccess) return BD_ERR_CUDA;
    if (cudaMalloc(&c.status, 256) != cudaSuccess) return BD_ERR_CUDA;
    if (cudaMemset(c.status, 0, 256) != cudaSuccess) return BD_ERR_CUDA;
    c.sm_count = sms;
    c.pairs = pairs;
    c.quads = quads;
    c.ready = true;
  }
  *out = &c;
  if (dev_out) *dev_out = dev;
  return BD_OK;
}

// ---------------------------------------------------------------- checks --
struct Call {
  int64_t P, d, V;
  int n_seq, n_slots, L, n_blocks, mask_id, T;
  int hdt, wdt;
  bool tc;          // tensor-core LM head
  bool pair;        // ... on CTA pairs (vocabulary on M), else the one-CTA kernel
  int64_t ldh, ldw;
  int64_t ldc;      // packed hidden rows (bf16), elements
  int64_t ldq;      // decoded e4m3 head (bf16), elements
  bool fused;       // pair kernel decodes an E4M3 / NVFP4 head itself (no bf16 copy)
  bool fp8_act = false;  // W8A8: token rows quantised to E4M3, kind::f8f6f4 MMAs on the E4M3 head
  bool split = false;    // W8A16 on the 8-bit path: bf16 rows as two E4M3 terms times the E4M3 head
};

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

int esize(int dt) { return dt == BD_F32 ? 4 : dt == BD_BF16 ? 2 : 1; }  // NVFP4: ld counts bytes

bool decoded_head(const Call& c) {
  return c.tc && !c.fused && !c.fp8_act && !c.split && (c.wdt == BD_E4M3 || c.wdt == BD_NVFP4);
}

// Decodes an FP8 or NVFP4 head into the bf16 workspace copy the tensor-core
// kernels read (both decodes are exact); wsrc / wld then describe that copy.
int decode_head(const Call& c, const bd_weight* weight, void* wq, int sm_count, cudaStream_t st, const void** wsrc,
                int64_t* wld) {
  const int V = static_cast<int>(c.V), d = static_cast<int>(c.d);
  cudaError_t e = c.wdt == BD_E4M3
                      ? bd::launch_dequant_e4m3(static_cast<const uint8_t*>(weight->data), c.ldw, V, d, wq, c.ldq,
                                                sm_count, st)
                      : bd::launch_dequant_nvfp4(static_cast<const uint8_t*>(weight->data), c.ldw,
                                                 weight->block_scale, weight->block_ld, V, d, wq, c.ldq, sm_count, st);
  *wsrc = wq;
  *wld = c.ldq;
  return e == cudaSuccess ? BD_OK : BD_ERR_CUDA;
}

int64_t round_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

int env_int(const char* name, int dflt, int lo, int hi);

// Checks shared by every entry point that runs the LM head: the head and the
// `rows` hidden rows, their dtypes and alignment, and the kernel choice. Fills
// the head fields of *c (d, V, dtypes, tc / pair, leading dimensions).
int check_head(const bd_hidden* h, const bd_weight* w, int64_t rows, int variant, Call* c) {
  if (w->vocab < 1 || w->vocab > MAX_VOCAB) return BD_ERR_SHAPE;
  if (w->dim < 1 || w->dim > MAX_DIM || h->cols != w->dim) return BD_ERR_SHAPE;
  if (h->ld < h->cols || w->ld < (w->dtype == BD_NVFP4 ? (w->dim + 1) / 2 : w->dim)) return BD_ERR_SHAPE;
  const int hdt = h->dtype, wdt = w->dtype;
  const bool combo_f32 = hdt == BD_F32 && wdt == BD_F32;
  const bool combo_bf16 = hdt == BD_BF16 && (wdt == BD_BF16 || wdt == BD_E4M3 || wdt == BD_NVFP4);
  if (!combo_f32 && !combo_bf16) return BD_ERR_DTYPE;
  const bool tc = variant >= 2 || (variant == 0 && combo_bf16);
  if (tc && !combo_bf16) return BD_ERR_DTYPE;
  if (rows > 0) {
    if (!h->data || !w->data) return BD_ERR_NULL;
    if (wdt == BD_E4M3 && !w->scale) return BD_ERR_NULL;
    if (wdt == BD_NVFP4 && !w->block_scale) return BD_ERR_NULL;
  }
  if (tc) {
    if (!aligned(h->data, 16) || (h->ld * 2) % 16 != 0) return BD_ERR_ALIGN;
    if (!aligned(w->data, 16) || (w->ld * esize(wdt)) % 16 != 0) return BD_ERR_ALIGN;
  } else {
    if (!aligned(h->data, esize(hdt)) || !aligned(w->data, esize(wdt))) return BD_ERR_ALIGN;
  }
  if (w->scale && (wdt == BD_E4M3 || wdt == BD_NVFP4) && !aligned(w->scale, 4)) return BD_ERR_ALIGN;
  if (wdt == BD_NVFP4 && w->block_ld < (w->dim + 15) / 16) return BD_ERR_SHAPE;
  c->d = w->dim;
  c->V = w->vocab;
  c->hdt = hdt;
  c->wdt = wdt;
  c->tc = tc;
  // automatic choice: the CTA-pair kernel (vocabulary on M, token dimension
  // padded only to a multiple of 32, 256 x 256 tiles per pair at large
  // windows) for bf16 heads at every size; heads decoded in the kernel by its
  // converter warps only while the window is small (at large windows the
  // one-CTA kernel on a decoded bf16 copy keeps the tensor pipe busier)
  const bool quant_head = wdt == BD_E4M3 || wdt == BD_NVFP4;
  c->pair = tc && (variant == 3 ||
                   (variant == 0 && (!quant_head || rows <= env_int("BD_PAIR_MAX_P", 8192, 0, 1 << 30))));
  c->ldh = h->ld;
  c->ldw = w->ld;
  c->ldc = round_up(c->d, 8);
  c->ldq = round_up(c->d, 8);
  // the pair kernel reads E4M3 / NVFP4 codes (and block scales) with TMA when
  // their rows start on 16-byte boundaries; otherwise the head is decoded to a
  // bf16 copy first
  c->fused = c->pair && (wdt == BD_E4M3 || wdt == BD_NVFP4) && env_int("BD_FUSED_DECODE", 1, 0, 1) != 0 &&
             aligned(w->data, 16) && w->ld % 16 == 0 && (wdt == BD_NVFP4 ? (w->dim + 1) / 2 : w->dim) >= 16 &&
             (wdt != BD_NVFP4 || (aligned(w->block_scale, 16) && w->block_ld % 16 == 0));
  return BD_OK;
}

int check_args(const bd_hidden* h, const bd_weight* w, const bd_mask_state* ms, const bd_tau_grid* tg,
               int variant, Call* c) {
  if (!h || !w || !ms || !tg) return BD_ERR_NULL;
  if (!tg->tau) return BD_ERR_TAU;
  if (tg->T < 1 || tg->T > 32) return BD_ERR_TAU;
  for (int k = 0; k < tg->T; ++k)
    if (std::isnan(tg->tau[k])) return BD_ERR_TAU;
  if (variant < 0 || variant > 3) return BD_ERR_ARG;
  if (ms->n_seq < 0 || ms->n_slots < 1 || ms->block_len < 1 || ms->block_len > 64) return BD_ERR_SHAPE;
  const int64_t n_blocks = int64_t(ms->n_seq) * ms->n_slots;
  const int64_t P = n_blocks * ms->block_len;
  if (P > MAX_POSITIONS) return BD_ERR_SHAPE;
  if (h->rows != P) return BD_ERR_SHAPE;
  if (const int rc = check_head(h, w, P, variant, c)) return rc;
  if (ms->mask_token_id < -1 || ms->mask_token_id >= w->vocab) return BD_ERR_ARG;
  if (ms->mask_token_id >= 0 && w->vocab < 2) return BD_ERR_SHAPE;  // nothing left to predict
  if (P > 0 && (!ms->pos_masked || !ms->block_flags)) return BD_ERR_NULL;
  // An E4M3 head on the commit step: the pair kernel multiplies its codes
  // directly on the 8-bit tensor path, with the bf16 rows packed as two E4M3
  // terms (needs 16-byte aligned code rows), at every window size.
  if (c->tc && w->dtype == BD_E4M3 && (variant == 0 || variant == 3) && env_int("BD_E4M3_SPLIT", 1, 0, 1) != 0 &&
      aligned(w->data, 16) && w->ld % 16 == 0 && w->dim >= 16) {
    c->pair = true;
    c->split = true;
    c->fused = false;
  }
  c->P = P;
  c->n_seq = ms->n_seq;
  c->n_slots = ms->n_slots;
  c->L = ms->block_len;
  c->n_blocks = static_cast<int>(n_blocks);
  c->mask_id = ms->mask_token_id;
  c->T = tg->T;
  return BD_OK;
}

// ------------------------------------------------------------- the plan --
int env_int(const char* name, int dflt, int lo, int hi) {
  const char* s = std::getenv(name);
  if (!s || !*s) return dflt;
  int v = std::atoi(s);
  return v < lo ? lo : v > hi ? hi : v;
}

// Bytes of one row of the LM head's token operand (the packed rows, or the
// caller's rows for the SIMT kernel).
int64_t row_operand_bytes(const Call& c) {
  if (!c.tc) return c.d * esize(c.hdt);
  if (c.fp8_act) return round_up(c.d, 16);
  if (c.split) return 2 * round_up(c.d, 16);
  return 2 * c.ldc;
}

// Bytes of one head row as the LM-head kernel reads it: the stored row for
// bf16 / E4M3 heads on the tensor-core kernels, the decoded bf16 copy where
// one is made, fp32 / stored rows for the SIMT kernel.
int64_t head_operand_bytes(const Call& c) {
  if (c.tc && !c.fused && !c.fp8_act && !c.split && (c.wdt == BD_E4M3 || c.wdt == BD_NVFP4)) return 2 * c.ldq;
  if (c.wdt == BD_NVFP4) return (c.d + 1) / 2;
  return c.d * esize(c.wdt);
}

BandPlan make_plan(const Call& c, int sm_count, int pairs, int quads) {
  BandPlan p{};
  p.mc = 1;
  if (c.pair) {
    p.BM = 0;  // token groups derived from N on the device
    p.BN = 256;
    p.G = pairs;
    p.cpu = 2;
    // heads staged by TMA as they are (bf16, the 8-bit paths): clusters of
    // two pairs that share every head tile where that measured faster than
    // single pairs on all SMs (clusters of 4 leave 8 of 152 SMs idle): windows
    // of at most two token groups, and windows whose packed rows exceed
    // 256 MiB (several bands: the head's L2 and DRAM re-reads dominate).
    // BD_PAIR_MC = 1 or 2 forces the choice.
    const int64_t rows_bytes = c.P * row_operand_bytes(c);
    const int mc_auto = (c.P <= 512 || rows_bytes > (int64_t(256) << 20)) ? 2 : 1;
    if (!c.fused && env_int("BD_PAIR_MC", mc_auto, 1, 2) == 2 && quads > 0) {
      p.mc = 2;
      p.G = quads;
      // the cluster's two pairs share head tiles (two token groups, one v-tile
      // at a time) or, with BD_PAIR_SHARE = 1, token rows (one token group,
      // two v-tiles at a time)
      if (env_int("BD_PAIR_SHARE", 0, 0, 1) == 1) {
        p.mc = 1;
        p.vc = 2;
      }
      // the pairs the clusters leave room for run as a concurrent spill
      // launch over the last v-tiles (BD_PAIR_SPILL = 0 / 1 forces it off /
      // on; BD_SPILL_PCT: a spill pair's time per tile against a cluster
      // pair's, in percent, which sets the vocabulary split)
      const int spare = pairs - 2 * quads;
      const int spill_auto = rows_bytes > (int64_t(256) << 20) ? 1 : 0;  // measured faster there only
      if (spare > 0 && env_int("BD_PAIR_SPILL", spill_auto, 0, 1) == 1) {
        p.G2 = spare;
        p.spill_pct = env_int("BD_SPILL_PCT", 100, 50, 400);
      }
    }
  } else if (c.tc) {
    p.BM = bd::TC_BM;
    p.BN = bd::TC_BN;
    p.G = sm_count;
    p.cpu = 1;
  } else {
    p.BM = bd::SIMT_BM;
    p.BN = bd::SIMT_BN;
    p.G = 2 * sm_count;
    p.cpu = 1;
  }
  // bands: GM derived on the device from the head and row bytes (0), or fixed
  p.GM = env_int("BD_PLAN_GM", 0, 0, 1 << 20);
  p.gv_fixed = env_int("BD_PLAN_GV", 0, 0, 1 << 20);
  p.rr = env_int("BD_PLAN_RR", 0, 0, 1);
  p.n_vt = static_cast<int>((c.V + p.BN - 1) / p.BN);
  p.vt_kb = static_cast<int>(std::max<int64_t>(1, int64_t(p.BN) * head_operand_bytes(c) / 1024));
  p.row_bytes = static_cast<int>(std::min<int64_t>(row_operand_bytes(c), int64_t(1) << 30));
  return p;
}

struct Layout {
  size_t hdr, idx, rowpos, pm, ps, pa, hc, tsc, wq, total;
};

Layout make_layout(const Call& c, const BandPlan& p) {
  Layout l{};
  size_t off = 0;
  auto take = [&off](size_t bytes, size_t align) {
    off = (off + align - 1) / align * align;
    size_t o = off;
    off += bytes;
    return o;
  };
  const size_t P = static_cast<size_t>(c.P);
  const size_t slots = static_cast<size_t>(plan_max_slots(p));
  l.hdr = take(256, 256);
  l.idx = take(4 * P, 256);
  l.rowpos = take(4 * P, 256);
  l.pm = take(4 * slots * P, 256);
  l.ps = take(4 * slots * P, 256);
  l.pa = take(4 * slots * P, 256);
  // bf16 rows, E4M3 rows (W8A8) or the two E4M3 terms of each row (W8A16 on the 8-bit path)
  const size_t hc_row = std::max<size_t>(2 * static_cast<size_t>(c.ldc), 2 * static_cast<size_t>(round_up(c.d, 16)));
  l.hc = c.tc ? take(hc_row * P, 1024) : 0;
  l.tsc = take(4 * P, 256);                                             // W8A8: per-row token scales
  l.wq = decoded_head(c) ? take(2 * static_cast<size_t>(c.ldq) * static_cast<size_t>(c.V), 1024) : 0;
  l.total = (off + 255) / 256 * 256;
  return l;
}

// Row stride (bytes) of the packed E4M3 token rows of the W8A8 variant.
int64_t ld_fp8_rows(const Call& c) { return round_up(c.d, 16); }

bool encode_bf16_2d(CUtensorMap* m, const void* base, int64_t inner, int64_t rows, int64_t ld_elems,
                    uint32_t box_inner, uint32_t box_rows) {
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld_elems * 2)};
  cuuint32_t box[2] = {box_inner, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// [rows, inner_bytes] bytes with row stride ld_bytes, boxes of box_inner bytes x box_rows.
bool encode_u8_2d(CUtensorMap* m, const void* base, int64_t inner_bytes, int64_t rows, int64_t ld_bytes,
                  uint32_t box_inner, uint32_t box_rows, bool swizzle128) {
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner_bytes), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld_bytes)};
  cuuint32_t box[2] = {box_inner, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// Records `ev` on `st`. Inside a stream capture a plain record would only add
// a dependency edge; the external flag makes it an event node of the graph,
// so replays still time the kernel.
cudaError_t record_event(void* ev, cudaStream_t st) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  cudaError_t e = cudaStreamIsCapturing(st, &cs);
  if (e != cudaSuccess) return e;
  if (cs == cudaStreamCaptureStatusActive)
    return cudaEventRecordWithFlags(static_cast<cudaEvent_t>(ev), st, cudaEventRecordExternal);
  return cudaEventRecord(static_cast<cudaEvent_t>(ev), st);
}

int cuda_status(cudaError_t e) {
  if (e == cudaSuccess) return BD_OK;
  if (e == cudaErrorNoKernelImageForDevice || e == cudaErrorInvalidDeviceFunction) return BD_ERR_DEVICE;
  return BD_ERR_CUDA;
}


// Partial-slot arrays of the LM head; t and x only on the verification path.
struct Partials {
  float* m;
  float* s;
  int* a;
  float* t;
  float* x;
};

// a1 + a2: decodes an FP8 / NVFP4 head if needed, builds the tensor maps over
// `rows` (the packed rows of the commit step, or the caller's rows for
// verification) and launches the LM-head kernel the plan chose, between the
// optional timing events. The SIMT kernel reads hidden->data through idx.
int launch_lmhead(const Call& c, const BandPlan& plan, const bd_hidden* hidden, const bd_weight* weight,
                  const void* rows, int64_t ld_rows, void* wq, const int* idx, const int* n_rows,
                  const int* draft_row, const Partials& part, uint32_t* status, int sm_count, void* ev_begin,
                  void* ev_end, cudaStream_t st, const float* tok_scale = nullptr) {
  const int P = static_cast<int>(c.P), V = static_cast<int>(c.V), d = static_cast<int>(c.d);
  const float* wscale = (c.wdt == BD_E4M3 || c.wdt == BD_NVFP4) ? weight->scale : nullptr;
  CUtensorMap tmA, tmB;
  bd::PairTokenMaps tmTok;
  bd::PairQuantMaps tmQ;
  std::memset(&tmB, 0, sizeof(tmB));
  std::memset(&tmQ, 0, sizeof(tmQ));
  const int hf = c.fp8_act ? bd::HF_W8A8
                 : c.split ? bd::HF_E4M3X2
                 : !c.fused ? bd::HF_BF16
                 : c.wdt == BD_NVFP4 ? bd::HF_NVFP4
                                     : bd::HF_E4M3;
  bd::PairTokenMaps tmLo;
  std::memset(&tmLo, 0, sizeof(tmLo));
  if (c.fused) {
    // codes: 128 bytes of a row per box (128 NVFP4 / E4M3 ... columns of d: 256 / 128)
    const int64_t code_bytes = c.wdt == BD_NVFP4 ? (c.d + 1) / 2 : c.d;
    if (!encode_u8_2d(&tmQ.codes, weight->data, code_bytes, c.V, c.ldw, 128, 128, true)) return BD_ERR_CUDA;
    if (c.wdt == BD_NVFP4 &&
        !encode_u8_2d(&tmQ.scales, weight->block_scale, (c.d + 15) / 16, c.V, weight->block_ld, 16, 128, false))
      return BD_ERR_CUDA;
  }
  if (c.tc) {
    const void* wsrc = weight->data;
    int64_t wld = c.ldw;
    if (decoded_head(c)) {
      const int rc = decode_head(c, weight, wq, sm_count, st, &wsrc, &wld);
      if (rc != BD_OK) return rc;
    }
    if (c.pair && (c.fp8_act || c.split)) {
      // W8A8 / two-term rows: E4M3 token rows and head rows, 128-byte
      // (128-column) boxes; the lo terms follow the hi terms' P rows
      for (int i = 0; i < 16; ++i) {
        if (!encode_u8_2d(&tmTok.m[i], rows, c.d, c.P, ld_rows, 128, 8 * (i + 1), true)) return BD_ERR_CUDA;
        if (c.split && !encode_u8_2d(&tmLo.m[i], static_cast<const uint8_t*>(rows) + c.P * ld_rows, c.d, c.P,
                                     ld_rows, 128, 8 * (i + 1), true))
          return BD_ERR_CUDA;
      }
      if (!encode_u8_2d(&tmB, weight->data, c.d, c.V, c.ldw, 128, 64, true)) return BD_ERR_CUDA;
    } else if (c.pair) {
      // token rows: one map per box height 8, 16, ..., 128 (half of a token group, or
      // the quarter a CTA loads for both pairs of a cluster that share token rows)
      for (int i = 0; i < 16; ++i)
        if (!encode_bf16_2d(&tmTok.m[i], rows, c.d, c.P, ld_rows, 64, 8 * (i + 1))) return BD_ERR_CUDA;
      if (!c.fused && !encode_bf16_2d(&tmB, wsrc, c.d, c.V, wld, 64, 64)) return BD_ERR_CUDA;
    } else {
      if (!encode_bf16_2d(&tmA, rows, c.d, c.P, ld_rows, bd::TC_BK, bd::TC_BM)) return BD_ERR_CUDA;
      if (!encode_bf16_2d(&tmB, wsrc, c.d, c.V, wld, bd::TC_BK, bd::TC_BN)) return BD_ERR_CUDA;
    }
  }
  if (ev_begin && record_event(ev_begin, st) != cudaSuccess) return BD_ERR_CUDA;
  int rc;
  if (c.tc) {
    bd::TcArgs a;
    a.n_rows = n_rows;
    a.wscale = wscale;
    a.V = V;
    a.d = d;
    a.P = P;
    a.mask_id = c.mask_id;
    a.plan = plan;
    a.part_m = part.m;
    a.part_s = part.s;
    a.part_a = part.a;
    a.status = status;
    a.draft_row = draft_row;
    a.part_t = part.t;
    a.part_x = part.x;
    a.tok_scale = tok_scale;
    a.l2_head = env_int("BD_L2_HEAD", bd::L2_EVICT_FIRST, 0, 2);
    a.l2_rows = env_int("BD_L2_ROWS", bd::L2_EVICT_LAST, 0, 2);
    rc = c.pair ? cuda_status(bd::launch_lmhead_pair(tmTok, tmB, c.fused ? &tmQ : nullptr, c.split ? &tmLo : nullptr,
                                                     hf, a, st))
                : cuda_status(bd::launch_lmhead_tc(tmA, tmB, a, env_int("BD_TC_STAGES", 4, 3, 4), st));
  } else {
    bd::SimtArgs a;
    a.hidden = hidden->data;
    a.ldh = c.ldh;
    a.hdtype = c.hdt;
    a.w = weight->data;
    a.ldw = c.ldw;
    a.wdtype = c.wdt;
    a.wbs = weight->block_scale;
    a.ldbs = weight->block_ld;
    a.wscale = wscale;
    a.idx = idx;
    a.n_rows = n_rows;
    a.V = V;
    a.d = d;
    a.P = P;
    a.mask_id = c.mask_id;
    a.plan = plan;
    a.part_m = part.m;
    a.part_s = part.s;
    a.part_a = part.a;
    a.draft_row = draft_row;
    a.part_t = part.t;
    a.part_x = part.x;
    rc = cuda_status(bd::launch_lmhead_simt(a, st));
  }
  if (rc != BD_OK) return rc;
  if (ev_end && record_event(ev_end, st) != cudaSuccess) return BD_ERR_CUDA;
  return BD_OK;
}

// Per-position partials of one vocabulary shard (bd_lmhead_partials).
struct EmitTarget {
  float* m;
  float* s;
  int32_t* a;
  int offset;  // global id of the shard's first vocabulary entry
};

// The launch sequence of one commit step (a0..a4) on `st`, working in `ws`
// laid out by `lay`; kernel timeouts are reported in `status`. With `emit`,
// the step ends after a3 with one merged partial per position (a head shard
// of a vocabulary-parallel split) instead of the commit.
int run_step(const Call& c, const BandPlan& plan, const Layout& lay, uint8_t* ws, uint32_t* status, int sm_count,
             const bd_hidden* hidden, const bd_weight* weight, const bd_mask_state* mask_state,
             const bd_tau_grid* tau_grid, int32_t* out_tokens, float* out_conf, uint32_t* out_commit,
             int32_t* out_counts, void* ev_begin, void* ev_end, cudaStream_t st, const EmitTarget* emit = nullptr) {
  int* n_rows = reinterpret_cast<int*>(ws + lay.hdr);
  int* idx = reinterpret_cast<int*>(ws + lay.idx);
  int* rowpos = reinterpret_cast<int*>(ws + lay.rowpos);
  float* pm = reinterpret_cast<float*>(ws + lay.pm);
  float* ps = reinterpret_cast<float*>(ws + lay.ps);
  int* pa = reinterpret_cast<int*>(ws + lay.pa);
  const int P = static_cast<int>(c.P), d = static_cast<int>(c.d);

  if (out_counts && !emit) {
    if (cudaMemsetAsync(out_counts, 0, sizeof(int32_t) * size_t(c.n_seq) * c.T, st) != cudaSuccess)
      return BD_ERR_CUDA;
  }

  // a0: compaction of the masked positions of active blocks (+ packing of their rows)
  // W8A8: the packed rows are quantised to E4M3 with one scale per row; a
  // head decoded inside the LM head: f16 rows scaled by a power of two per row
  const int row_format = c.fp8_act ? bd::ROWS_E4M3
                         : c.split ? bd::ROWS_E4M3X2
                         : c.fused ? bd::ROWS_F16_POW2
                                   : bd::ROWS_BF16;
  float* tsc = row_format != bd::ROWS_BF16 ? reinterpret_cast<float*>(ws + lay.tsc) : nullptr;
  const int64_t ld_rows = (c.fp8_act || c.split) ? ld_fp8_rows(c) : c.ldc;
  int rc = cuda_status(bd::launch_prep_rows(mask_state->pos_masked, mask_state->block_flags, P, c.L,
                                            c.tc ? hidden->data : nullptr, c.ldh, d, c.tc ? ws + lay.hc : nullptr,
                                            ld_rows, idx, rowpos, n_rows, sm_count, st, plan, tsc, row_format,
                                            status));
  if (rc != BD_OK) return rc;

  rc = launch_lmhead(c, plan, hidden, weight, ws + lay.hc, ld_rows, ws + lay.wq, idx, n_rows, nullptr,
                     Partials{pm, ps, pa, nullptr, nullptr}, status, sm_count, ev_begin, ev_end, st, tsc);
  if (rc != BD_OK) return rc;

  // a3 + a4: merge and the multi-threshold commit
  bd::CommitArgs ca;
  ca.pos_masked = mask_state->pos_masked;
  ca.block_flags = mask_state->block_flags;
  ca.rowpos = rowpos;
  ca.n_rows = n_rows;
  ca.plan = plan;
  ca.P = P;
  ca.part_m = pm;
  ca.part_s = ps;
  ca.part_a = pa;
  ca.n_blocks = c.n_blocks;
  ca.n_slots = c.n_slots;
  ca.block_len = c.L;
  std::memset(&ca.taus, 0, sizeof(ca.taus));
  for (int k = 0; k < c.T; ++k) ca.taus.tau[k] = tau_grid->tau[k];
  ca.taus.T = c.T;
  ca.out_tokens = out_tokens;
  ca.out_conf = out_conf;
  ca.out_commit = out_commit;
  ca.out_counts = out_counts;
  ca.status = status;
  if (emit) {
    ca.emit_m = emit->m;
    ca.emit_s = emit->s;
    ca.emit_a = emit->a;
    ca.vocab_offset = emit->offset;
    ca.out_counts = nullptr;
    return cuda_status(bd::launch_merge_commit(ca, st, bd::MERGE_EMIT));
  }
  return cuda_status(bd::launch_merge_commit(ca, st));
}

// check_args plus the bd_exec flags (W8A8 runs on the CTA-pair kernel with an
// E4M3 head read by TMA).
int check_exec_args(const bd_hidden* hidden, const bd_weight* weight, const bd_mask_state* mask_state,
                    const bd_tau_grid* tau_grid, int variant, int flags, Call* c) {
  if (flags & ~BD_EXEC_FP8_ACTIVATIONS) return BD_ERR_ARG;
  int rc = check_args(hidden, weight, mask_state, tau_grid, variant, c);
  if (rc != BD_OK) return rc;
  if (flags & BD_EXEC_FP8_ACTIVATIONS) {
    if (c->wdt != BD_E4M3 || c->hdt != BD_BF16 || !c->pair) return BD_ERR_ARG;
    if (!aligned(weight->data, 16) || weight->ld % 16 != 0 || c->d < 16) return BD_ERR_ALIGN;
    c->fp8_act = true;
    c->fused = false;
    c->split = false;
  }
  return BD_OK;
}

// Drops the cached device addresses of the allocation-free entry point's
// array (defined with it, below); the caller holds g_mu.
void forget_static_devices();
}  // namespace

extern "C" {

int bd_version(void) { return 100; }

const char* bd_status_string(int status) {
  switch (status) {
    case BD_OK: return "ok";
    case BD_ERR_NULL: return "a required pointer is NULL";
    case BD_ERR_SHAPE: return "sizes disagree or are out of range";
    case BD_ERR_DTYPE: return "unsupported dtype or dtype combination";
    case BD_ERR_ALIGN: return "pointer or row stride misaligned";
    case BD_ERR_TAU: return "invalid threshold grid (T outside 1..32, NULL or NaN)";
    case BD_ERR_WORKSPACE: return "workspace too small";
    case BD_ERR_CUDA: return "a CUDA call or kernel launch failed";
    case BD_ERR_TIMEOUT: return "a bounded device-side wait gave up";
    case BD_ERR_DEVICE: return "the current device cannot run this library (needs sm_103)";
    case BD_ERR_ARG: return "invalid argument";
    case BD_ERR_BOUNDS: return "a device-side index check failed (bounds-checked build)";
    default: return "unknown status";
  }
}

size_t bd_workspace_size(const bd_hidden* hidden, const bd_weight* weight, const bd_mask_state* mask_state,
                         const bd_tau_grid* tau_grid) {
  Call c;
  if (check_args(hidden, weight, mask_state, tau_grid, 0, &c) != BD_OK) return 0;
  DevCtx* ctx = nullptr;
  if (device_ctx(&ctx) != BD_OK) return 0;
  return make_layout(c, make_plan(c, ctx->sm_count, ctx->pairs, ctx->quads)).total;
}

int bd_plan_header(const bd_hidden* hidden, const bd_weight* weight, const bd_mask_state* mask_state,
                   const bd_tau_grid* tau_grid, const bd_exec* exec, int32_t n_rows, int32_t* out, int32_t n_out) {
  if (!out || n_out < 0 || n_rows < 0) return BD_ERR_ARG;
  Call c;
  const int rc = check_exec_args(hidden, weight, mask_state, tau_grid, exec ? exec->variant : 0,
                                 exec ? exec->flags : 0, &c);
  if (rc != BD_OK) return rc;
  if (n_rows > c.P) return BD_ERR_ARG;
  DevCtx* ctx = nullptr;
  if (device_ctx(&ctx) != BD_OK) return BD_ERR_DEVICE;
  const BandPlan plan = make_plan(c, ctx->sm_count, ctx->pairs, ctx->quads);
  int hdr[bd::HDR_WORDS] = {0};
  bd::plan_header(plan, n_rows, hdr);
  for (int i = 0; i < n_out && i < bd::HDR_WORDS; ++i) out[i] = hdr[i];
  return bd::HDR_WORDS;
}

int bd_step_kernels(const bd_hidden* hidden, const bd_weight* weight, const bd_mask_state* mask_state,
                    const bd_tau_grid* tau_grid, const bd_exec* exec) {
  Call c;
  const int rc = check_exec_args(hidden, weight, mask_state, tau_grid, exec ? exec->variant : 0,
                                 exec ? exec->flags : 0, &c);
  if (rc != BD_OK) return rc;
  if (c.P == 0) return 0;
  DevCtx* ctx = nullptr;
  if (device_ctx(&ctx) != BD_OK) return BD_ERR_DEVICE;
  const BandPlan plan = make_plan(c, ctx->sm_count, ctx->pairs, ctx->quads);
  // compaction + row packing, the head decode where a bf16 copy is made, the
  // LM head (two launches with spill pairs), merge + commit
  return 1 + (c.tc && decoded_head(c) ? 1 : 0) + (c.pair && plan.G2 > 0 ? 2 : 1) + 1;
}

int bd_commit_step_ex(const bd_hidden* hidden, const bd_weight* weight, const bd_mask_state* mask_state,
                      const bd_tau_grid* tau_grid, int32_t* out_tokens, float* out_conf, uint32_t* out_commit,
                      const bd_exec* exec) {
  bd::TraceRange trace("bd_commit_step");
  const int variant = exec ? exec->variant : 0;
  const int flags = exec ? exec->flags : 0;
  Call c;
  int rc = check_exec_args(hidden, weight, mask_state, tau_grid, variant, flags, &c);
  if (rc != BD_OK) return rc;
  if (c.P == 0) return BD_OK;
  if (!out_tokens || !out_conf || !out_commit) return BD_ERR_NULL;
  if (!aligned(out_tokens, 4) || !aligned(out_conf, 4) || !aligned(out_commit, 4)) return BD_ERR_ALIGN;
  if (exec && exec->out_counts && !aligned(exec->out_counts, 4)) return BD_ERR_ALIGN;
  if (exec && exec->workspace && !aligned(exec->workspace, 256)) return BD_ERR_ALIGN;

  DevCtx* ctx = nullptr;
  rc = device_ctx(&ctx);
  if (rc != BD_OK) return rc;
  const BandPlan plan = make_plan(c, ctx->sm_count, ctx->pairs, ctx->quads);
  const Layout lay = make_layout(c, plan);

  uint8_t* ws = nullptr;
  if (exec && exec->workspace) {
    if (exec->workspace_bytes < lay.total) return BD_ERR_WORKSPACE;
    ws = static_cast<uint8_t*>(exec->workspace);
  } else {
    std::lock_guard<std::mutex> lk(g_mu);
    if (ctx->ws_bytes < lay.total) {
      if (ctx->ws) cudaFree(ctx->ws);  // synchronises the device: no call can still use it
      ctx->ws = nullptr;
      ctx->ws_bytes = 0;
      if (cudaMalloc(&ctx->ws, lay.total) != cudaSuccess) return BD_ERR_CUDA;
      ctx->ws_bytes = lay.total;
    }
    ws = static_cast<uint8_t*>(ctx->ws);
  }

  cudaStream_t st = static_cast<cudaStream_t>(exec ? exec->stream : nullptr);
  return run_step(c, plan, lay, ws, ctx->status, ctx->sm_count, hidden, weight, mask_state, tau_grid, out_tokens,
                  out_conf, out_commit, exec ? exec->out_counts : nullptr, exec ? exec->lmhead_event_begin : nullptr,
                  exec ? exec->lmhead_event_end : nullptr, st);
}

int bd_commit_step(const bd_hidden* hidden, const bd_weight* weight, const bd_mask_state* mask_state,
                   const bd_tau_grid* tau_grid, int32_t* out_tokens, float* out_conf, uint32_t* out_commit) {
  return bd_commit_step_ex(hidden, weight, mask_state, tau_grid, out_tokens, out_conf, out_commit, nullptr);
}

int bd_lmhead_partials(const bd_hidden* hidden, const bd_weight* shard, int64_t vocab_offset,
                       const bd_mask_state* mask_state, const bd_partials* out, const bd_exec* exec) {
  bd::TraceRange trace("bd_lmhead_partials");
  if (!hidden || !shard || !mask_state || !out) return BD_ERR_NULL;
  if (vocab_offset < 0 || vocab_offset + shard->vocab > MAX_VOCAB) return BD_ERR_ARG;
  if (mask_state->mask_token_id < -1) return BD_ERR_ARG;
  if (exec && (exec->flags != 0 || exec->out_counts || exec->lmhead_event_begin || exec->lmhead_event_end))
    return BD_ERR_ARG;
  // the mask token, a global id, is suppressed by the shard that holds it
  bd_mask_state local = *mask_state;
  const int64_t mid = mask_state->mask_token_id;
  local.mask_token_id = (mid >= vocab_offset && mid < vocab_offset + shard->vocab)
                            ? static_cast<int32_t>(mid - vocab_offset) : -1;
  const float tau1 = 0.5f;  // the shared checks want a grid; the shard step commits nothing
  const bd_tau_grid tg{&tau1, 1};
  Call c;
  int rc = check_args(hidden, shard, &local, &tg, exec ? exec->variant : 0, &c);
  if (rc != BD_OK) return rc;
  if (c.P == 0) return BD_OK;
  if (!out->m || !out->s || !out->a) return BD_ERR_NULL;
  if (!aligned(out->m, 4) || !aligned(out->s, 4) || !aligned(out->a, 4)) return BD_ERR_ALIGN;
  if (exec && exec->workspace && !aligned(exec->workspace, 256)) return BD_ERR_ALIGN;
  DevCtx* ctx = nullptr;
  rc = device_ctx(&ctx);
  if (rc != BD_OK) return rc;
  const BandPlan plan = make_plan(c, ctx->sm_count, ctx->pairs, ctx->quads);
  const Layout lay = make_layout(c, plan);
  uint8_t* ws = nullptr;
  if (exec && exec->workspace) {
    if (exec->workspace_bytes < lay.total) return BD_ERR_WORKSPACE;
    ws = static_cast<uint8_t*>(exec->workspace);
  } else {
    std::lock_guard<std::mutex> lk(g_mu);
    if (ctx->ws_bytes < lay.total) {
      if (ctx->ws) cudaFree(ctx->ws);  // synchronises the device: no call can still use it
      ctx->ws = nullptr;
      ctx->ws_bytes = 0;
      if (cudaMalloc(&ctx->ws, lay.total) != cudaSuccess) return BD_ERR_CUDA;
      ctx->ws_bytes = lay.total;
    }
    ws = static_cast<uint8_t*>(ctx->ws);
  }
  const EmitTarget emit{out->m, out->s, out->a, static_cast<int>(vocab_offset)};
  cudaStream_t st = static_cast<cudaStream_t>(exec ? exec->stream : nullptr);
  return run_step(c, plan, lay, ws, ctx->status, ctx->sm_count, hidden, shard, &local, &tg, nullptr, nullptr,
                  nullptr, nullptr, nullptr, nullptr, st, &emit);
}

int bd_merge_commit(const bd_partials* gathered, int32_t n_parts, const bd_mask_state* mask_state,
                    const bd_tau_grid* tau_grid, int32_t* out_tokens, float* out_conf, uint32_t* out_commit,
                    const bd_exec* exec) {
  bd::TraceRange trace("bd_merge_commit");
  if (!gathered || !mask_state || !tau_grid) return BD_ERR_NULL;
  if (n_parts < 1 || n_parts > 4096) return BD_ERR_ARG;
  if (!tau_grid->tau) return BD_ERR_TAU;
  if (tau_grid->T < 1 || tau_grid->T > 32) return BD_ERR_TAU;
  for (int k = 0; k < tau_grid->T; ++k)
    if (std::isnan(tau_grid->tau[k])) return BD_ERR_TAU;
  if (exec && (exec->flags != 0 || exec->workspace || exec->lmhead_event_begin || exec->lmhead_event_end))
    return BD_ERR_ARG;
  const bd_mask_state* ms = mask_state;
  if (ms->n_seq < 0 || ms->n_slots < 1 || ms->block_len < 1 || ms->block_len > 64) return BD_ERR_SHAPE;
  const int64_t n_blocks = int64_t(ms->n_seq) * ms->n_slots;
  const int64_t P = n_blocks * ms->block_len;
  if (P > MAX_POSITIONS || P * n_parts > (int64_t(1) << 31)) return BD_ERR_SHAPE;
  if (P == 0) return BD_OK;
  if (!ms->pos_masked || !ms->block_flags) return BD_ERR_NULL;
  if (!gathered->m || !gathered->s || !gathered->a || !out_tokens || !out_conf || !out_commit) return BD_ERR_NULL;
  if (!aligned(gathered->m, 4) || !aligned(gathered->s, 4) || !aligned(gathered->a, 4) || !aligned(out_tokens, 4) ||
      !aligned(out_conf, 4) || !aligned(out_commit, 4))
    return BD_ERR_ALIGN;
  if (exec && exec->out_counts && !aligned(exec->out_counts, 4)) return BD_ERR_ALIGN;
  DevCtx* ctx = nullptr;
  const int rc = device_ctx(&ctx);
  if (rc != BD_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(exec ? exec->stream : nullptr);
  int32_t* out_counts = exec ? exec->out_counts : nullptr;
  if (out_counts &&
      cudaMemsetAsync(out_counts, 0, sizeof(int32_t) * size_t(ms->n_seq) * tau_grid->T, st) != cudaSuccess)
    return BD_ERR_CUDA;
  bd::CommitArgs ca;
  std::memset(&ca.plan, 0, sizeof(ca.plan));
  ca.pos_masked = ms->pos_masked;
  ca.block_flags = ms->block_flags;
  ca.rowpos = nullptr;
  ca.n_rows = nullptr;
  ca.P = static_cast<int>(P);
  ca.part_m = gathered->m;
  ca.part_s = gathered->s;
  ca.part_a = gathered->a;
  ca.n_blocks = static_cast<int>(n_blocks);
  ca.n_slots = ms->n_slots;
  ca.block_len = ms->block_len;
  std::memset(&ca.taus, 0, sizeof(ca.taus));
  for (int k = 0; k < tau_grid->T; ++k) ca.taus.tau[k] = tau_grid->tau[k];
  ca.taus.T = tau_grid->T;
  ca.out_tokens = out_tokens;
  ca.out_conf = out_conf;
  ca.out_commit = out_commit;
  ca.out_counts = out_counts;
  ca.status = ctx->status;
  ca.n_parts = n_parts;
  return cuda_status(bd::launch_merge_commit(ca, st, bd::MERGE_GATHERED));
}

int bd_get_device_status(void* stream) {
  DevCtx* ctx = nullptr;
  int rc = device_ctx(&ctx);
  if (rc != BD_OK) return rc;
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return BD_ERR_CUDA;
  uint32_t word = 0;
  if (cudaMemcpy(&word, ctx->status, sizeof(word), cudaMemcpyDeviceToHost) != cudaSuccess) return BD_ERR_CUDA;
  if (word != 0 && cudaMemset(ctx->status, 0, sizeof(word)) != cudaSuccess) return BD_ERR_CUDA;
  if (word & bd::DEV_TIMEOUT) return BD_ERR_TIMEOUT;
  if (word & bd::DEV_BAD_LAUNCH) return BD_ERR_CUDA;
  if (word & bd::DEV_BOUNDS) return BD_ERR_BOUNDS;
  return BD_OK;
}

int bd_selftest_timeout(void* stream) {
  DevCtx* ctx = nullptr;
  int rc = device_ctx(&ctx);
  if (rc != BD_OK) return rc;
  return cuda_status(bd::launch_timeout_selftest(ctx->status, static_cast<cudaStream_t>(stream)));
}

int bd_shutdown(void) {
  std::lock_guard<std::mutex> lk(g_mu);
  int cur = 0;
  if (cudaGetDevice(&cur) != cudaSuccess) return BD_ERR_CUDA;
  int rc = BD_OK;
  for (int dev = 0; dev < MAX_DEVICES; ++dev) {
    DevCtx& c = g_dev[dev];
    if (!c.ready) continue;
    if (cudaSetDevice(dev) != cudaSuccess) {
      rc = BD_ERR_CUDA;
      continue;
    }
    if (c.ws) cudaFree(c.ws);
    if (c.status) cudaFree(c.status);
    c = DevCtx();
  }
  cudaSetDevice(cur);
  forget_static_devices();
  return rc;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// bd_commit_step_static: the commit step for callers that cannot allocate.
// Its workspace is the file-scope device array below; nothing here calls
// cudaMalloc, cudaFree or any allocating routine.
// ---------------------------------------------------------------------------
namespace {

static __device__ __align__(256) uint8_t g_static_scratch[BD_STATIC_SCRATCH_BYTES];

// Offset, inside the workspace header, of the word the LM-head kernel reports
// a timed-out wait in (the compacted row count sits at offset 0).
constexpr size_t STATIC_STATUS_OFFSET = 128;

struct StaticCtx {
  bool ready = false;
  int sm_count = 0;
  int pairs = 0;
  int quads = 0;
  uint8_t* scratch = nullptr;  // device address of g_static_scratch on this device
};
StaticCtx g_static[MAX_DEVICES];

// After bd_shutdown (and possibly a device reset) the module may be loaded
// again at another address: the next call resolves it anew.
void forget_static_devices() {
  for (int dev = 0; dev < MAX_DEVICES; ++dev) g_static[dev] = StaticCtx();
}

// Once per device, with that device current: checks the device, fetches the
// tensor-map encoder and resolves the device address of g_static_scratch.
// (In host code the array's name is only a host-side stand-in, so kernels
// must be given the resolved address.)
int static_ctx(StaticCtx** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return BD_ERR_CUDA;
  if (dev < 0 || dev >= MAX_DEVICES) return BD_ERR_DEVICE;
  std::lock_guard<std::mutex> lk(g_mu);
  StaticCtx& s = g_static[dev];
  if (!s.ready) {
    int maj = 0, mnr = 0, sms = 0;
    if (cudaDeviceGetAttribute(&maj, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&mnr, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return BD_ERR_CUDA;
    if (maj != 10 || mnr != 3) return BD_ERR_DEVICE;
    if (g_encode == nullptr) {
      cudaDriverEntryPointQueryResult q;
      void* fn = nullptr;
      if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
              cudaSuccess ||
          q != cudaDriverEntryPointSuccess || fn == nullptr)
        return BD_ERR_CUDA;
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    int pairs = 0, quads = 0;
    if (bd::lmhead_pair_max_clusters(sms, 1, &pairs) != cudaSuccess) return BD_ERR_CUDA;
    if (bd::lmhead_pair_max_clusters(sms, 2, &quads) != cudaSuccess) return BD_ERR_CUDA;
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch);
    if (e != cudaSuccess || p == nullptr) return e == cudaSuccess ? BD_ERR_CUDA : cuda_status(e);
    s.scratch = static_cast<uint8_t*>(p);
    // the status word starts clear; afterwards only bd_static_device_status clears it
    if (cudaMemset(s.scratch + STATIC_STATUS_OFFSET, 0, sizeof(uint32_t)) != cudaSuccess) return BD_ERR_CUDA;
    s.sm_count = sms;
    s.pairs = pairs;
    s.quads = quads;
    s.ready = true;
  }
  *out = &s;
  return BD_OK;
}

}  // namespace

extern "C" int bd_commit_step_static(const bd_hidden* hidden, const bd_weight* weight,
                                     const bd_mask_state* mask_state, const bd_tau_grid* tau_grid,
                                     int32_t* out_tokens, float* out_conf, uint32_t* out_commit, void* stream) {
  bd::TraceRange trace("bd_commit_step_static");
  Call c;
  int rc = check_args(hidden, weight, mask_state, tau_grid, 0, &c);
  if (rc != BD_OK) return rc;
  if (c.P == 0) return BD_OK;
  if (!out_tokens || !out_conf || !out_commit) return BD_ERR_NULL;
  if (!aligned(out_tokens, 4) || !aligned(out_conf, 4) || !aligned(out_commit, 4)) return BD_ERR_ALIGN;

  StaticCtx* sctx = nullptr;
  rc = static_ctx(&sctx);
  if (rc != BD_OK) return rc;
  const BandPlan plan = make_plan(c, sctx->sm_count, sctx->pairs, sctx->quads);
  const Layout lay = make_layout(c, plan);
  if (lay.total > BD_STATIC_SCRATCH_BYTES) return BD_ERR_WORKSPACE;

  uint8_t* ws = sctx->scratch;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // The array keeps the previous call's contents: everything the step reads
  // it writes first, except the status word, which is cleared once at set-up
  // and then by bd_static_device_status (a failure stays recorded until read).
  uint32_t* status = reinterpret_cast<uint32_t*>(ws + lay.hdr + STATIC_STATUS_OFFSET);
  return run_step(c, plan, lay, ws, status, sctx->sm_count, hidden, weight, mask_state, tau_grid, out_tokens,
                  out_conf, out_commit, nullptr, nullptr, nullptr, st);
}

namespace {
int static_status_of(uint32_t word) {
  if (word & bd::DEV_TIMEOUT) return BD_ERR_TIMEOUT;
  if (word & bd::DEV_BAD_LAUNCH) return BD_ERR_CUDA;
  if (word & bd::DEV_BOUNDS) return BD_ERR_BOUNDS;
  return BD_OK;
}
}  // namespace

extern "C" int bd_static_device_status(void* stream) {
  StaticCtx* sctx = nullptr;
  const int rc = static_ctx(&sctx);
  if (rc != BD_OK) return rc;
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return BD_ERR_CUDA;
  uint32_t word = 0;
  uint8_t* at = sctx->scratch + STATIC_STATUS_OFFSET;
  if (cudaMemcpy(&word, at, sizeof(word), cudaMemcpyDeviceToHost) != cudaSuccess) return BD_ERR_CUDA;
  if (word != 0 && cudaMemset(at, 0, sizeof(word)) != cudaSuccess) return BD_ERR_CUDA;
  return static_status_of(word);
}

extern "C" int bd_static_selftest_timeout(void* stream) {
  StaticCtx* sctx = nullptr;
  const int rc = static_ctx(&sctx);
  if (rc != BD_OK) return rc;
  return cuda_status(bd::launch_timeout_selftest(reinterpret_cast<uint32_t*>(sctx->scratch + STATIC_STATUS_OFFSET),
                                                 static_cast<cudaStream_t>(stream)));
}

// ---------------------------------------------------------------------------
// bd_verify_step: speculative-decoding verification on the same LM head
// (typical-acceptance and lossless-reference appendices).
// ---------------------------------------------------------------------------
namespace {

struct VerifyCall {
  Call c;  // P = rows, T = E
  int n_req, n_draft;
};

int check_verify(const bd_hidden* h, const bd_weight* w, const bd_draft* dr, const bd_eps_grid* eg, int variant,
                 VerifyCall* vc) {
  if (!h || !w || !dr || !eg) return BD_ERR_NULL;
  if (!eg->eps || eg->E < 1 || eg->E > 31) return BD_ERR_TAU;
  for (int k = 0; k < eg->E; ++k)
    if (!(eg->eps[k] > 0.f && eg->eps[k] <= 1.f)) return BD_ERR_TAU;  // NaN fails too
  if (variant < 0 || variant > 3) return BD_ERR_ARG;
  if (dr->n_req < 0 || dr->n_draft < 1 || dr->n_draft > 32) return BD_ERR_SHAPE;
  const int64_t R = int64_t(dr->n_req) * (dr->n_draft + 1);
  if (R > MAX_POSITIONS || h->rows != R) return BD_ERR_SHAPE;
  Call& c = vc->c;
  c = Call{};
  if (const int rc = check_head(h, w, R, variant, &c)) return rc;
  if (R > 0 && !dr->draft) return BD_ERR_NULL;
  if (R > 0 && !aligned(dr->draft, 4)) return BD_ERR_ALIGN;
  c.P = R;
  c.n_seq = dr->n_req;
  c.n_slots = 1;
  c.L = dr->n_draft + 1;
  c.n_blocks = dr->n_req;
  c.mask_id = -1;  // the target's full distribution
  c.T = eg->E;
  c.ldc = h->ld;  // the rows are read in place
  vc->n_req = dr->n_req;
  vc->n_draft = dr->n_draft;
  return BD_OK;
}

struct VerifyLayout {
  size_t hdr, idx, draft_row, pm, ps, pa, pt, px, wq, total;
};

VerifyLayout make_verify_layout(const Call& c, const BandPlan& p) {
  VerifyLayout l{};
  size_t off = 0;
  auto take = [&off](size_t bytes, size_t align) {
    off = (off + align - 1) / align * align;
    size_t o = off;
    off += bytes;
    return o;
  };
  const size_t R = static_cast<size_t>(c.P);
  const size_t slots = static_cast<size_t>(plan_max_slots(p));
  l.hdr = take(256, 256);
  l.idx = take(4 * R, 256);
  l.draft_row = take(4 * R, 256);
  l.pm = take(4 * slots * R, 256);
  l.ps = take(4 * slots * R, 256);
  l.pa = take(4 * slots * R, 256);
  l.pt = take(4 * slots * R, 256);
  l.px = take(4 * slots * R, 256);
  l.wq = decoded_head(c) ? take(2 * static_cast<size_t>(c.ldq) * static_cast<size_t>(c.V), 1024) : 0;
  l.total = (off + 255) / 256 * 256;
  return l;
}

int run_verify(const VerifyCall& vc, const BandPlan& plan, const VerifyLayout& lay, uint8_t* ws, uint32_t* status,
               int sm_count, const bd_hidden* hidden, const bd_weight* weight, const bd_draft* draft,
               const bd_eps_grid* eps, int32_t* out_tokens, float* out_p_draft, float* out_entropy,
               uint32_t* out_accept, int32_t* out_accepted, void* ev_begin, void* ev_end, cudaStream_t st) {
  const Call& c = vc.c;
  int* n_rows = reinterpret_cast<int*>(ws + lay.hdr);
  int* idx = reinterpret_cast<int*>(ws + lay.idx);
  int* draft_row = reinterpret_cast<int*>(ws + lay.draft_row);
  float* pm = reinterpret_cast<float*>(ws + lay.pm);
  float* ps = reinterpret_cast<float*>(ws + lay.ps);
  int* pa = reinterpret_cast<int*>(ws + lay.pa);
  float* pt = reinterpret_cast<float*>(ws + lay.pt);
  float* px = reinterpret_cast<float*>(ws + lay.px);
  const int R = static_cast<int>(c.P);

  int rc = cuda_status(bd::launch_prep_verify(draft->draft, vc.n_req, vc.n_draft, idx, draft_row, n_rows, plan, st));
  if (rc != BD_OK) return rc;

  rc = launch_lmhead(c, plan, hidden, weight, hidden->data, c.ldh, ws + lay.wq, idx, n_rows, draft_row,
                     Partials{pm, ps, pa, pt, px}, status, sm_count, ev_begin, ev_end, st);
  if (rc != BD_OK) return rc;

  bd::VerifyArgs va;
  va.draft_row = draft_row;
  va.n_rows = n_rows;
  va.plan = plan;
  va.P = R;
  va.part_m = pm;
  va.part_s = ps;
  va.part_a = pa;
  va.part_t = pt;
  va.part_x = px;
  va.n_req = vc.n_req;
  va.n_draft = vc.n_draft;
  va.E = eps->E;
  std::memset(va.eps, 0, sizeof(va.eps));
  std::memset(va.sqrt_eps, 0, sizeof(va.sqrt_eps));
  for (int k = 0; k < eps->E; ++k) {
    va.eps[k] = eps->eps[k];
    va.sqrt_eps[k] = static_cast<float>(std::sqrt(static_cast<double>(eps->eps[k])));
  }
  va.out_tokens = out_tokens;
  va.out_p_draft = out_p_draft;
  va.out_entropy = out_entropy;
  va.out_accept = out_accept;
  va.out_accepted = out_accepted;
  return cuda_status(bd::launch_merge_verify(va, st));
}

}  // namespace

extern "C" {

size_t bd_verify_workspace_size(const bd_hidden* hidden, const bd_weight* weight, const bd_draft* draft,
                                const bd_eps_grid* eps) {
  VerifyCall vc;
  if (check_verify(hidden, weight, draft, eps, 0, &vc) != BD_OK) return 0;
  DevCtx* ctx = nullptr;
  if (device_ctx(&ctx) != BD_OK) return 0;
  return make_verify_layout(vc.c, make_plan(vc.c, ctx->sm_count, ctx->pairs, ctx->quads)).total;
}

int bd_verify_step(const bd_hidden* hidden, const bd_weight* weight, const bd_draft* draft, const bd_eps_grid* eps,
                   int32_t* out_tokens, float* out_p_draft, float* out_entropy, uint32_t* out_accept,
                   int32_t* out_accepted, const bd_exec* exec) {
  bd::TraceRange trace("bd_verify_step");
  const int variant = exec ? exec->variant : 0;
  if (exec && (exec->flags != 0 || exec->out_counts != nullptr)) return BD_ERR_ARG;
  VerifyCall vc;
  int rc = check_verify(hidden, weight, draft, eps, variant, &vc);
  if (rc != BD_OK) return rc;
  if (vc.c.P == 0) return BD_OK;
  if (!out_tokens || !out_p_draft || !out_entropy || !out_accept || !out_accepted) return BD_ERR_NULL;
  if (!aligned(out_tokens, 4) || !aligned(out_p_draft, 4) || !aligned(out_entropy, 4) || !aligned(out_accept, 4) ||
      !aligned(out_accepted, 4))
    return BD_ERR_ALIGN;
  if (exec && exec->workspace && !aligned(exec->workspace, 256)) return BD_ERR_ALIGN;

  DevCtx* ctx = nullptr;
  rc = device_ctx(&ctx);
  if (rc != BD_OK) return rc;
  const BandPlan plan = make_plan(vc.c, ctx->sm_count, ctx->pairs, ctx->quads);
  const VerifyLayout lay = make_verify_layout(vc.c, plan);
  uint8_t* ws = nullptr;
  if (exec && exec->workspace) {
    if (exec->workspace_bytes < lay.total) return BD_ERR_WORKSPACE;
    ws = static_cast<uint8_t*>(exec->workspace);
  } else {
    std::lock_guard<std::mutex> lk(g_mu);
    if (ctx->ws_bytes < lay.total) {
      if (ctx->ws) cudaFree(ctx->ws);  // synchronises the device: no call can still use it
      ctx->ws = nullptr;
      ctx->ws_bytes = 0;
      if (cudaMalloc(&ctx->ws, lay.total) != cudaSuccess) return BD_ERR_CUDA;
      ctx->ws_bytes = lay.total;
    }
    ws = static_cast<uint8_t*>(ctx->ws);
  }
  cudaStream_t st = static_cast<cudaStream_t>(exec ? exec->stream : nullptr);
  return run_verify(vc, plan, lay, ws, ctx->status, ctx->sm_count, hidden, weight, draft, eps, out_tokens,
                    out_p_draft, out_entropy, out_accept, out_accepted, exec ? exec->lmhead_event_begin : nullptr,
                    exec ? exec->lmhead_event_end : nullptr, st);
}

}  // extern "C"
