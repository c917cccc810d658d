// LM-head projection + mask-suppressed softmax statistics on a CTA pair
// (tcgen05 cta_group::2) with the vocabulary on the MMA M side (App. B.1: the
// LM head and the softmax the engine commits from).
//
// A pair of CTAs (a cluster of 2) computes, per v-tile, logits of 256
// vocabulary rows (128 in each CTA's tensor memory, one row per TMEM lane)
// against a group of NT <= 256 token rows (NT columns): one
// tcgen05.mma.cta_group::2 M=256 N=NT K=16 per 16 columns of d, issued by one
// thread of the even CTA; each CTA stages its own 128 head rows and its half of
// the token rows. A pipeline stage covers 128 columns of d (eight MMAs per
// barrier wait and commit, which keeps the single issuing thread ahead of the
// tensor pipe even at NT = 160), i.e. 32 KB + NT x 128 B per CTA; the number of
// stages follows from NT (4 at NT = 160, 3 at NT = 256). Token tiles are loaded
// with boxes of exactly NT/2 rows (one tensor map per height).
// Compared with tokens on M, the token dimension is padded only to a multiple
// of 32 (e.g. 294 rows -> 2 groups of 160, not 3 m-tiles of 128).
//
// The softmax reduction runs over vocabulary rows, i.e. over TMEM lanes. Each
// epilogue warp owns 32 lanes; per 32 token columns it moves its 32 x 32
// logits through a shared-memory transpose so that each thread holds one
// token's 32 logits, and keeps a running (max, sum of exponentials, argmax)
// per token across the v-tiles of its unit. The warps' states are combined
// once per unit, and each CTA writes its own partial per token. Accumulators
// live in TMEM: three of 160 columns for groups of at most 160 tokens (the
// epilogue of one tile overlaps two tiles of MMAs), else two of 256.
//
// Two pairs per cluster (the plan's MC = 2, clusters of 4 CTAs): the pairs
// hold adjacent token groups of the same vocabulary part, so they need the
// same head tiles. Each head tile is then read from L2 once for both: every
// CTA loads a 64-row half of its 128 head rows and multicasts it to the CTA
// of the same rank in the other pair; a stage is free again when both
// pairs' MMAs have consumed it (each pair's issuer commits to the stage's
// empty barrier of all four CTAs). Halving the head's L2-to-SM traffic this
// way cut the 8 x 2 x 32 bf16 LM head by ~11% in a diagnostic build in which
// one of the two pairs skipped its head loads.
//
// Or the two pairs share token rows (the plan's vc = 2): they hold the same
// token group and take the two v-tiles of each step of their vocabulary part
// (v-tiles 2t and 2t + 1), each CTA loading its own head rows and a quarter
// of its pair's token rows, multicast to the CTA of the same rank in the
// other pair. Stage release is the same; each pair keeps its own running
// state and writes its own partials. This halves the token rows' L2-to-SM
// traffic instead, the larger operand when the rows are two E4M3 terms per
// element against a one-byte head.
//
// CTA layout (bf16 heads, 192 threads): warp 0 TMA producer, warp 1 TMEM
// allocation (both CTAs) and the MMA issuer (even CTA), warps 2..5 epilogue.
// The producer and issuer loops run in the whole warp and one elected lane
// issues, which keeps the MMA issue rate at the tensor pipe's rate (N = 160:
// 80 cycles per MMA). Every wait is bounded (see common.cuh).
//
// The verification instantiation (VERIFY = true, speculative decoding) also
// carries, per token, the entropy accumulator sum exp(l - m) (l - m) log2(e)
// and the logit of the token's draft entry (typical-acceptance appendix); its
// larger combine buffers cost shared memory, so it may run one stage fewer.
//
// W8A8 (HF = HF_W8A8): E4M3 head rows times E4M3 token rows (quantised per
// row by the compaction kernel) with tcgen05.mma kind::f8f6f4, K = 32 per
// MMA, one 128-column (128-byte) atom per stage; an 8-bit tile takes half the
// tensor time of a bf16 one, so the epilogue has eight warps (two per lane
// quarter, alternate 32-column chunks; 320 threads). Each token's scale
// multiplies its logits through the exponent's factor.
//
// W8A16 on the 8-bit path (HF = HF_E4M3X2): an E4M3 head times bf16 token
// rows, each row packed by the compaction kernel as two E4M3 terms hi + lo of
// the row scaled by a power of two (exact for every element of at least 2^-10
// of the row's largest). Per 128-column stage the head atom is staged once
// and multiplied into the same accumulator by the hi and the lo token atoms:
// eight K = 32 kind::f8f6f4 MMAs, the tensor time of the bf16 head's stage,
// at half its head bytes and with no decode of the head at all. The E4M3 x
// E4M3 products are exact in fp32.
//
// Heads decoded in the kernel (HF = HF_E4M3, HF_NVFP4: the precision levers):
// HBM carries the stored head only. A raw-code producer warp streams this
// CTA's head codes (and NVFP4 block scales) with TMA into a raw ring, and
// eight converter warps decode them exactly into the operand tile of each
// 64-column stage, in its 128-byte-swizzled layout: f16 on the commit step
// (the token rows then come as f16 scaled by a power of two per row, undone
// on the logits like W8A8's scales), bf16 for verification. Each CTA
// multiplies its 128 head rows by all NT token rows with cta_group::1 MMAs,
// so converters signal only their own CTA; the operand stage is full when
// its eight converter warps have arrived and the token rows' bytes have
// landed. E4M3 raw stages hold 128 columns of d, NVFP4 raw stages 256 (128
// bytes of codes per row either way); 480 threads.
#include <atomic>
#include <cstring>

#include "kernels.h"

namespace bd {

namespace {

// Heads decoded in the kernel by converter warps (E4M3 / NVFP4 codes); the
// W8A8 variant multiplies E4M3 codes directly on the 8-bit tensor path.
template <int HF>
__host__ __device__ constexpr bool is_quant() {
  return HF == HF_E4M3 || HF == HF_NVFP4;
}
// Instantiations that issue cta_group::2 MMAs and must run as clusters of 2
// (the heads decoded in the kernel run one CTA per half v-tile instead).
template <int HF>
__host__ __device__ constexpr bool pair_cluster() {
  return !is_quant<HF>();
}
// E4M3 head codes read by TMA straight into the MMA operand (8-bit atoms)
template <int HF>
__host__ __device__ constexpr bool is_8bit() {
  return HF == HF_W8A8 || HF == HF_E4M3X2;
}
// token-operand terms per stage: hi and lo for the two-term rows, else one
template <int HF>
__host__ __device__ constexpr int b_terms() {
  return HF == HF_E4M3X2 ? 2 : 1;
}
// columns of d per operand stage: two 64-column 16-bit swizzle atoms for bf16
// heads; one 128-column 8-bit atom for W8A8; one 16-bit atom for heads decoded
// in the kernel, whose small stages leave room for a deep raw ring
template <int HF>
__host__ __device__ constexpr int stage_k() {
  return is_quant<HF>() ? 64 : 128;
}
// columns of one 128-byte swizzle atom
template <int HF>
__host__ __device__ constexpr int atom_cols() {
  return is_8bit<HF>() ? 128 : 64;
}
constexpr int MAX_STAGES = 8;
constexpr uint32_t ATOM_ROWS_BYTES = 128;  // one row of a swizzle atom (64 16-bit or 128 8-bit columns)
constexpr uint32_t A_BLOCK = 128 * ATOM_ROWS_BYTES;  // this CTA's 128 head rows x one atom
constexpr uint32_t TMEM_COLS = 512;  // two accumulators of up to 256 columns, or three of up to 160
constexpr int MAX_ACC = 3;
constexpr int EPI_WARPS = 4;  // epilogue warps of the bf16 and decoded-head instantiations
constexpr int TR = 34;  // padded row of the transpose buffers: 8-byte aligned rows, conflict-free column reads
constexpr int MAX_CHUNKS = 8;
constexpr int MAX_RAW = 8;
constexpr int QUANT_STAGES = 4;  // operand stages next to the raw ring (quantised heads)
constexpr int CONV_WARPS = 8;                            // converter warps 6..13 (quantised heads)
constexpr int CONV_THREADS = CONV_WARPS * 32;
constexpr int RAW_PRODUCER = 2 + EPI_WARPS + CONV_WARPS;  // warp streaming the quantised codes

// Epilogue warps: W8A8's MMAs take half the time of bf16's per tile, so two
// warps per TMEM lane quarter (each taking every other 32-column chunk of the
// accumulator) keep the epilogue off the critical path.
template <int HF>
__host__ __device__ constexpr int epi_warps() {
  return HF == HF_W8A8 ? 2 * EPI_WARPS : EPI_WARPS;
}
template <int HF>
__host__ __device__ constexpr int pair_threads() {
  return is_quant<HF>() ? (RAW_PRODUCER + 1) * 32 : (2 + epi_warps<HF>()) * 32;
}
static_assert(pair_threads<HF_BF16>() == TC_THREADS, "bf16 pair kernel: producer, MMA and four epilogue warps");
// Raw ring of a quantised head: stages of 128 head rows x 128 bytes of codes
// (SW128), plus 16 bytes of NVFP4 block scales per row.
constexpr uint32_t RAW_CODE_BYTES = 128 * 128;
template <int HF>
__host__ __device__ constexpr uint32_t raw_bytes() {
  return HF == HF_NVFP4 ? RAW_CODE_BYTES + 128 * 16 : RAW_CODE_BYTES;
}
// operand stages per raw stage (a raw stage holds 256 NVFP4 or 128 E4M3 columns)
template <int HF>
__host__ __device__ constexpr int raw_k() {
  return (HF == HF_NVFP4 ? 256 : 128) / stage_k<HF>();
}

struct PairCtl {
  uint64_t full[MAX_STAGES];
  uint64_t empty[MAX_STAGES];
  uint64_t tfull[MAX_ACC];
  uint64_t tempty[MAX_ACC];
  uint64_t drain;
  uint64_t epi_sync;  // rendezvous of the 128 epilogue threads (bounded, unlike bar.sync)
  uint64_t rfull[MAX_RAW];   // quantised heads: raw codes landed (TMA transaction bytes)
  uint64_t rempty[MAX_RAW];  // ... and consumed by the converter warps
  uint32_t tmem_base;
  int abort_flag;
};

// One buffer per epilogue warp: the 32 x 33 transpose during the tiles of a
// unit; after the warp's last tile, the same warp's running states (max, sum,
// argmax for up to 256 tokens; with VERIFY also the entropy accumulator and
// the draft logit) for the cross-warp combine. A warp only ever writes its own
// buffer before the rendezvous, so no warp can overwrite a buffer another warp
// is still transposing in.
template <bool VERIFY>
struct PairWarpBuf {
  union {
    float tr[32 * TR];
    struct {
      float m[256];
      float s[256];
      int a[256];
      float t[VERIFY ? 256 : 1];
      float x[VERIFY ? 256 : 1];
    } st;
  };
};

template <bool VERIFY, int EW>
struct PairTail {
  PairWarpBuf<VERIFY> w[EW];
  PairCtl ctl;
};

constexpr size_t SMEM_BYTES = 232448;  // the whole opt-in shared memory of an SM
template <int HF, bool VERIFY>
__host__ __device__ constexpr size_t stage_area() {
  return SMEM_BYTES - 1024 - sizeof(PairTail<VERIFY, epi_warps<HF>()>);
}

// Stage layout for a token group of NT rows (NT/2 in each CTA), one block per
// atom: [A block 0 (| A block 1) | B block 0 (| B block 1)], A = 128 head
// rows, B = NT/2 token rows (all NT for heads decoded in the kernel), each
// block 1 KB aligned.
template <int HF>
__host__ __device__ constexpr uint32_t stage_bytes(int nt) {
  // heads decoded in the kernel: one CTA multiplies its 128 head rows by all NT token rows
  return is_quant<HF>() ? A_BLOCK + static_cast<uint32_t>(nt) * ATOM_ROWS_BYTES
                        : (stage_k<HF>() / atom_cols<HF>()) *
                              (A_BLOCK + b_terms<HF>() * static_cast<uint32_t>(nt / 2) * ATOM_ROWS_BYTES);
}
// Operand stages: as many as fit (at most MAX_STAGES) for bf16 heads; for
// quantised heads at most QUANT_STAGES next to a raw ring of at least three
// stages, which takes the rest of the area.
template <int HF, bool VERIFY>
__host__ __device__ constexpr int stage_count(int nt) {
  return is_quant<HF>()
             ? (static_cast<int>((stage_area<HF, VERIFY>() - 3 * raw_bytes<HF>()) / stage_bytes<HF>(nt)) < QUANT_STAGES
                    ? static_cast<int>((stage_area<HF, VERIFY>() - 3 * raw_bytes<HF>()) / stage_bytes<HF>(nt))
                    : QUANT_STAGES)
         : static_cast<int>(stage_area<HF, VERIFY>() / stage_bytes<HF>(nt)) < MAX_STAGES
             ? static_cast<int>(stage_area<HF, VERIFY>() / stage_bytes<HF>(nt))
             : MAX_STAGES;
}
template <int HF, bool VERIFY>
__host__ __device__ constexpr int raw_count(int nt) {
  return !is_quant<HF>() ? 0
         : static_cast<int>((stage_area<HF, VERIFY>() - stage_count<HF, VERIFY>(nt) * stage_bytes<HF>(nt)) /
                            raw_bytes<HF>()) < MAX_RAW
             ? static_cast<int>((stage_area<HF, VERIFY>() - stage_count<HF, VERIFY>(nt) * stage_bytes<HF>(nt)) /
                                raw_bytes<HF>())
             : MAX_RAW;
}
static_assert(stage_count<HF_BF16, false>(256) >= 3 && stage_count<HF_BF16, true>(256) >= 3, "three stages at NT = 256");
static_assert(stage_count<HF_BF16, false>(160) == 4, "four stages at NT = 160 on the commit path");
static_assert(stage_count<HF_W8A8, false>(160) == 7 && stage_count<HF_W8A8, false>(256) >= 5,
              "W8A8: seven 26 KB stages at NT = 160, five 32 KB stages at NT = 256");
static_assert(stage_count<HF_E4M3X2, false>(160) == 5 && stage_count<HF_E4M3X2, false>(256) == 4,
              "two-term rows: five 36 KB stages at NT = 160, four 48 KB stages at NT = 256");
static_assert(stage_count<HF_NVFP4, false>(160) == 4 && stage_count<HF_E4M3, false>(160) == 4 &&
                  stage_count<HF_NVFP4, true>(160) == 4 && stage_count<HF_E4M3, true>(160) == 4,
              "four operand stages at NT = 160 for quantised heads");
static_assert(stage_count<HF_NVFP4, true>(256) >= 3 && stage_count<HF_E4M3, true>(256) >= 3 &&
                  raw_count<HF_NVFP4, true>(256) >= 3 && raw_count<HF_E4M3, true>(256) >= 3,
              "three operand and three raw stages at NT = 256");

// Decodes this thread's share of one operand stage (128 head rows x 64
// columns, global columns kcol0..) from the raw stage at raw_base into the
// f16 (F16) or bf16 A tile at a_base (one SW128 atom); both are exact. h:
// which 64-column part of the raw stage. Columns at or past d decode to zero.
// ct: 0..CONV_THREADS-1.
template <int HF, bool F16>
__device__ __forceinline__ void convert_stage(uint32_t raw_base, int h, uint32_t a_base, int ct, int kcol0, int d) {
  static_assert(!is_quant<HF>() || stage_k<HF>() == 64, "one atom per quantised operand stage");
  if constexpr (HF == HF_NVFP4) {
#pragma unroll
    for (int i = 0; i < 256 / CONV_THREADS; ++i) {
      const int ci = ct + CONV_THREADS * i;
      const int row = ci >> 1, j = ci & 1;  // 32-column chunk j of the stage
      const int c = h * 2 + j;              // its 16 bytes of codes within the raw row
      const uint4 q = ld_shared_v4(raw_base + row * 128 + ((c ^ (row & 7)) << 4));
      const uint32_t s01 = e4m3x2_to_f16x2(ld_shared_u16(raw_base + RAW_CODE_BYTES + row * 16 + c * 2));
      const uint32_t sc[2] = {__byte_perm(s01, 0, 0x1010), __byte_perm(s01, 0, 0x3232)};
      const uint32_t words[4] = {q.x, q.y, q.z, q.w};
      uint32_t w[16];
#pragma unroll
      for (int b = 0; b < 16; ++b)  // byte b: elements 2b (low nibble), 2b + 1; 16 elements per block scale
      {
        const uint32_t hv = hmul2_u32(e2m1x2_to_f16x2(__byte_perm(words[b >> 2], 0, 0x4440 + (b & 3))), sc[b >> 3]);
        w[b] = F16 ? hv : f16x2_to_bf16x2(hv);
      }
      const int col0 = kcol0 + j * 32;
      if (col0 + 32 > d) {
#pragma unroll
        for (int b = 0; b < 16; ++b) {
          if (col0 + 2 * b >= d) w[b] = 0u;
          else if (col0 + 2 * b + 1 >= d) w[b] &= 0xFFFFu;
        }
      }
      const uint32_t rowbase = a_base + row * 128;
#pragma unroll
      for (int u = 0; u < 4; ++u)
        st_shared_v4(rowbase + (((j * 4 + u) ^ (row & 7)) << 4), w[4 * u], w[4 * u + 1], w[4 * u + 2], w[4 * u + 3]);
    }
  } else {
#pragma unroll
    for (int i = 0; i < 512 / CONV_THREADS; ++i) {
      const int ci = ct + CONV_THREADS * i;
      const int row = ci >> 2, j = ci & 3;  // 16-column chunk j of the stage
      const int c = h * 4 + j;              // its 16 bytes of codes within the raw row
      const uint4 q = ld_shared_v4(raw_base + row * 128 + ((c ^ (row & 7)) << 4));
      const uint32_t words[4] = {q.x, q.y, q.z, q.w};
      uint32_t w[8];
#pragma unroll
      for (int b = 0; b < 8; ++b)  // bytes 2b, 2b + 1: elements 2b, 2b + 1
      {
        const uint32_t hv = e4m3x2_to_f16x2(__byte_perm(words[b >> 1], 0, (b & 1) ? 0x4432 : 0x4410));
        w[b] = F16 ? hv : f16x2_to_bf16x2(hv);
      }
      const int col0 = kcol0 + j * 16;
      if (col0 + 16 > d) {
#pragma unroll
        for (int b = 0; b < 8; ++b) {
          if (col0 + 2 * b >= d) w[b] = 0u;
          else if (col0 + 2 * b + 1 >= d) w[b] &= 0xFFFFu;
        }
      }
      const uint32_t rowbase = a_base + row * 128;
#pragma unroll
      for (int u = 0; u < 2; ++u)
        st_shared_v4(rowbase + (((j * 2 + u) ^ (row & 7)) << 4), w[4 * u], w[4 * u + 1], w[4 * u + 2], w[4 * u + 3]);
    }
  }
}

}  // namespace

template <int HF, bool VERIFY>
__global__ void __launch_bounds__(pair_threads<HF>(), 1)
    lmhead_pair_kernel(const __grid_constant__ PairTokenMaps tmH, const __grid_constant__ CUtensorMap tmW,
                       const __grid_constant__ PairQuantMaps tmQ, const __grid_constant__ PairTokenMaps tmL,
                       TcArgs a) {
  constexpr bool QUANT = is_quant<HF>();
  constexpr bool W8A8 = HF == HF_W8A8;
  constexpr bool X2 = HF == HF_E4M3X2;
  static_assert(!((W8A8 || X2) && VERIFY), "the 8-bit instantiations serve the commit step");
  // commit step with a head decoded in the kernel: f16 operands (the decode
  // ends at f16), token rows pre-scaled by a power of two per row
  constexpr bool F16OPS = QUANT && !VERIFY;
  // the packed rows carry a per-row scale that multiplies their logits
  constexpr bool TOKS = W8A8 || X2 || F16OPS;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  constexpr int EW = epi_warps<HF>();
  PairTail<VERIFY, EW>* tail = reinterpret_cast<PairTail<VERIFY, EW>*>(smem + stage_area<HF, VERIFY>());
  PairCtl* ctl = &tail->ctl;
  const uint32_t smem_base = smem_u32(smem);

  // pairs per cluster (two share each head tile by multicast); quantised
  // heads run without clusters
  // pairs per cluster: two sharing head tiles (mc = 2) or token rows (vc = 2)
  const int VC = QUANT ? 1 : plan_vc(a.plan);
  const int MC = QUANT ? 1 : plan_mc(a.plan) * VC;
  if constexpr (pair_cluster<HF>()) {
    // launched without its cluster there is no peer CTA to map or to pair
    // MMAs with: report and do nothing
    if (cluster_nctarank() != static_cast<uint32_t>(2 * MC)) {
      if (threadIdx.x == 0) atomicOr(a.status, DEV_BAD_LAUNCH);
      return;
    }
  }
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t crank = QUANT ? 0u : cluster_ctarank();
  // 0: the CTA that issues the pair's MMAs (bf16 heads); quantised heads: the
  // half of the v-tile this CTA takes on its own
  const uint32_t rank = QUANT ? (blockIdx.x & 1u) : (crank & 1u);
  const int pp = static_cast<int>(crank >> 1);  // this pair's token group (vc = 1) or v-tile (vc = 2) in the runner
  const int pp_mt = VC == 1 ? pp : 0;           // ... its token group within the runner's m-tiles
  const uint32_t lead = crank & ~1u;            // cluster rank of this pair's issuing CTA
  const uint32_t pair_mask = 3u << (2 * pp);    // both CTAs of this pair
  const uint32_t all_mask = (1u << (2 * MC)) - 1u;
  const int pair = QUANT ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x) / (2 * MC);

  if (threadIdx.x == 0) {
    if constexpr (QUANT) {
      prefetch_tmap(&tmQ.codes);
      if constexpr (HF == HF_NVFP4) prefetch_tmap(&tmQ.scales);
      for (int r = 0; r < MAX_RAW; ++r) {
        mbar_init(smem_u32(&ctl->rfull[r]), 1);
        mbar_init(smem_u32(&ctl->rempty[r]), CONV_WARPS);
      }
    } else {
      prefetch_tmap(&tmW);
    }
    for (int s = 0; s < MAX_STAGES; ++s) {
      // quantised heads: the token bytes' arrival plus the CTA's converter warps
      mbar_init(smem_u32(&ctl->full[s]), QUANT ? 1 + CONV_WARPS : 1);
      // commits of the issuing CTA of every pair that reads this stage
      mbar_init(smem_u32(&ctl->empty[s]), static_cast<uint32_t>(MC));
    }
    for (int i = 0; i < MAX_ACC; ++i) {
      mbar_init(smem_u32(&ctl->tfull[i]), 1);
      mbar_init(smem_u32(&ctl->tempty[i]), QUANT ? EW : 2 * EW);
    }
    mbar_init(smem_u32(&ctl->drain), 1);
    mbar_init(smem_u32(&ctl->epi_sync), EW * 32);
    ctl->abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    if constexpr (QUANT) {
      tmem_alloc(smem_u32(&ctl->tmem_base), TMEM_COLS);
      tmem_relinquish();
    } else {
      tmem_alloc_pair(smem_u32(&ctl->tmem_base), TMEM_COLS);
      tmem_relinquish_pair();
    }
  }
  tc_fence_before();
  if constexpr (QUANT)
    __syncthreads();
  else
    cluster_sync_all();  // barriers initialised and TMEM allocated in both CTAs
  tc_fence_after();
  const uint32_t tmem_base = ctl->tmem_base;
  volatile int* abort_flag = &ctl->abort_flag;

  // The packed rows and the header (N, the plan) come from the preceding
  // kernel. A spill launch (role 1) follows the main launch, which waited for
  // that kernel before letting it start; with a spill launch behind it the
  // main launch lets it start at once, onto the SMs this grid leaves free.
  const bool spill = a.plan.role == 1;
  if (!spill) griddep_wait();
  if (!spill && a.plan.G2 > 0) griddep_launch_dependents();
  const int n_rows = hdr_word(a.n_rows, HDR_N);
  constexpr int BK = stage_k<HF>();
  constexpr int ACOLS = atom_cols<HF>();
  constexpr int NATOM = BK / ACOLS;
  const int nk = cdiv(a.d, BK);
  const int NT = pair_group_rows(n_rows);
  const int half = NT / 2;
  // accumulators in TMEM: three of 160 columns when a group has at most 160
  // tokens (the epilogue of one tile then overlaps two tiles of MMAs), else two of 256
  const uint32_t NACC = NT <= 160 ? 3u : 2u;
  const uint32_t ACC_COLS = NT <= 160 ? 160u : 256u;
  const int nch = NT / 32;
  const uint32_t SB = stage_bytes<HF>(NT);
  const uint32_t B_BLOCK = static_cast<uint32_t>(half) * ATOM_ROWS_BYTES;
  const int STAGES = stage_count<HF, VERIFY>(NT);
  const int RSTAGES = raw_count<HF, VERIFY>(NT);
  // bf16 heads: both CTAs' bytes land on the even CTA's barrier; quantised
  // heads: this CTA's token rows only
  const uint32_t tx_total = QUANT ? static_cast<uint32_t>(NT) * ATOM_ROWS_BYTES : 2u * SB;
  const uint32_t raw_base = smem_base + static_cast<uint32_t>(STAGES) * SB;  // quantised heads' raw ring
  const CUtensorMap* tm_tok = &tmH.m[half / 8 - 1];  // box of exactly `half` rows
  const CUtensorMap* tm_lo = &tmL.m[half / 8 - 1];   // two-term rows: the lo terms
  // vc = 2: boxes of a quarter of the group (NT is a multiple of 32)
  const CUtensorMap* tm_tok_q = &tmH.m[half / 16 - 1];
  const CUtensorMap* tm_lo_q = &tmL.m[half / 16 - 1];

  if (warp == 0) {
    // ------------------------------------------------------ TMA producer
    // the whole warp walks the stages (warp-uniform waits); one lane issues
    const bool leader = elect_one();
    // head rows: fetched from HBM once per band and re-read from L2 by the
    // band's other token groups; token rows: re-read for every v-tile
    const uint64_t pol_w = l2_policy(a.l2_head);
    const uint64_t pol_h = l2_policy(a.l2_rows);
    const uint32_t full0_leader = mapa_shared(smem_u32(&ctl->full[0]), lead);
    const uint16_t head_mc = static_cast<uint16_t>(5u << rank);  // this rank's CTA in both pairs
    uint32_t stage = 0, phase = 0;
    uint32_t issued_mask = 0, issued_phase = 0;
    TileIter it;
    it.init(a.plan, a.n_rows, pair);
    bool ok = true;
    while (ok && it.next_unit()) {
      const int tok0 = (it.m_tile + pp_mt) * NT + (QUANT ? 0 : static_cast<int>(rank) * half);
      for (int step = it.vt; ok && step < it.vt_end; ++step) {
        int vt = step * VC + (VC == 2 ? pp : 0);
        // vc = 2 and an odd v-tile count: the last step's second v-tile lies past
        // V; load the one before it (its logits are all dead in the epilogue)
        if (vt > 0 && vt * 256 >= a.V) --vt;
        const int vrow = vt * 256 + static_cast<int>(rank) * 128;
        for (int kb = 0; kb < nk; ++kb) {
          if (!mbar_wait_warp(smem_u32(&ctl->empty[stage]), phase ^ 1u, abort_flag, a.status)) {
            ok = false;
            break;
          }
          if (leader) {
            const uint32_t sa = smem_base + stage * SB;
            if constexpr (QUANT) {
              // all NT token rows of the group, as two boxes of NT/2 rows
              const uint32_t fb = smem_u32(&ctl->full[stage]);
              mbar_expect_tx(fb, tx_total);
              tma_load_2d(sa + A_BLOCK, tm_tok, fb, kb * BK, tok0, pol_h);
              tma_load_2d(sa + A_BLOCK + B_BLOCK, tm_tok, fb, kb * BK, tok0 + half, pol_h);
            } else {
              if (rank == 0) mbar_expect_tx(smem_u32(&ctl->full[stage]), tx_total);
              const uint32_t fb = full0_leader + 8u * stage;
#pragma unroll
              for (int j = 0; j < NATOM; ++j) {
                // the head atom's 128 rows as two boxes of 64: both loaded here, or
                // (two pairs per cluster) this pair's half multicast to both pairs
                if (MC == 1 || VC == 2) {
                  tma_load_2d_pair(sa + j * A_BLOCK, &tmW, fb, kb * BK + ACOLS * j, vrow, pol_w);
                  tma_load_2d_pair(sa + j * A_BLOCK + A_BLOCK / 2, &tmW, fb, kb * BK + ACOLS * j, vrow + 64, pol_w);
                } else {
                  tma_load_2d_pair_mc(sa + j * A_BLOCK + pp * (A_BLOCK / 2), &tmW, fb, kb * BK + ACOLS * j,
                                      vrow + 64 * pp, head_mc, pol_w);
                }
                if (VC == 2) {
                  // this CTA's quarter of its pair's token rows, for both pairs
                  tma_load_2d_pair_mc(sa + NATOM * A_BLOCK + j * B_BLOCK + pp * (B_BLOCK / 2), tm_tok_q, fb,
                                      kb * BK + ACOLS * j, tok0 + pp * (half / 2), head_mc, pol_h);
                } else {
                  tma_load_2d_pair(sa + NATOM * A_BLOCK + j * B_BLOCK, tm_tok, fb, kb * BK + ACOLS * j, tok0, pol_h);
                }
              }
              if constexpr (X2) {
                if (VC == 2)
                  tma_load_2d_pair_mc(sa + A_BLOCK + B_BLOCK + pp * (B_BLOCK / 2), tm_lo_q, fb, kb * BK,
                                      tok0 + pp * (half / 2), head_mc, pol_h);
                else
                  tma_load_2d_pair(sa + A_BLOCK + B_BLOCK, tm_lo, fb, kb * BK, tok0, pol_h);
              }
            }
          }
          __syncwarp();
          issued_mask |= 1u << stage;
          issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
    }
    // The even CTA's full barriers count both CTAs' bytes: once they have
    // flipped for the last issue of every stage, no copy is in flight.
    if (rank == 0 && leader)
      for (int s = 0; s < STAGES; ++s)
        if (issued_mask & (1u << s)) mbar_drain(smem_u32(&ctl->full[s]), (issued_phase >> s) & 1u);
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------ MMA issuer (even CTA; every CTA for quantised heads)
    if (rank == 0 || QUANT) {
      const bool leader = elect_one();
      const uint32_t idesc = (W8A8 || X2) ? idesc_e4m3_f32(256, NT)
                             : F16OPS ? idesc_f16_f32(128, NT)
                                      : idesc_bf16_f32(QUANT ? 128 : 256, NT);
      uint32_t stage = 0, phase = 0;
      uint32_t acc = 0, acc_phase = 0;
      TileIter it;
      it.init(a.plan, a.n_rows, pair);
      bool ok = true;
      while (ok && it.next_unit()) {
        for (int vt = it.vt; ok && vt < it.vt_end; ++vt) {
          if (!mbar_wait_warp(smem_u32(&ctl->tempty[acc]), acc_phase ^ 1u, abort_flag, a.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + acc * ACC_COLS;
          for (int kb = 0; kb < nk; ++kb) {
            if (!mbar_wait_warp(smem_u32(&ctl->full[stage]), phase, abort_flag, a.status)) {
              ok = false;
              break;
            }
            tc_fence_after();
            if (leader) {
              const uint32_t sa = smem_base + stage * SB;
#pragma unroll
              for (int j = 0; j < NATOM; ++j) {
                const uint64_t adesc = sw128_kmajor_desc(sa + j * A_BLOCK);
                const uint64_t bdesc = sw128_kmajor_desc(sa + NATOM * A_BLOCK + j * B_BLOCK);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                  // +32 bytes along K per MMA (16 bf16 / 32 E4M3 columns) = +2 in the address field
                  if constexpr (QUANT) {
                    umma_bf16(d_tmem, adesc + 2u * k, bdesc + 2u * k, idesc, (kb | j | k) != 0);
                  } else if constexpr (X2) {
                    // the head atom times the hi terms, then times the lo terms
                    const uint64_t ldesc = sw128_kmajor_desc(sa + A_BLOCK + B_BLOCK);
                    umma_f8_pair(d_tmem, adesc + 2u * k, bdesc + 2u * k, idesc, (kb | k) != 0);
                    umma_f8_pair(d_tmem, adesc + 2u * k, ldesc + 2u * k, idesc, true);
                  } else if constexpr (W8A8) {
                    umma_f8_pair(d_tmem, adesc + 2u * k, bdesc + 2u * k, idesc, (kb | j | k) != 0);
                  } else {
                    umma_bf16_pair(d_tmem, adesc + 2u * k, bdesc + 2u * k, idesc, (kb | j | k) != 0);
                  }
                }
              }
              if constexpr (QUANT)
                umma_commit(smem_u32(&ctl->empty[stage]));
              else  // the stage's head halves came from both pairs: free it in every CTA
                umma_commit_pair_mc(smem_u32(&ctl->empty[stage]), static_cast<uint16_t>(all_mask));
            }
            __syncwarp();
            if (++stage == STAGES) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (!ok) break;
          if (leader) {
            if constexpr (QUANT)
              umma_commit(smem_u32(&ctl->tfull[acc]));
            else
              umma_commit_pair_mc(smem_u32(&ctl->tfull[acc]), static_cast<uint16_t>(pair_mask));
          }
          __syncwarp();
          if (++acc == NACC) {
            acc = 0;
            acc_phase ^= 1u;
          }
        }
      }
      if (leader) {
        if constexpr (QUANT)
          umma_commit(smem_u32(&ctl->drain));
        else
          umma_commit_pair_mc(smem_u32(&ctl->drain), static_cast<uint16_t>(1u << crank));
        mbar_drain(smem_u32(&ctl->drain), 0);
      }
      __syncwarp();
    }
  } else if (QUANT && warp == RAW_PRODUCER) {
    // ------------------------------------------------------ raw-code producer (quantised heads)
    const bool leader = elect_one();
    const uint64_t pol = l2_policy(a.l2_head);  // the codes of the band's head tiles, as above
    const int RS = RSTAGES;
    const int nkr = cdiv(nk, raw_k<HF>());
    uint32_t r = 0, rph = 0;
    uint32_t issued_mask = 0, issued_phase = 0;
    TileIter it;
    it.init(a.plan, a.n_rows, pair);
    bool ok = true;
    while (ok && it.next_unit()) {
      for (int vt = it.vt; ok && vt < it.vt_end; ++vt) {
        const int vrow = vt * 256 + static_cast<int>(rank) * 128;
        for (int kr = 0; kr < nkr; ++kr) {
          if (!mbar_wait_warp(smem_u32(&ctl->rempty[r]), rph ^ 1u, abort_flag, a.status)) {
            ok = false;
            break;
          }
          if (leader) {
            const uint32_t fb = smem_u32(&ctl->rfull[r]);
            const uint32_t dst = raw_base + r * raw_bytes<HF>();
            mbar_expect_tx(fb, raw_bytes<HF>());
            tma_load_2d(dst, &tmQ.codes, fb, kr * 128, vrow, pol);
            if constexpr (HF == HF_NVFP4) tma_load_2d(dst + RAW_CODE_BYTES, &tmQ.scales, fb, kr * 16, vrow, pol);
          }
          __syncwarp();
          issued_mask |= 1u << r;
          issued_phase = (issued_phase & ~(1u << r)) | (rph << r);
          if (++r == static_cast<uint32_t>(RS)) {
            r = 0;
            rph ^= 1u;
          }
        }
      }
    }
    if (leader)
      for (int q = 0; q < RS; ++q)
        if (issued_mask & (1u << q)) mbar_drain(smem_u32(&ctl->rfull[q]), (issued_phase >> q) & 1u);
    __syncwarp();
  } else if (QUANT && warp >= 2 + EPI_WARPS) {
    // ------------------------------------------------------ converters (quantised heads)
    const int ct = threadIdx.x - (2 + EPI_WARPS) * 32;  // 0..CONV_THREADS-1
    const int RS = RSTAGES;
    constexpr int RK = raw_k<HF>();
    uint32_t r = 0, rph = 0, stage = 0, phase = 0;
    TileIter it;
    it.init(a.plan, a.n_rows, pair);
    bool ok = true;
    while (ok && it.next_unit()) {
      for (int vt = it.vt; ok && vt < it.vt_end; ++vt) {
        for (int kb = 0; kb < nk; ++kb) {
          const int h = kb % RK;
          if (h == 0 && !mbar_wait_warp(smem_u32(&ctl->rfull[r]), rph, abort_flag, a.status)) {
            ok = false;
            break;
          }
          if (!mbar_wait_warp(smem_u32(&ctl->empty[stage]), phase ^ 1u, abort_flag, a.status)) {
            ok = false;
            break;
          }
          convert_stage<HF, F16OPS>(raw_base + r * raw_bytes<HF>(), h, smem_base + stage * SB, ct, kb * BK, a.d);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&ctl->full[stage]));
          if (h == RK - 1 || kb == nk - 1) {
            if (lane == 0) mbar_arrive(smem_u32(&ctl->rempty[r]));
            if (++r == static_cast<uint32_t>(RS)) {
              r = 0;
              rph ^= 1u;
            }
          }
          if (++stage == static_cast<uint32_t>(STAGES)) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
    }
  } else {
    // ------------------------------------------------------ epilogue
    const int ew = warp - 2;  // epilogue warp 0..EW-1
    const int quarter = warp & 3;
    // with eight epilogue warps, warp ew takes the chunks c with c % 2 == ew / 4
    const int chunk_par = EW == 8 ? (ew >> 2) : -1;
    const uint32_t lane_addr = static_cast<uint32_t>(quarter * 32) << 16;
    float* tr = tail->w[ew].tr;
    const uint32_t tempty_local0 = smem_u32(&ctl->tempty[0]);
    const uint32_t tempty_leader0 = mapa_shared(tempty_local0, lead);
    const uint32_t epi_sync = smem_u32(&ctl->epi_sync);
    uint32_t epi_phase = 0;
    uint32_t acc = 0, acc_phase = 0;
    TileIter it;
    it.init(a.plan, a.n_rows, pair);
    bool ok = true;
    while (ok && it.next_unit()) {
      float m[MAX_CHUNKS], s[MAX_CHUNKS];
      int arg[MAX_CHUNKS];
      float t[MAX_CHUNKS], lx[MAX_CHUNKS];  // VERIFY only
      int xd[MAX_CHUNKS];                   // VERIFY only: draft entry of this thread's token
      // W8A8 and f16 rows: this thread's token scale ts (1 for an all-zero row). The
      // running max m is kept in unscaled accumulator units (ts > 0 keeps
      // the max and argmax), the exponents use k2 = ts * log2(e), and the
      // partial max is scaled by ts when written.
      float ts[MAX_CHUNKS], k2[MAX_CHUNKS];
#pragma unroll
      for (int c = 0; c < MAX_CHUNKS; ++c) {
        m[c] = -INFINITY;
        s[c] = 0.f;
        arg[c] = 0x7fffffff;
        t[c] = 0.f;
        lx[c] = -INFINITY;
        xd[c] = -1;
        ts[c] = 1.f;
        if constexpr (TOKS) {
          const int row = (it.m_tile + pp_mt) * NT + c * 32 + lane;
          if (c < nch && row < n_rows && a.tok_scale[row] != 0.f) ts[c] = a.tok_scale[row];
        }
        k2[c] = ts[c] * LOG2E;
        if constexpr (VERIFY) {
          const int row = (it.m_tile + pp_mt) * NT + c * 32 + lane;
          if (c < nch && row < n_rows) xd[c] = a.draft_row[row];
        }
      }
      for (int step = it.vt; step < it.vt_end; ++step) {
        const int vt = step * VC + (VC == 2 ? pp : 0);
        if (!mbar_wait_warp(smem_u32(&ctl->tfull[acc]), acc_phase, abort_flag, a.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const int vrow0 = vt * 256 + static_cast<int>(rank) * 128 + quarter * 32;  // vocabulary row of lane 0
        const int my_v = vrow0 + lane;
        const bool dead = my_v >= a.V || my_v == a.mask_id;
        const bool scaled = a.wscale != nullptr;
        const float sc = (scaled && !dead) ? __ldg(a.wscale + my_v) : 1.f;
#pragma unroll
        for (int c = 0; c < MAX_CHUNKS; ++c) {
          if (c < nch && (chunk_par < 0 || (c & 1) == chunk_par)) {
            float v[32];
            tmem_ld32(tmem_base + lane_addr + acc * ACC_COLS + c * 32, v);
            // this lane's row of the transpose, two floats per store; the mask
            // entry and rows past V are -inf, the e4m3 row scale applies to live rows
            float2* row = reinterpret_cast<float2*>(tr + lane * TR);
            if (dead) {
#pragma unroll
              for (int j = 0; j < 16; ++j) row[j] = make_float2(-INFINITY, -INFINITY);
            } else if (scaled) {
#pragma unroll
              for (int j = 0; j < 16; ++j) row[j] = make_float2(v[2 * j] * sc, v[2 * j + 1] * sc);
            } else {
#pragma unroll
              for (int j = 0; j < 16; ++j) row[j] = make_float2(v[2 * j], v[2 * j + 1]);
            }
            __syncwarp();
            float x[32];
#pragma unroll
            for (int r = 0; r < 32; ++r) x[r] = tr[r * TR + lane];
            if constexpr (VERIFY) {
              const int rel = xd[c] - vrow0;
              if (rel >= 0 && rel < 32) lx[c] = tr[rel * TR + lane];
            }
            __syncwarp();
            // this thread: token column c*32 + lane, vocabulary rows vrow0 + r
            float cm = x[0];
#pragma unroll
            for (int r = 1; r < 32; ++r) cm = fmaxf(cm, x[r]);
            if (cm > m[c]) {
              int rr = 31;
#pragma unroll
              for (int r = 31; r >= 0; --r)
                if (x[r] == cm) rr = r;
              arg[c] = vrow0 + rr;
              if constexpr (VERIFY) {
                if (m[c] == -INFINITY) {
                  s[c] = 0.f;
                  t[c] = 0.f;
                } else {
                  const float dm = (m[c] - cm) * LOG2E;
                  const float f = ex2_approx(dm);
                  t[c] = f * fmaf(dm, s[c], t[c]);
                  s[c] *= f;
                }
              } else {
                s[c] = (m[c] == -INFINITY) ? 0.f : s[c] * ex2_approx((m[c] - cm) * k2[c]);
              }
              m[c] = cm;
            }
            if (m[c] != -INFINITY) {
              const float mc = m[c] * k2[c];
              const bool wide = !(fabsf(mc) < FUSED_SHIFT_LIMIT);  // take x - m first (see common.cuh)
              if constexpr (VERIFY) {
                // -inf logits give u = -inf, e = 0; clamping u keeps e * u at 0
                float s0 = 0.f, s1 = 0.f, t0 = 0.f, t1 = 0.f;
#pragma unroll
                for (int r = 0; r < 32; r += 2) {
                  const float u0 = wide ? (x[r] - m[c]) * k2[c] : fmaf(x[r], k2[c], -mc);
                  const float u1 = wide ? (x[r + 1] - m[c]) * k2[c] : fmaf(x[r + 1], k2[c], -mc);
                  const float e0 = ex2_approx(u0), e1 = ex2_approx(u1);
                  s0 += e0;
                  s1 += e1;
                  t0 = fmaf(e0, fmaxf(u0, -256.f), t0);
                  t1 = fmaf(e1, fmaxf(u1, -256.f), t1);
                }
                s[c] += s0 + s1;
                t[c] += t0 + t1;
              } else {
                float s0 = 0.f, s1 = 0.f;
                if (!wide) {
#pragma unroll
                  for (int r = 0; r < 32; r += 2) {
                    s0 += ex2_approx(fmaf(x[r], k2[c], -mc));
                    s1 += ex2_approx(fmaf(x[r + 1], k2[c], -mc));
                  }
                } else {
#pragma unroll
                  for (int r = 0; r < 32; r += 2) {
                    s0 += ex2_approx((x[r] - m[c]) * k2[c]);
                    s1 += ex2_approx((x[r + 1] - m[c]) * k2[c]);
                  }
                }
                s[c] += s0 + s1;
              }
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (rank == 0 || QUANT)
            mbar_arrive(tempty_local0 + 8u * acc);
          else
            mbar_arrive_cluster(tempty_leader0 + 8u * acc);
        }
        if (++acc == NACC) {
          acc = 0;
          acc_phase ^= 1u;
        }
      }
      if (!ok) break;
      // combine the four warps' running states and write this CTA's partials
#pragma unroll
      for (int c = 0; c < MAX_CHUNKS; ++c) {
        if (c < nch && (chunk_par < 0 || (c & 1) == chunk_par)) {
          tail->w[ew].st.m[c * 32 + lane] = TOKS ? m[c] * ts[c] : m[c];
          tail->w[ew].st.s[c * 32 + lane] = s[c];
          tail->w[ew].st.a[c * 32 + lane] = arg[c];
          if constexpr (VERIFY) {
            tail->w[ew].st.t[c * 32 + lane] = t[c];
            tail->w[ew].st.x[c * 32 + lane] = lx[c];
          }
        }
      }
      mbar_arrive(epi_sync);
      if (!mbar_wait_warp(epi_sync, epi_phase, abort_flag, a.status)) break;
      epi_phase ^= 1u;
      for (int j = ew * 32 + lane; j < NT; j += EW * 32) {
        // the four warps (one per lane quarter) that hold token j's states
        const int w0 = EW == 8 ? 4 * ((j >> 5) & 1) : 0;
        float M = tail->w[w0].st.m[j], S = tail->w[w0].st.s[j];
        int A = tail->w[w0].st.a[j];
        float T = 0.f, LX = -INFINITY;
        if constexpr (VERIFY) {
          T = tail->w[w0].st.t[j];
          LX = tail->w[w0].st.x[j];
        }
#pragma unroll
        for (int q = 1; q < 4; ++q) {
          const int w = w0 + q;
          if constexpr (VERIFY) {
            softmax_combine_t(M, S, A, T, tail->w[w].st.m[j], tail->w[w].st.s[j], tail->w[w].st.a[j],
                              tail->w[w].st.t[j]);
            LX = fmaxf(LX, tail->w[w].st.x[j]);
          } else {
            softmax_combine(M, S, A, tail->w[w].st.m[j], tail->w[w].st.s[j], tail->w[w].st.a[j]);
          }
        }
        const int row = (it.m_tile + pp_mt) * NT + j;
        if (row < n_rows) {
          // slot: the unit's first (2 per pair, both pairs with vc = 2), then pair and CTA
          const int slot = it.slot0 + it.part * 2 * VC + (VC == 2 ? 2 * pp : 0) + static_cast<int>(rank);
          const int64_t o = static_cast<int64_t>(slot) * a.P + row;
          a.part_m[o] = M;
          a.part_s[o] = S;
          a.part_a[o] = A;
          if constexpr (VERIFY) {
            a.part_t[o] = T;
            a.part_x[o] = LX;
          }
        }
      }
      mbar_arrive(epi_sync);
      if (!mbar_wait_warp(epi_sync, epi_phase, abort_flag, a.status)) break;
      epi_phase ^= 1u;
    }
  }

  __syncwarp();
  griddep_launch_dependents();
  tc_fence_before();
  if constexpr (QUANT)
    __syncthreads();
  else
    cluster_sync_all();  // both CTAs done: no MMA, copy or remote arrival is pending
  tc_fence_after();
  if (warp == 1) {
    if constexpr (QUANT)
      tmem_dealloc(tmem_base, TMEM_COLS);
    else
      tmem_dealloc_pair(tmem_base, TMEM_COLS);
  }
  // the spill launch completes only after the main launch: the kernel after
  // it (the merge) waits on this grid alone
  if (spill) griddep_wait();
}

size_t pair_smem_bytes() { return SMEM_BYTES; }

template <int HF, bool VERIFY>
static cudaError_t pair_opt_in() {
  static std::atomic<uint64_t> opted_in{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if ((opted_in.load() & bit) == 0) {
    e = cudaFuncSetAttribute(lmhead_pair_kernel<HF, VERIFY>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(SMEM_BYTES));
    if (e != cudaSuccess) return e;
    opted_in.fetch_or(bit);
  }
  return cudaSuccess;
}

// runners: clusters of `mc` CTA pairs (mc = 1 without clusters for quantised heads)
static void pair_config(cudaLaunchConfig_t* cfg, cudaLaunchAttribute* attr, int runners, int threads, cudaStream_t st,
                        bool programmatic, bool cluster = true, int mc = 1) {
  *cfg = cudaLaunchConfig_t{};
  cfg->gridDim = dim3(2 * mc * runners, 1, 1);
  cfg->blockDim = dim3(threads, 1, 1);
  cfg->dynamicSmemBytes = SMEM_BYTES;
  cfg->stream = st;
  cfg->attrs = attr;
  cfg->numAttrs = 0;
  if (cluster) {
    attr[cfg->numAttrs].id = cudaLaunchAttributeClusterDimension;
    attr[cfg->numAttrs].val.clusterDim.x = 2 * mc;
    attr[cfg->numAttrs].val.clusterDim.y = 1;
    attr[cfg->numAttrs].val.clusterDim.z = 1;
    ++cfg->numAttrs;
  }
  if (programmatic) {
    attr[cfg->numAttrs].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[cfg->numAttrs].val.programmaticStreamSerializationAllowed = 1;
    ++cfg->numAttrs;
  }
}

cudaError_t lmhead_pair_max_clusters(int sm_count, int mc, int* clusters) {
  cudaError_t e = pair_opt_in<HF_BF16, false>();
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[2];
  pair_config(&cfg, attr, sm_count / (2 * mc), pair_threads<HF_BF16>(), nullptr, false, true, mc);
  int n = 0;
  e = cudaOccupancyMaxActiveClusters(&n, lmhead_pair_kernel<HF_BF16, false>, &cfg);
  if (e != cudaSuccess) return e;
  *clusters = n < 1 ? 1 : n;
  return cudaSuccess;
}

template <int HF, bool VERIFY>
static cudaError_t launch_pair(const PairTokenMaps& tmH, const CUtensorMap& tmW, const PairQuantMaps& tmQ,
                               const PairTokenMaps& tmL, const TcArgs& a, cudaStream_t st) {
  cudaError_t e = pair_opt_in<HF, VERIFY>();
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[2];
  const int ppc = plan_mc(a.plan) * plan_vc(a.plan);  // pairs per cluster
  if (a.plan.G2 > 0) {
    // clusters of two pairs and the spill launch of single pairs behind them
    // (the header's vocabulary split assumes both run)
    if (!pair_cluster<HF>() || ppc != 2) return cudaErrorInvalidValue;
    TcArgs main = a;
    main.plan.role = 0;
    pair_config(&cfg, attr, a.plan.G, pair_threads<HF>(), st, true, true, 2);
    e = cudaLaunchKernelEx(&cfg, lmhead_pair_kernel<HF, VERIFY>, tmH, tmW, tmQ, tmL, main);
    if (e != cudaSuccess) return e;
    TcArgs side = a;
    side.plan.role = 1;
    side.plan.G = a.plan.G2;
    side.plan.mc = 1;
    side.plan.vc = 1;
    side.plan.cpu = SPILL_UNIT_SLOTS;
    pair_config(&cfg, attr, side.plan.G, pair_threads<HF>(), st, true, true, 1);
    return cudaLaunchKernelEx(&cfg, lmhead_pair_kernel<HF, VERIFY>, tmH, tmW, tmQ, tmL, side);
  }
  if (!pair_cluster<HF>() && ppc != 1) return cudaErrorInvalidValue;
  pair_config(&cfg, attr, a.plan.G, pair_threads<HF>(), st, true, pair_cluster<HF>(), pair_cluster<HF>() ? ppc : 1);
  return cudaLaunchKernelEx(&cfg, lmhead_pair_kernel<HF, VERIFY>, tmH, tmW, tmQ, tmL, a);
}

cudaError_t launch_lmhead_pair(const PairTokenMaps& tmH, const CUtensorMap& tmW, const PairQuantMaps* tmQ,
                               const PairTokenMaps* tmLo, int hf, const TcArgs& a, cudaStream_t st) {
  const bool verify = a.part_t != nullptr;
  PairQuantMaps none;
  std::memset(&none, 0, sizeof(none));
  const PairQuantMaps& q = tmQ ? *tmQ : none;
  static const PairTokenMaps no_lo = [] {
    PairTokenMaps m;
    std::memset(&m, 0, sizeof(m));
    return m;
  }();
  const PairTokenMaps& lo = tmLo ? *tmLo : no_lo;
  switch (hf) {
    case HF_W8A8:
      if (verify) return cudaErrorInvalidValue;
      return launch_pair<HF_W8A8, false>(tmH, tmW, q, lo, a, st);
    case HF_E4M3X2:
      if (verify || tmLo == nullptr) return cudaErrorInvalidValue;
      return launch_pair<HF_E4M3X2, false>(tmH, tmW, q, lo, a, st);
    case HF_E4M3:
      return verify ? launch_pair<HF_E4M3, true>(tmH, tmW, q, lo, a, st)
                    : launch_pair<HF_E4M3, false>(tmH, tmW, q, lo, a, st);
    case HF_NVFP4:
      return verify ? launch_pair<HF_NVFP4, true>(tmH, tmW, q, lo, a, st)
                    : launch_pair<HF_NVFP4, false>(tmH, tmW, q, lo, a, st);
    default:
      return verify ? launch_pair<HF_BF16, true>(tmH, tmW, q, lo, a, st)
                    : launch_pair<HF_BF16, false>(tmH, tmW, q, lo, a, st);
  }
}

}  // namespace bd
