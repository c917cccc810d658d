// Host-side launchers of the kernels of libbdcommit (internal interface
// between api.cu and the kernel translation units).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "common.cuh"

namespace bd {

struct TauParams {
  float tau[32];
  int T;
};

// a0: compaction of the masked positions of active blocks (App. F slot
// states) and, when `hidden` is not null, packing of their bf16 rows into hc.
// Writes idx[r] = position of compacted row r (ascending positions),
// rowpos[p] = r or -1, hc[r] = hidden[idx[r]] and *n_rows = N.
// Packed row formats. ROWS_E4M3 (W8A8): E4M3 codes (ldc in bytes, a multiple
// of 8) quantised per row, tok_scale[r] = row r's dequantisation scale.
// ROWS_F16_POW2 (heads decoded to f16 in the LM head): f16 rows (ldc in
// elements) holding the bf16 values times 2^s_r, s_r chosen so the row's
// largest magnitude lands in [2^14, 2^15), tok_scale[r] = 2^-s_r (exact).
// ROWS_E4M3X2 (E4M3 heads on the 8-bit tensor path, W8A16): each bf16 row,
// scaled by a power of two 2^s so its largest magnitude lies in [128, 256),
// as two E4M3 terms hi + lo (hi rows at hc, lo rows at hc + P * ldc, ldc in
// bytes, a multiple of 16), exact for every element of at least 2^-10 of the
// row's largest; tok_scale[r] = 2^-s.
enum : int { ROWS_BF16 = 0, ROWS_E4M3 = 1, ROWS_F16_POW2 = 2, ROWS_E4M3X2 = 3 };
// n_rows: the workspace header (N and the LM head's plan for N, HDR_* words of
// common.cuh), written by the CTA that holds the last position.
cudaError_t launch_prep_rows(const uint8_t* pos_masked, const uint8_t* block_flags, int P, int block_len,
                             const void* hidden, int64_t ld, int d, void* hc, int64_t ldc, int* idx, int* rowpos,
                             int* n_rows, int sm_count, cudaStream_t st, const BandPlan& plan,
                             float* tok_scale = nullptr, int row_format = ROWS_BF16, uint32_t* status = nullptr);

// Decodes FP8 e4m3 weight codes to bf16 (exact), row by row: out[v] = code(w[v]).
cudaError_t launch_dequant_e4m3(const uint8_t* w, int64_t ldw, int V, int d, void* out, int64_t ldo,
                                int sm_count, cudaStream_t st);

// Decodes NVFP4 rows to bf16 (exact: every E2M1 x E4M3 product is a bf16):
// out[v][k] = e2m1(nibble k of codes[v]) * e4m3(bs[v][k / 16]).
cudaError_t launch_dequant_nvfp4(const uint8_t* codes, int64_t ldw, const uint8_t* bs, int64_t ldbs, int V, int d,
                                 void* out, int64_t ldo, int sm_count, cudaStream_t st);

// a1+a2 on the tensor cores: tcgen05 LM-head GEMM with the online softmax
// epilogue. tmA describes hc [P, d] bf16, tmB the head [V, d] bf16.
struct TcArgs {
  const int* n_rows;
  const float* wscale;  // [V] or nullptr
  int V, d, P, mask_id;
  BandPlan plan;
  float* part_m;
  float* part_s;
  int* part_a;
  uint32_t* status;
  // verification path only (part_t != nullptr selects it): the draft token of
  // each row (-1: none), and per partial the entropy accumulator t and the
  // draft token's logit (-inf where the part does not hold it)
  const int* draft_row = nullptr;
  float* part_t = nullptr;
  float* part_x = nullptr;
  // W8A8 only: the dequantisation scale of each packed token row
  const float* tok_scale = nullptr;
  // L2 eviction priorities (L2_EVICT_*) of the head tiles and of the token rows
  int l2_head = L2_EVICT_FIRST;
  int l2_rows = L2_EVICT_LAST;
};
constexpr int TC_BM = 128;
constexpr int TC_BN = 256;
constexpr int TC_BK = 64;
constexpr int TC_THREADS = 192;
size_t tc_smem_bytes(int stages);
cudaError_t launch_lmhead_tc(const CUtensorMap& tmA, const CUtensorMap& tmB, const TcArgs& a, int stages,
                             cudaStream_t st);

// a1+a2 on a CTA pair (tcgen05 cta_group::2), vocabulary on the MMA M side.
// tmH.m[i] describes hc [P, d] bf16 with 64-column boxes of 16 * (i + 1) rows
// (one per possible half token group), tmW the head [V, d] bf16 with 64 x 64
// boxes (64 rows: half of a CTA's head rows, see the kernel). plan.G = runners
// (clusters of plan.mc CTA pairs), plan.BM = 0, plan.cpu = 2.
struct PairTokenMaps {
  CUtensorMap m[16];  // box heights 8, 16, ..., 128 rows: m[h / 8 - 1]
};
// Head formats of the pair kernel: bf16 rows staged as they are, or E4M3 /
// NVFP4 codes decoded to bf16 inside the kernel (codes: [V, ld] bytes with
// 128 x 128-byte SW128 boxes; NVFP4 block scales: [V, block_ld] bytes with
// 16 x 128-byte boxes).
// HF_W8A8: E4M3 head and E4M3 token rows (per-row scales), multiplied with
// tcgen05.mma kind::f8f6f4 (the W8A8 variant of the precision lever).
// HF_E4M3X2: E4M3 head times bf16 token rows packed as two E4M3 terms
// (ROWS_E4M3X2), both multiplied on kind::f8f6f4 into one accumulator (W8A16).
enum : int { HF_BF16 = 0, HF_E4M3 = 1, HF_NVFP4 = 2, HF_W8A8 = 3, HF_E4M3X2 = 4 };
struct PairQuantMaps {
  CUtensorMap codes;
  CUtensorMap scales;
};
size_t pair_smem_bytes();
// CTA-pair clusters of mc pairs (clusters of 2 * mc CTAs) that fit on the device at once.
cudaError_t lmhead_pair_max_clusters(int sm_count, int mc, int* clusters);
// hf: HF_BF16 (tmW describes the bf16 head; tmQ unused, may be null) or
// HF_E4M3 / HF_NVFP4 (tmQ describes the codes, and the NVFP4 block scales;
// tmW unused). E4M3 and NVFP4 need the TcArgs row scale wscale.
// tmLo: the lo-term maps of HF_E4M3X2 (same boxes as tmH), else may be null.
cudaError_t launch_lmhead_pair(const PairTokenMaps& tmH, const CUtensorMap& tmW, const PairQuantMaps* tmQ,
                               const PairTokenMaps* tmLo, int hf, const TcArgs& a, cudaStream_t st);

// a1+a2 with fp32 FMA on the CUDA cores (exact fp32 path; any dtype combo).
struct SimtArgs {
  const void* hidden;
  int64_t ldh;
  int hdtype;  // BD_F32 / BD_BF16
  const void* w;
  int64_t ldw;
  int wdtype;  // BD_F32 / BD_BF16 / BD_E4M3 / BD_NVFP4
  const uint8_t* wbs;  // BD_NVFP4 block scales [V, ldbs]
  int64_t ldbs;
  const float* wscale;
  const int* idx;
  const int* n_rows;
  int V, d, P, mask_id;
  BandPlan plan;
  float* part_m;
  float* part_s;
  int* part_a;
  const int* draft_row = nullptr;  // verification path, as in TcArgs
  float* part_t = nullptr;
  float* part_x = nullptr;
};
constexpr int SIMT_BM = 32;
constexpr int SIMT_BN = 64;
cudaError_t launch_lmhead_simt(const SimtArgs& a, cudaStream_t st);

// a3+a4: merge of the partials per row, then the threshold commit with the
// per-block top-1 fallback for every tau of the grid.
struct CommitArgs {
  const uint8_t* pos_masked;
  const uint8_t* block_flags;
  const int* rowpos;
  const int* n_rows;
  BandPlan plan;
  int P;
  const float* part_m;
  const float* part_s;
  const int* part_a;
  int n_blocks, n_slots, block_len;
  TauParams taus;
  int32_t* out_tokens;
  float* out_conf;
  uint32_t* out_commit;
  int32_t* out_counts;
  uint32_t* status = nullptr;  // device status word (index checks of the bounds-checked build)
  // vocabulary-parallel split: MERGE_EMIT writes each position's merged
  // partial (token id + vocab_offset; -inf / 0 / -1 where nothing is
  // predicted) to emit_*; MERGE_GATHERED reads n_parts partials per position
  // from part_* laid out [n_parts, P] (position-indexed, no compaction)
  int vocab_offset = 0;
  int n_parts = 0;
  float* emit_m = nullptr;
  float* emit_s = nullptr;
  int* emit_a = nullptr;
};
enum : int { MERGE_ROWS = 0, MERGE_EMIT = 1, MERGE_GATHERED = 2 };
cudaError_t launch_merge_commit(const CommitArgs& a, cudaStream_t st, int mode = MERGE_ROWS);

// Verification path (speculative decoding, typical acceptance). Rows are
// r = q * (n_draft + 1) + i; row i < n_draft of request q verifies draft
// token draft[q * n_draft + i], the last row of a request gives its bonus token.
// Prep: idx[r] = r, draft_row[r] = that draft token or -1, and the workspace
// header n_rows (R and the LM head's plan for R rows, HDR_* words of common.cuh).
cudaError_t launch_prep_verify(const int32_t* draft, int n_req, int n_draft, int* idx, int* draft_row, int* n_rows,
                               const BandPlan& plan, cudaStream_t st);

struct VerifyArgs {
  const int* draft_row;
  const int* n_rows;
  BandPlan plan;
  int P;  // rows
  const float* part_m;
  const float* part_s;
  const int* part_a;
  const float* part_t;
  const float* part_x;
  int n_req, n_draft, E;
  float eps[31];
  float sqrt_eps[31];
  int32_t* out_tokens;
  float* out_p_draft;
  float* out_entropy;
  uint32_t* out_accept;
  int32_t* out_accepted;
};
cudaError_t launch_merge_verify(const VerifyArgs& a, cudaStream_t st);

// One CTA that runs the bounded mbarrier wait on a barrier nothing completes
// (failure-detection self-test): sets DEV_TIMEOUT in *status after the limit.
cudaError_t launch_timeout_selftest(uint32_t* status, cudaStream_t st);

}  // namespace bd
