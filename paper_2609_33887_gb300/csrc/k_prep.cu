// Preparation kernels of the commit step: compaction of the still-masked
// positions of active blocks, packing of their hidden rows, and the FP8 e4m3
// and NVFP4 -> bf16 weight decodes of the precision levers.
#include "checks.h"
#include "kernels.h"

namespace bd {

// ---------------------------------------------------------------------------
// Compaction and row packing in one launch. Only masked positions of active
// blocks need a prediction (App. F: the accept threshold resolves positions of
// active blocks). Rows keep ascending position order, so the masked positions
// of a block are consecutive rows.
//
// CTA c owns positions [c*chunk, (c+1)*chunk). It counts the live positions
// before its chunk itself (no inter-CTA communication), scans its chunk, writes
// idx / rowpos for it, copies the hidden rows of its live positions into hc
// (bf16 tensor-core paths) and, if it holds the last position, writes N.
// ---------------------------------------------------------------------------
constexpr int PREP_THREADS = 256;

__device__ __forceinline__ int live_at(const uint8_t* __restrict__ pos_masked, const uint8_t* __restrict__ block_flags,
                                       int p, int block_len) {
  return (pos_masked[p] != 0 && (block_flags[p / block_len] & 1u)) ? 1 : 0;
}

__device__ __forceinline__ int block_sum(int v, int* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  if (lane == 0) red[warp] = v;
  __syncthreads();
  int t = 0;
  for (int w = 0; w < PREP_THREADS / 32; ++w) t += red[w];
  __syncthreads();
  return t;
}

// Two float32 values -> two E4M3 codes (round to nearest even, saturating at
// 448), `lo` in the low byte.
__device__ __forceinline__ uint32_t f32x2_to_e4m3x2(float lo, float hi) {
  uint16_t r;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(hi), "f"(lo));
  return r;
}

// f16x2 bit pattern -> two float32 values (exact).
__device__ __forceinline__ float2 f16x2_bits_to_float2(uint32_t h2) {
  return __half22float2(*reinterpret_cast<const __half2*>(&h2));
}

template <int FMT>  // the packed row format (ROWS_*); one instantiation per format
__global__ void __launch_bounds__(PREP_THREADS) prep_rows_kernel(
    const uint8_t* __restrict__ pos_masked, const uint8_t* __restrict__ block_flags, int P, int block_len, int chunk,
    const __nv_bfloat16* __restrict__ hidden, int64_t ld, int d, __nv_bfloat16* __restrict__ hc, int64_t ldc,
    int* __restrict__ idx, int* __restrict__ rowpos, int* __restrict__ n_rows, float* __restrict__ tok_scale,
    uint32_t* __restrict__ status, BandPlan plan) {
  __shared__ int red[PREP_THREADS / 32];
  __shared__ int warp_excl[PREP_THREADS / 32];
  __shared__ int rows_s[2048];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  griddep_launch_dependents();  // every CTA of this grid is resident once all have got here
  const int p0 = blockIdx.x * chunk;
  const int p1 = min(P, p0 + chunk);

  // 1. live positions before this chunk
  int before = 0;
  for (int p = tid; p < p0; p += PREP_THREADS) before += live_at(pos_masked, block_flags, p, block_len);
  const int prefix = block_sum(before, red);

  // 2. exclusive scan of the chunk: thread t takes `per` consecutive positions
  const int per = (chunk + PREP_THREADS - 1) / PREP_THREADS;
  const int q0 = p0 + tid * per;
  int cnt = 0;
  for (int i = 0; i < per; ++i) {
    const int p = q0 + i;
    if (p < p1) cnt += live_at(pos_masked, block_flags, p, block_len);
  }
  int incl = cnt;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  if (lane == 31) warp_excl[warp] = incl;
  __syncthreads();
  if (tid == 0) {
    int run = 0;
    for (int w = 0; w < PREP_THREADS / 32; ++w) {
      const int t = warp_excl[w];
      warp_excl[w] = run;
      run += t;
    }
    red[0] = run;  // live positions of the chunk
  }
  __syncthreads();
  const int local_total = red[0];
  int r = prefix + warp_excl[warp] + incl - cnt;
  for (int i = 0; i < per; ++i) {
    const int p = q0 + i;
    if (p < p1) {
      if (live_at(pos_masked, block_flags, p, block_len)) {
        if (index_ok(r, P, status)) idx[r] = p;
        rowpos[p] = r;
        if (r - prefix < 2048) rows_s[r - prefix] = p;
        ++r;
      } else {
        rowpos[p] = -1;
      }
    }
  }
  // The CTA holding the last position knows N: its warp 0 writes N and the
  // plan for it into the header the later kernels read, while the CTA's other
  // warps pack its rows (the plan's evaluation stays off the packing's path).
  const bool header_warp = p1 == P && warp == 0;
  if (hidden == nullptr) {
    if (header_warp) plan_write_header(plan, prefix + local_total, n_rows);
    return;
  }
  __syncthreads();
  if (header_warp) {
    plan_write_header(plan, prefix + local_total, n_rows);
    return;
  }
  // the packing warps: all of them, or all but warp 0 in the header's CTA
  const int w0 = p1 == P ? 1 : 0;
  const int n_pack = PREP_THREADS / 32 - w0;

  const int nvec = d / 8;
  if constexpr (FMT == ROWS_F16_POW2) {
    // 3''. f16 rows for an LM head whose operands are f16: row r holds
    // h * 2^s with s = 15 - e for max |h| in [2^(e-1), 2^e) (so the largest
    // magnitude lands in [2^14, 2^15) and every bf16 value at or above 2^-14
    // after scaling is exact in f16), s at most 126 so 2^-s stays a normal
    // float; tok_scale = 2^-s, 0 for an all-zero row.
    for (int i = warp - w0; i < local_total; i += n_pack) {
      if (!index_ok(prefix + i, P, status)) continue;
      const int p = i < 2048 ? rows_s[i] : idx[prefix + i];
      const __nv_bfloat16* src = hidden + static_cast<int64_t>(p) * ld;
      const uint4* s4 = reinterpret_cast<const uint4*>(src);
      float amax = 0.f;
#pragma unroll 4
      for (int v = lane; v < nvec; v += 32) {
        const uint4 q = __ldg(s4 + v);
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[j]));
          amax = fmaxf(amax, fmaxf(fabsf(f.x), fabsf(f.y)));
        }
      }
      for (int e = nvec * 8 + lane; e < d; e += 32) amax = fmaxf(amax, fabsf(__bfloat162float(src[e])));
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
      // biased exponent E of amax: amax in [2^(E-127), 2^(E-126)) for E > 0,
      // so s = 15 - (E - 126); E = 0 (zero or below 2^-126) takes the cap
      const int E = static_cast<int>(__float_as_uint(amax) >> 23);
      const int sh = amax > 0.f ? min(141 - E, 126) : 0;
      const float up = __uint_as_float(static_cast<uint32_t>(sh + 127) << 23);  // 2^s, exact
      __half* dst = reinterpret_cast<__half*>(hc) + static_cast<int64_t>(prefix + i) * ldc;
      uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll 4
      for (int v = lane; v < nvec; v += 32) {
        const uint4 q = __ldg(s4 + v);
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
        uint32_t o[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[j]));
          const __half2 h2 = __floats2half2_rn(f.x * up, f.y * up);
          o[j] = *reinterpret_cast<const uint32_t*>(&h2);
        }
        d4[v] = make_uint4(o[0], o[1], o[2], o[3]);
      }
      for (int e = nvec * 8 + lane; e < d; e += 32) dst[e] = __float2half_rn(__bfloat162float(src[e]) * up);
      if (lane == 0) tok_scale[prefix + i] = amax > 0.f ? __uint_as_float(static_cast<uint32_t>(127 - sh) << 23) : 0.f;
    }
    return;
  }
  if constexpr (FMT == ROWS_E4M3X2) {
    // 3'''. bf16 rows as two E4M3 terms for an E4M3 head on the 8-bit tensor
    // path (W8A16): row r is scaled by 2^s so that its largest magnitude lands
    // in [128, 256) (s = 134 - E for the biased exponent E of max |h|, between
    // -126 and 126 so 2^s and 2^-s stay normal floats; exact), then
    // y = h * 2^s becomes hi = e4m3(y) and lo = e4m3(y - hi), both rounded to
    // nearest even. y has at most 8 significant bits and y - hi (exact in
    // float32) at most 4 more, so hi + lo == y exactly whenever |y| >= 2^-2,
    // i.e. for every element of at least 2^-10 times the row's largest; a
    // smaller element is off by at most 2^-10 (half the smallest E4M3 step),
    // 2^-17 of the row's largest. hi rows at hc, lo rows at hc + P * ldc (ldc
    // in bytes); tok_scale = 2^-s (0 for an all-zero row).
    uint8_t* hq = reinterpret_cast<uint8_t*>(hc);
    uint8_t* lq = hq + static_cast<int64_t>(P) * ldc;
    // rows of up to 32 * RC vectors (5120 bf16) are read once, into
    // registers: every lane's loads of the row are in flight together
    constexpr int RC = 20;
    const bool cached = nvec <= 32 * RC;
    auto amax_of = [](const uint4& q) {
      const uint32_t w[4] = {q.x, q.y, q.z, q.w};
      float m = 0.f;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[j]));
        m = fmaxf(m, fmaxf(fabsf(f.x), fabsf(f.y)));
      }
      return m;
    };
    for (int i = warp - w0; i < local_total; i += n_pack) {
      if (!index_ok(prefix + i, P, status)) continue;
      const int p = i < 2048 ? rows_s[i] : idx[prefix + i];
      const __nv_bfloat16* src = hidden + static_cast<int64_t>(p) * ld;
      const uint4* s4 = reinterpret_cast<const uint4*>(src);
      uint4 qc[RC];
      float amax = 0.f;
      if (cached) {
#pragma unroll
        for (int k = 0; k < RC; ++k) {
          const int v = lane + 32 * k;
          qc[k] = v < nvec ? __ldg(s4 + v) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int k = 0; k < RC; ++k) amax = fmaxf(amax, amax_of(qc[k]));
      } else {
#pragma unroll 4
        for (int v = lane; v < nvec; v += 32) amax = fmaxf(amax, amax_of(__ldg(s4 + v)));
      }
      for (int e = nvec * 8 + lane; e < d; e += 32) amax = fmaxf(amax, fabsf(__bfloat162float(src[e])));
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
      const int E = static_cast<int>(__float_as_uint(amax) >> 23);
      const int sh = amax > 0.f ? max(min(134 - E, 126), -126) : 0;
      const float up = __uint_as_float(static_cast<uint32_t>(sh + 127) << 23);  // 2^s, exact
      uint8_t* dh = hq + static_cast<int64_t>(prefix + i) * ldc;
      uint8_t* dl = lq + static_cast<int64_t>(prefix + i) * ldc;
      // vector v of the row: eight elements as eight hi and eight lo codes
      auto convert_store = [&](const uint4& q, int v) {
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
        uint32_t oh[2], ol[2];
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          uint32_t h4 = 0, l4 = 0;
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[2 * j + u]));
            const float y0 = f.x * up, y1 = f.y * up;
            const uint32_t h2 = f32x2_to_e4m3x2(y0, y1);
            const float2 back = f16x2_bits_to_float2(e4m3x2_to_f16x2(h2));
            const uint32_t l2 = f32x2_to_e4m3x2(y0 - back.x, y1 - back.y);
            h4 |= h2 << (16 * u);
            l4 |= l2 << (16 * u);
          }
          oh[j] = h4;
          ol[j] = l4;
        }
        *reinterpret_cast<uint2*>(dh + 8 * v) = make_uint2(oh[0], oh[1]);
        *reinterpret_cast<uint2*>(dl + 8 * v) = make_uint2(ol[0], ol[1]);
      };
      if (cached) {
#pragma unroll
        for (int k = 0; k < RC; ++k) {
          const int v = lane + 32 * k;
          if (v < nvec) convert_store(qc[k], v);
        }
      } else {
#pragma unroll 4
        for (int v = lane; v < nvec; v += 32) convert_store(__ldg(s4 + v), v);
      }
      for (int e = nvec * 8 + lane; e < d; e += 32) {
        const float y = __bfloat162float(src[e]) * up;
        const uint32_t h2 = f32x2_to_e4m3x2(y, 0.f);
        const float back = f16x2_bits_to_float2(e4m3x2_to_f16x2(h2)).x;
        dh[e] = static_cast<uint8_t>(h2 & 0xFFu);
        dl[e] = static_cast<uint8_t>(f32x2_to_e4m3x2(y - back, 0.f) & 0xFFu);
      }
      if (lane == 0) tok_scale[prefix + i] = amax > 0.f ? __uint_as_float(static_cast<uint32_t>(127 - sh) << 23) : 0.f;
    }
    return;
  }
  if constexpr (FMT == ROWS_E4M3) {
    // 3'. W8A8: quantise the chunk's live rows to E4M3 with one scale per row,
    // one warp per row: a = max |h|, inv = 448 / a, code = e4m3(h * inv) (round
    // to nearest even, saturating), scale = a / 448; an all-zero row gets codes
    // 0 and scale 0. Each float32 step is one correctly rounded operation.
    uint8_t* hq = reinterpret_cast<uint8_t*>(hc);  // ldc counts bytes here
    for (int i = warp - w0; i < local_total; i += n_pack) {
      if (!index_ok(prefix + i, P, status)) continue;
      const int p = i < 2048 ? rows_s[i] : idx[prefix + i];
      const __nv_bfloat16* src = hidden + static_cast<int64_t>(p) * ld;
      const uint4* s4 = reinterpret_cast<const uint4*>(src);
      float amax = 0.f;
#pragma unroll 4
      for (int v = lane; v < nvec; v += 32) {
        const uint4 q = __ldg(s4 + v);
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[j]));
          amax = fmaxf(amax, fmaxf(fabsf(f.x), fabsf(f.y)));
        }
      }
      for (int e = nvec * 8 + lane; e < d; e += 32) amax = fmaxf(amax, fabsf(__bfloat162float(src[e])));
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
      const float inv = amax > 0.f ? __fdiv_rn(448.f, amax) : 0.f;
      uint8_t* dst = hq + static_cast<int64_t>(prefix + i) * ldc;
#pragma unroll 4
      for (int v = lane; v < nvec; v += 32) {
        const uint4 q = __ldg(s4 + v);
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
        uint32_t out[2];
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          const float2 f0 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[2 * j]));
          const float2 f1 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[2 * j + 1]));
          out[j] = f32x2_to_e4m3x2(__fmul_rn(f0.x, inv), __fmul_rn(f0.y, inv)) |
                   (f32x2_to_e4m3x2(__fmul_rn(f1.x, inv), __fmul_rn(f1.y, inv)) << 16);
        }
        *reinterpret_cast<uint2*>(dst + 8 * v) = make_uint2(out[0], out[1]);
      }
      for (int e = nvec * 8 + lane; e < d; e += 32)
        dst[e] = static_cast<uint8_t>(f32x2_to_e4m3x2(__fmul_rn(__bfloat162float(src[e]), inv), 0.f) & 0xFFu);
      if (lane == 0) tok_scale[prefix + i] = amax > 0.f ? __fdiv_rn(amax, 448.f) : 0.f;
    }
    return;
  }

  // 3. copy the chunk's live rows, one warp per row, 16-byte vectors
  for (int i = warp - w0; i < local_total; i += n_pack) {
    if (!index_ok(prefix + i, P, status)) continue;
    const int p = i < 2048 ? rows_s[i] : idx[prefix + i];
    const __nv_bfloat16* src = hidden + static_cast<int64_t>(p) * ld;
    __nv_bfloat16* dst = hc + static_cast<int64_t>(prefix + i) * ldc;
    const uint4* s4 = reinterpret_cast<const uint4*>(src);
    uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll 4
    for (int v = lane; v < nvec; v += 32) d4[v] = __ldg(s4 + v);
    for (int e = nvec * 8 + lane; e < d; e += 32) dst[e] = src[e];
  }
}

int prep_chunk(int P, int sm_count) {
  int chunk = (P + 2 * sm_count - 1) / (2 * sm_count);
  chunk = (chunk + 31) / 32 * 32;
  if (chunk < 32) chunk = 32;
  if (chunk > 2048) chunk = 2048;
  return chunk;
}

cudaError_t launch_prep_rows(const uint8_t* pos_masked, const uint8_t* block_flags, int P, int block_len,
                             const void* hidden, int64_t ld, int d, void* hc, int64_t ldc, int* idx, int* rowpos,
                             int* n_rows, int sm_count, cudaStream_t st, const BandPlan& plan, float* tok_scale,
                             int row_format, uint32_t* status) {
  if (row_format != ROWS_BF16 && (tok_scale == nullptr || hc == nullptr)) return cudaErrorInvalidValue;
  const int chunk = prep_chunk(P, sm_count);
  const int grid = (P + chunk - 1) / chunk;
  auto* kern = row_format == ROWS_F16_POW2 ? prep_rows_kernel<ROWS_F16_POW2>
               : row_format == ROWS_E4M3  ? prep_rows_kernel<ROWS_E4M3>
               : row_format == ROWS_E4M3X2 ? prep_rows_kernel<ROWS_E4M3X2>
                                           : prep_rows_kernel<ROWS_BF16>;
  kern<<<grid, PREP_THREADS, 0, st>>>(pos_masked, block_flags, P, block_len, chunk,
                                      static_cast<const __nv_bfloat16*>(hidden), ld, d,
                                      static_cast<__nv_bfloat16*>(hc), ldc, idx, rowpos, n_rows, tok_scale, status,
                                      plan);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Verification rows need no compaction: every row is live. Row
// r = q * (n_draft + 1) + i verifies draft token i of request q (i < n_draft);
// the last row of a request verifies nothing.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) prep_verify_kernel(const int32_t* __restrict__ draft, int n_req, int n_draft,
                                                          int* __restrict__ idx, int* __restrict__ draft_row,
                                                          int* __restrict__ n_rows, BandPlan plan) {
  griddep_launch_dependents();
  const int R = n_req * (n_draft + 1);
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < R; r += gridDim.x * blockDim.x) {
    const int q = r / (n_draft + 1), i = r % (n_draft + 1);
    idx[r] = r;
    draft_row[r] = i < n_draft ? draft[q * n_draft + i] : -1;
  }
  if (blockIdx.x == 0 && threadIdx.x < 32) plan_write_header(plan, R, n_rows);  // N and the plan for it
}

cudaError_t launch_prep_verify(const int32_t* draft, int n_req, int n_draft, int* idx, int* draft_row, int* n_rows,
                               const BandPlan& plan, cudaStream_t st) {
  const int R = n_req * (n_draft + 1);
  int grid = (R + 255) / 256;
  if (grid < 1) grid = 1;
  if (grid > 1024) grid = 1024;
  prep_verify_kernel<<<grid, 256, 0, st>>>(draft, n_req, n_draft, idx, draft_row, n_rows, plan);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// FP8 E4M3 -> bf16. Every e4m3 value (subnormals included) is exactly
// representable in f16 and in bf16, so the decode is exact; the per-row
// scale is applied later, to the fp32 logit.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t e4m3x2_to_bf16x2(uint16_t two) {
  uint32_t h2;
  asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(h2) : "h"(two));
  __half2 h = *reinterpret_cast<__half2*>(&h2);
  float2 f = __half22float2(h);
  __nv_bfloat162 b = __floats2bfloat162_rn(f.x, f.y);
  return *reinterpret_cast<uint32_t*>(&b);
}

// One warp per row (grid-stride over rows). The row is cut into 8-element
// chunks; lane l takes chunks l, l + 32, ..., so every warp load reads 256
// contiguous code bytes and every warp store writes 512 contiguous output
// bytes; four chunks per lane are in flight at once. No index needs a division.
__global__ void __launch_bounds__(256) dequant_e4m3_kernel(const uint8_t* __restrict__ w, int64_t ldw, int V, int d,
                                                           __nv_bfloat16* __restrict__ out, int64_t ldo) {
  const int lane = threadIdx.x & 31;
  const int warps = gridDim.x * (blockDim.x >> 5);
  const int nchunk = (d + 7) / 8;
  for (int v = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); v < V; v += warps) {
    const uint8_t* src_row = w + static_cast<int64_t>(v) * ldw;
    __nv_bfloat16* dst_row = out + static_cast<int64_t>(v) * ldo;
    for (int c0 = lane; c0 < nchunk; c0 += 128) {
      uint2 q[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int c = c0 + 32 * u;
        // 8 codes at 8c: inside the row (ldw % 16 == 0 and ldw >= d)
        if (c < nchunk) q[u] = __ldg(reinterpret_cast<const uint2*>(src_row + 8 * c));
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int c = c0 + 32 * u;
        if (c >= nchunk) break;
        uint4 o;
        o.x = e4m3x2_to_bf16x2(static_cast<uint16_t>(q[u].x & 0xFFFFu));
        o.y = e4m3x2_to_bf16x2(static_cast<uint16_t>(q[u].x >> 16));
        o.z = e4m3x2_to_bf16x2(static_cast<uint16_t>(q[u].y & 0xFFFFu));
        o.w = e4m3x2_to_bf16x2(static_cast<uint16_t>(q[u].y >> 16));
        __nv_bfloat16* dst = dst_row + 8 * c;
        if (8 * c + 8 <= d) {
          *reinterpret_cast<uint4*>(dst) = o;  // ldo % 8 == 0: 16-byte aligned
        } else {
          const __nv_bfloat16* ov = reinterpret_cast<const __nv_bfloat16*>(&o);
#pragma unroll
          for (int j = 0; j < 8; ++j)
            if (8 * c + j < d) dst[j] = ov[j];
        }
      }
    }
  }
}

cudaError_t launch_dequant_e4m3(const uint8_t* w, int64_t ldw, int V, int d, void* out, int64_t ldo, int sm_count,
                                cudaStream_t st) {
  int grid = sm_count * 8;
  dequant_e4m3_kernel<<<grid, 256, 0, st>>>(w, ldw, V, d, static_cast<__nv_bfloat16*>(out), ldo);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// NVFP4 -> bf16. An E2M1 code is 1 sign bit, 2 exponent bits (bias 1) and 1
// mantissa bit; its value (1 + m/2) * 2^(e-1), or m/2 for e = 0, is built
// directly as a binary32 bit pattern. Times the E4M3 block scale the product
// has at most 5 significant bits, so the bf16 result is exact; the per-row
// scale is applied later, to the fp32 logit.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float e2m1_value(uint32_t c) {
  const uint32_t e = (c >> 1) & 3u, m = c & 1u;
  const uint32_t mag = e == 0 ? (m ? 0x3F000000u : 0u) : (((126u + e) << 23) | (m << 22));
  return __uint_as_float(mag | ((c & 8u) << 28));
}

__device__ __forceinline__ float e4m3_value(uint8_t c) {
  uint32_t h2;
  asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(h2) : "h"(static_cast<uint16_t>(c)));
  return __half2float(__ushort_as_half(static_cast<unsigned short>(h2 & 0xffffu)));
}

// One warp per row (grid-stride over rows). The row is cut into 8-element
// chunks (4 code bytes, 16 output bytes); lane l takes chunks l, l + 32, ...,
// so every warp load reads 128 contiguous code bytes and every warp store
// writes 512 contiguous output bytes; four chunks per lane are in flight at
// once. Chunk c uses block scale c / 2. No index needs a division.
__global__ void __launch_bounds__(256) dequant_nvfp4_kernel(const uint8_t* __restrict__ codes, int64_t ldw,
                                                            const uint8_t* __restrict__ bs, int64_t ldbs, int V,
                                                            int d, __nv_bfloat16* __restrict__ out, int64_t ldo) {
  const int lane = threadIdx.x & 31;
  const int warps = gridDim.x * (blockDim.x >> 5);
  const int nchunk = (d + 7) / 8;
  for (int v = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); v < V; v += warps) {
    const uint8_t* crow = codes + static_cast<int64_t>(v) * ldw;
    const uint8_t* brow = bs + static_cast<int64_t>(v) * ldbs;
    __nv_bfloat16* orow = out + static_cast<int64_t>(v) * ldo;
    for (int c0 = lane; c0 < nchunk; c0 += 128) {
      uint32_t q[4];
      uint8_t sb[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int c = c0 + 32 * u;
        // 4 code bytes at 4c: inside the row (ldw % 16 == 0 and ldw >= ceil(d / 2))
        if (c < nchunk) {
          q[u] = __ldg(reinterpret_cast<const uint32_t*>(crow + 4 * c));
          sb[u] = brow[c >> 1];
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int c = c0 + 32 * u;
        if (c >= nchunk) break;
        const float sc = e4m3_value(sb[u]);
        uint32_t ow[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t byte = (q[u] >> (8 * j)) & 0xFFu;
          __nv_bfloat162 pr = __floats2bfloat162_rn(e2m1_value(byte & 0xFu) * sc, e2m1_value(byte >> 4) * sc);
          ow[j] = *reinterpret_cast<uint32_t*>(&pr);
        }
        __nv_bfloat16* dst = orow + 8 * c;
        if (8 * c + 8 <= d) {
          *reinterpret_cast<uint4*>(dst) = make_uint4(ow[0], ow[1], ow[2], ow[3]);  // ldo % 8 == 0
        } else {
          const __nv_bfloat16* ov = reinterpret_cast<const __nv_bfloat16*>(ow);
#pragma unroll
          for (int j = 0; j < 8; ++j)
            if (8 * c + j < d) dst[j] = ov[j];
        }
      }
    }
  }
}

cudaError_t launch_dequant_nvfp4(const uint8_t* codes, int64_t ldw, const uint8_t* bs, int64_t ldbs, int V, int d,
                                 void* out, int64_t ldo, int sm_count, cudaStream_t st) {
  int grid = sm_count * 8;
  dequant_nvfp4_kernel<<<grid, 256, 0, st>>>(codes, ldw, bs, ldbs, V, d, static_cast<__nv_bfloat16*>(out), ldo);
  return cudaGetLastError();
}

}  // namespace bd
