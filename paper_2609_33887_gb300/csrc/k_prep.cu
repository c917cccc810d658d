// Preparation kernels of the commit step: compaction of the still-masked
// positions of active blocks, packing of their hidden rows, and the FP8 e4m3
// -> bf16 weight decode of the precision lever.
#include "kernels.h"

namespace bd {

// ---------------------------------------------------------------------------
// Compaction (one CTA). Only masked positions of active blocks need a
// prediction (App. F: the accept threshold resolves positions of active
// blocks). Rows keep ascending position order, so the masked positions of a
// block are consecutive rows.
// ---------------------------------------------------------------------------
constexpr int COMPACT_THREADS = 1024;
constexpr int COMPACT_ITEMS = 8;

__global__ void __launch_bounds__(COMPACT_THREADS) compact_kernel(const uint8_t* __restrict__ pos_masked,
                                                                  const uint8_t* __restrict__ block_flags,
                                                                  int P, int block_len, int* __restrict__ idx,
                                                                  int* __restrict__ rowpos,
                                                                  int* __restrict__ n_rows) {
  __shared__ int warp_tot[COMPACT_THREADS / 32];
  __shared__ int carry_s;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) carry_s = 0;
  __syncthreads();
  for (int base = 0; base < P; base += COMPACT_THREADS * COMPACT_ITEMS) {
    const int p0 = base + tid * COMPACT_ITEMS;
    uint32_t live = 0;
    int cnt = 0;
#pragma unroll
    for (int i = 0; i < COMPACT_ITEMS; ++i) {
      int p = p0 + i;
      if (p < P && pos_masked[p] != 0 && (block_flags[p / block_len] & 1u)) {
        live |= 1u << i;
        ++cnt;
      }
    }
    int incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int t = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += t;
    }
    if (lane == 31) warp_tot[warp] = incl;
    __syncthreads();
    if (warp == 0) {
      int w = warp_tot[lane];
      int wi = w;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        int t = __shfl_up_sync(0xffffffffu, wi, o);
        if (lane >= o) wi += t;
      }
      warp_tot[lane] = wi - w;  // exclusive prefix of the warp totals
    }
    __syncthreads();
    const int carry = carry_s;
    int r = carry + warp_tot[warp] + incl - cnt;
#pragma unroll
    for (int i = 0; i < COMPACT_ITEMS; ++i) {
      int p = p0 + i;
      if (p < P) {
        if (live & (1u << i)) {
          idx[r] = p;
          rowpos[p] = r;
          ++r;
        } else {
          rowpos[p] = -1;
        }
      }
    }
    __syncthreads();
    if (tid == COMPACT_THREADS - 1) carry_s = r;  // last thread ends at the chunk total
    __syncthreads();
  }
  if (tid == 0) *n_rows = carry_s;
}

cudaError_t launch_compact(const uint8_t* pos_masked, const uint8_t* block_flags, int P, int block_len, int* idx,
                           int* rowpos, int* n_rows, cudaStream_t st) {
  compact_kernel<<<1, COMPACT_THREADS, 0, st>>>(pos_masked, block_flags, P, block_len, idx, rowpos, n_rows);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Row packing: hc[r, :] = hidden[idx[r], :] for r < N (bf16, 16-byte vectors
// when the width allows).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) pack_rows_bf16_kernel(const __nv_bfloat16* __restrict__ hidden, int64_t ld,
                                                             int d, const int* __restrict__ idx,
                                                             const int* __restrict__ n_rows,
                                                             __nv_bfloat16* __restrict__ hc, int64_t ldc) {
  const int N = *n_rows;
  const int nvec = d / 8;
  for (int r = blockIdx.x; r < N; r += gridDim.x) {
    const __nv_bfloat16* src = hidden + static_cast<int64_t>(idx[r]) * ld;
    __nv_bfloat16* dst = hc + static_cast<int64_t>(r) * ldc;
    const uint4* s4 = reinterpret_cast<const uint4*>(src);
    uint4* d4 = reinterpret_cast<uint4*>(dst);
    for (int i = threadIdx.x; i < nvec; i += blockDim.x) d4[i] = __ldg(s4 + i);
    for (int i = nvec * 8 + threadIdx.x; i < d; i += blockDim.x) dst[i] = src[i];
  }
}

cudaError_t launch_pack_rows_bf16(const void* hidden, int64_t ld, int d, const int* idx, const int* n_rows, int P,
                                  void* hc, int64_t ldc, int sm_count, cudaStream_t st) {
  int grid = sm_count * 8;
  if (grid > P) grid = P;
  if (grid < 1) grid = 1;
  pack_rows_bf16_kernel<<<grid, 256, 0, st>>>(static_cast<const __nv_bfloat16*>(hidden), ld, d, idx, n_rows,
                                              static_cast<__nv_bfloat16*>(hc), ldc);
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

__global__ void __launch_bounds__(256) dequant_e4m3_kernel(const uint8_t* __restrict__ w, int64_t ldw, int V, int d,
                                                           __nv_bfloat16* __restrict__ out, int64_t ldo) {
  // one thread per 16 codes of a row; rows are 16-byte aligned (ldw % 16 == 0)
  const int per_row = (d + 15) / 16;
  const int64_t total = static_cast<int64_t>(V) * per_row;
  for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < total;
       t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int v = static_cast<int>(t / per_row);
    const int c0 = static_cast<int>(t % per_row) * 16;
    const uint8_t* src = w + static_cast<int64_t>(v) * ldw + c0;
    __nv_bfloat16* dst = out + static_cast<int64_t>(v) * ldo + c0;
    if (c0 + 16 <= d) {
      uint4 q = __ldg(reinterpret_cast<const uint4*>(src));
      const uint16_t* q2 = reinterpret_cast<const uint16_t*>(&q);
      uint4 o0, o1;
      o0.x = e4m3x2_to_bf16x2(q2[0]);
      o0.y = e4m3x2_to_bf16x2(q2[1]);
      o0.z = e4m3x2_to_bf16x2(q2[2]);
      o0.w = e4m3x2_to_bf16x2(q2[3]);
      o1.x = e4m3x2_to_bf16x2(q2[4]);
      o1.y = e4m3x2_to_bf16x2(q2[5]);
      o1.z = e4m3x2_to_bf16x2(q2[6]);
      o1.w = e4m3x2_to_bf16x2(q2[7]);
      // ldo % 8 == 0 and c0 % 16 == 0 keep both stores 16-byte aligned
      reinterpret_cast<uint4*>(dst)[0] = o0;
      reinterpret_cast<uint4*>(dst)[1] = o1;
    } else {
      for (int i = 0; c0 + i < d; ++i) {
        uint32_t b2 = e4m3x2_to_bf16x2(static_cast<uint16_t>(src[i]));
        dst[i] = *reinterpret_cast<__nv_bfloat16*>(&b2);
      }
    }
  }
}

cudaError_t launch_dequant_e4m3(const uint8_t* w, int64_t ldw, int V, int d, void* out, int64_t ldo, int sm_count,
                                cudaStream_t st) {
  int grid = sm_count * 16;
  dequant_e4m3_kernel<<<grid, 256, 0, st>>>(w, ldw, V, d, static_cast<__nv_bfloat16*>(out), ldo);
  return cudaGetLastError();
}

}  // namespace bd
