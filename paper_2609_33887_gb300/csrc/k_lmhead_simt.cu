// LM-head projection + mask-suppressed softmax statistics with fp32 FMA on
// the CUDA cores. This is the exact-fp32 path (fp32 hidden states and head),
// and it accepts bf16 / e4m3 heads too. Same band plan and partial layout as
// the tensor-core kernel, with 32-row m-tiles and 256-entry v-tiles. The
// verification instantiation (VERIFY = true) also carries the entropy
// accumulator and the logit of each row's draft entry.
//
// A CTA of 256 threads computes a 32-row x 64-entry tile in 64-column K
// steps, each step's operands loaded into registers one step ahead: thread t owns
// vocabulary column t % 64 of the tile for rows 8 (t / 64) .. 8 (t / 64) + 7,
// so a small window still spreads over many CTAs (the 32 x 4096 fp32 window:
// 64 v-tiles).
#include <cuda_fp16.h>

#include "bdcommit.h"
#include "kernels.h"

namespace bd {

namespace {

// hidden columns staged per K step: 64, or 32 for the verification
// instantiation (its larger epilogue state leaves fewer registers for the
// step loaded ahead at two CTAs per SM)
template <bool VERIFY>
__host__ __device__ constexpr int kc_of() { return VERIFY ? 32 : 64; }
constexpr int THREADS = 256;
constexpr int ROW_GROUPS = THREADS / SIMT_BN;   // 4 groups of rows
constexpr int RPT = SIMT_BM / ROW_GROUPS;        // 8 rows per thread
constexpr int CPL = SIMT_BN / 32;                // columns a lane scans in the reductions
static_assert(THREADS % SIMT_BN == 0 && SIMT_BM % ROW_GROUPS == 0, "column x row-group split");
static_assert(SIMT_BM == 32, "one row per lane in the reductions");
static_assert((SIMT_BM * 32) % THREADS == 0 && (SIMT_BN * 32) % THREADS == 0, "whole staging rounds");

__device__ __forceinline__ float load_h(const void* p, int64_t i, int dt) {
  if (dt == BD_F32) return static_cast<const float*>(p)[i];
  return __bfloat162float(static_cast<const __nv_bfloat16*>(p)[i]);
}

__device__ __forceinline__ float e4m3_to_float(uint8_t c) {
  uint32_t h2;
  asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(h2) : "h"(static_cast<uint16_t>(c)));
  return __half2float(__ushort_as_half(static_cast<unsigned short>(h2 & 0xffffu)));
}

__device__ __forceinline__ float load_w(const void* p, int64_t i, int dt) {
  if (dt == BD_F32) return static_cast<const float*>(p)[i];
  if (dt == BD_BF16) return __bfloat162float(static_cast<const __nv_bfloat16*>(p)[i]);
  return e4m3_to_float(static_cast<const uint8_t*>(p)[i]);
}

// NVFP4 element (v, k): the E2M1 nibble k of row v (low nibble first) times
// the E4M3 scale of its 16-element block; the value is built from the code's
// bit fields (sign, 2-bit exponent with bias 1, 1-bit mantissa).
__device__ __forceinline__ float load_w_nvfp4(const void* p, const uint8_t* bs, int v, int k, int64_t ldw,
                                              int64_t ldbs) {
  const uint8_t byte = static_cast<const uint8_t*>(p)[static_cast<int64_t>(v) * ldw + k / 2];
  const uint32_t c = (k & 1) ? (byte >> 4) : (byte & 0xFu);
  const uint32_t e = (c >> 1) & 3u, m = c & 1u;
  const uint32_t mag = e == 0 ? (m ? 0x3F000000u : 0u) : (((126u + e) << 23) | (m << 22));
  return __uint_as_float(mag | ((c & 8u) << 28)) * e4m3_to_float(bs[static_cast<int64_t>(v) * ldbs + k / 16]);
}

template <int KC>
struct SimtSmem {
  int rix[SIMT_BM];  // the m-tile's hidden rows (-1 past N)
  float hs[SIMT_BM][KC + 1];
  union {
    float ws[SIMT_BN][KC + 1];         // head tile during the K loop
    float lg[SIMT_BM][SIMT_BN + 1];    // logits of the tile after it
  } u;
  float rm[SIMT_BM], rs[SIMT_BM];
  int ra[SIMT_BM];
  float rt[SIMT_BM], rx[SIMT_BM];  // VERIFY only
  int xd[SIMT_BM];
};

}  // namespace

template <bool VERIFY>
__global__ void __launch_bounds__(THREADS, 2) lmhead_simt_kernel(SimtArgs a) {
  constexpr int KC = kc_of<VERIFY>();
  constexpr int HE = SIMT_BM * KC / THREADS;  // hidden elements a thread stages per step
  constexpr int WE = SIMT_BN * KC / THREADS;  // head elements a thread stages per step
  __shared__ SimtSmem<KC> sm;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int col = tid % SIMT_BN, rg = tid / SIMT_BN;  // this thread's column and row group
  griddep_wait();  // idx and N come from the preceding kernel
  const int n_rows = a.n_rows[HDR_N];

  TileIter it;
  it.init(a.plan, a.n_rows);
  while (it.next_unit()) {
    const int r0 = it.m_tile * SIMT_BM;
    if (tid < SIMT_BM) {
      sm.rix[tid] = r0 + tid < n_rows ? a.idx[r0 + tid] : -1;
      sm.rm[tid] = -INFINITY;
      sm.rs[tid] = 0.f;
      sm.ra[tid] = 0x7fffffff;
      if constexpr (VERIFY) {
        sm.rt[tid] = 0.f;
        sm.rx[tid] = -INFINITY;
        sm.xd[tid] = r0 + tid < n_rows ? a.draft_row[r0 + tid] : -1;
      }
    }
    __syncthreads();
    for (int vt = it.vt; vt < it.vt_end; ++vt) {
      const int v = vt * SIMT_BN + col;
      float acc[RPT];
#pragma unroll
      for (int r = 0; r < RPT; ++r) acc[r] = 0.f;
      // 32 hidden rows (gathered through idx) and SIMT_BN head rows x KC
      // columns per step, loaded into registers one step ahead: the next
      // step's loads are in flight while this step's FMAs run
      float hv[HE], wv[WE];
      auto load_step = [&](int k0) {
#pragma unroll
        for (int i = 0; i < HE; ++i) {
          const int e = tid + i * THREADS, r = e / KC, kk = e % KC;
          const int src = sm.rix[r];
          hv[i] = (src >= 0 && k0 + kk < a.d) ? load_h(a.hidden, static_cast<int64_t>(src) * a.ldh + k0 + kk, a.hdtype)
                                              : 0.f;
        }
#pragma unroll
        for (int i = 0; i < WE; ++i) {
          const int e = tid + i * THREADS, vr = e / KC, kk = e % KC;
          const int vv = vt * SIMT_BN + vr;
          float x = 0.f;
          if (vv < a.V && k0 + kk < a.d)
            x = a.wdtype == BD_NVFP4 ? load_w_nvfp4(a.w, a.wbs, vv, k0 + kk, a.ldw, a.ldbs)
                                     : load_w(a.w, static_cast<int64_t>(vv) * a.ldw + k0 + kk, a.wdtype);
          wv[i] = x;
        }
      };
      load_step(0);
      for (int k0 = 0; k0 < a.d; k0 += KC) {
#pragma unroll
        for (int i = 0; i < HE; ++i) {
          const int e = tid + i * THREADS;
          sm.hs[e / KC][e % KC] = hv[i];
        }
#pragma unroll
        for (int i = 0; i < WE; ++i) {
          const int e = tid + i * THREADS;
          sm.u.ws[e / KC][e % KC] = wv[i];
        }
        __syncthreads();
        if (k0 + KC < a.d) load_step(k0 + KC);
#pragma unroll 8
        for (int kk = 0; kk < KC; ++kk) {
          const float wk = sm.u.ws[col][kk];
#pragma unroll
          for (int r = 0; r < RPT; ++r) acc[r] = fmaf(sm.hs[rg * RPT + r][kk], wk, acc[r]);
        }
        __syncthreads();
      }
      const bool dead = (v >= a.V) || (v == a.mask_id);
      const float sc = (a.wscale != nullptr && v < a.V) ? a.wscale[v] : 1.f;
#pragma unroll
      for (int r = 0; r < RPT; ++r) {
        const int row = rg * RPT + r;
        const float l = dead ? -INFINITY : acc[r] * sc;
        sm.u.lg[row][col] = l;
        if constexpr (VERIFY) {
          if (v == sm.xd[row]) sm.rx[row] = l;  // one column per row holds the draft entry
        }
      }
      __syncthreads();
      // warp w reduces rows 4w..4w+3; lane l scans columns CPL l .. CPL l + CPL - 1 in order
      for (int rr = 0; rr < SIMT_BM / 8; ++rr) {
        const int r = warp * (SIMT_BM / 8) + rr;
        float m = -INFINITY, s = 0.f, t = 0.f;
        int arg = 0x7fffffff;
#pragma unroll
        for (int j = 0; j < CPL; ++j) {
          const float x = sm.u.lg[r][lane * CPL + j];
          if (x != -INFINITY) {
            // one logit is a state of max x, sum 1 and first moment 0
            if constexpr (VERIFY)
              softmax_combine_t(m, s, arg, t, x, 1.f, vt * SIMT_BN + lane * CPL + j, 0.f);
            else
              softmax_combine(m, s, arg, x, 1.f, vt * SIMT_BN + lane * CPL + j);
          }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
          const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
          const int a2 = __shfl_xor_sync(0xffffffffu, arg, o);
          if constexpr (VERIFY) {
            const float t2 = __shfl_xor_sync(0xffffffffu, t, o);
            softmax_combine_t(m, s, arg, t, m2, s2, a2, t2);
          } else {
            softmax_combine(m, s, arg, m2, s2, a2);
          }
        }
        if (lane == 0) {
          float M = sm.rm[r], S = sm.rs[r];
          int A = sm.ra[r];
          if constexpr (VERIFY) {
            float T = sm.rt[r];
            softmax_combine_t(M, S, A, T, m, s, arg, t);
            sm.rt[r] = T;
          } else {
            softmax_combine(M, S, A, m, s, arg);
          }
          sm.rm[r] = M;
          sm.rs[r] = S;
          sm.ra[r] = A;
        }
      }
      __syncthreads();
    }
    if (tid < SIMT_BM && r0 + tid < n_rows) {
      const int64_t o = static_cast<int64_t>(it.part) * a.P + r0 + tid;
      a.part_m[o] = sm.rm[tid];
      a.part_s[o] = sm.rs[tid];
      a.part_a[o] = sm.ra[tid];
      if constexpr (VERIFY) {
        a.part_t[o] = sm.rt[tid];
        a.part_x[o] = sm.rx[tid];
      }
    }
    __syncthreads();
  }
  griddep_launch_dependents();
}

cudaError_t launch_lmhead_simt(const SimtArgs& a, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.plan.G, 1, 1);
  cfg.blockDim = dim3(THREADS, 1, 1);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return a.part_t != nullptr ? cudaLaunchKernelEx(&cfg, lmhead_simt_kernel<true>, a)
                             : cudaLaunchKernelEx(&cfg, lmhead_simt_kernel<false>, a);
}

}  // namespace bd
