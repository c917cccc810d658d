// LM-head projection + mask-suppressed softmax statistics on the tcgen05
// tensor cores (the engine's LM head and the softmax it commits from,
// App. B.1). Logits live only in tensor memory: the epilogue reduces every
// row of every 128 x 256 tile to a running (max, sum of exponentials,
// argmax) and writes one partial per (row, vocabulary part).
//
// CTA layout (192 threads, one CTA per SM, persistent over the band plan):
//   warp 0      TMA producer: A (packed hidden rows) and B (head rows) tiles
//               of 64 columns (128 B, 128-byte swizzle) into a STAGES ring
//   warp 1      allocates 512 TMEM columns; an elected lane issues tcgen05.mma
//               (M=128, N=256, K=16) into one of two 256-column fp32
//               accumulators, so the epilogue of tile i overlaps tile i+1
//   warps 2..5  epilogue: warp w reads TMEM lanes 32*(w%4)..+31 (one row per
//               thread), 32 columns at a time
// The producer and issuer loops run in the whole warp (warp-uniform waits) and
// one elected lane issues the copies and MMAs.
// Every wait is bounded; on timeout the CTA raises DEV_TIMEOUT in the status
// word, drains its copies and MMAs, frees TMEM and returns.
// The verification instantiation (VERIFY = true) also carries the entropy
// accumulator sum exp(l - m) (l - m) log2(e) and the logit of the row's draft
// entry (typical-acceptance appendix).
#include <atomic>

#include "kernels.h"

namespace bd {

namespace {

constexpr int BM = TC_BM, BN = TC_BN, BK = TC_BK;
constexpr uint32_t A_BYTES = BM * BK * 2;  // 16 KB
constexpr uint32_t B_BYTES = BN * BK * 2;  // 32 KB
constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t IDESC = idesc_bf16_f32(BM, BN);

struct Ctl {
  uint64_t full[8];
  uint64_t empty[8];
  uint64_t tfull[2];
  uint64_t tempty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort_flag;
};


}  // namespace

template <int STAGES, bool VERIFY>
__global__ void __launch_bounds__(TC_THREADS, 1)
    lmhead_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, TcArgs a) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Ctl* ctl = reinterpret_cast<Ctl*>(smem + STAGES * STAGE_BYTES);
  const uint32_t smem_base = smem_u32(smem);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(smem_u32(&ctl->full[s]), 1);
      mbar_init(smem_u32(&ctl->empty[s]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&ctl->tfull[i]), 1);
      mbar_init(smem_u32(&ctl->tempty[i]), 4);
    }
    mbar_init(smem_u32(&ctl->drain), 1);
    ctl->abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&ctl->tmem_base), TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = ctl->tmem_base;
  volatile int* abort_flag = &ctl->abort_flag;

  griddep_wait();  // the packed rows and N come from the preceding kernel
  const int n_rows = a.n_rows[HDR_N];
  const int nk = cdiv(a.d, BK);

  if (warp == 0) {
    // ------------------------------------------------------ TMA producer
    // the whole warp walks the stages (warp-uniform waits); one lane issues
    const bool leader = elect_one();
    const uint64_t pol_a = l2_policy(a.l2_rows);  // hidden rows: re-read by every part
    const uint64_t pol_b = l2_policy(a.l2_head);  // head rows: fetched once per band, re-read from L2 by its m-tiles
    uint32_t stage = 0, phase = 0;
    uint32_t issued_mask = 0, issued_phase = 0;  // per stage: issued at least once / parity of last issue
    TileIter it;
    it.init(a.plan, a.n_rows);
    bool ok = true;
    while (ok && it.next_unit()) {
      for (int vt = it.vt; ok && vt < it.vt_end; ++vt) {
        for (int kb = 0; kb < nk; ++kb) {
          if (!mbar_wait_warp(smem_u32(&ctl->empty[stage]), phase ^ 1u, abort_flag, a.status)) {
            ok = false;
            break;
          }
          if (leader) {
            const uint32_t fb = smem_u32(&ctl->full[stage]);
            mbar_expect_tx(fb, STAGE_BYTES);
            const uint32_t sa = smem_base + stage * STAGE_BYTES;
            tma_load_2d(sa, &tmA, fb, kb * BK, it.m_tile * BM, pol_a);
            tma_load_2d(sa + A_BYTES, &tmB, fb, kb * BK, vt * BN, pol_b);
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
    // Wait for the last load issued into every stage (immediate unless aborted).
    if (leader)
      for (int s = 0; s < STAGES; ++s)
        if (issued_mask & (1u << s)) mbar_drain(smem_u32(&ctl->full[s]), (issued_phase >> s) & 1u);
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------ MMA issuer
    const bool leader = elect_one();
    uint32_t stage = 0, phase = 0;
    uint32_t acc = 0, acc_phase = 0;
    TileIter it;
    it.init(a.plan, a.n_rows);
    bool ok = true;
    while (ok && it.next_unit()) {
      for (int vt = it.vt; ok && vt < it.vt_end; ++vt) {
        if (!mbar_wait_warp(smem_u32(&ctl->tempty[acc]), acc_phase ^ 1u, abort_flag, a.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        for (int kb = 0; kb < nk; ++kb) {
          if (!mbar_wait_warp(smem_u32(&ctl->full[stage]), phase, abort_flag, a.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          if (leader) {
            const uint32_t sa = smem_base + stage * STAGE_BYTES;
            const uint64_t adesc = sw128_kmajor_desc(sa);
            const uint64_t bdesc = sw128_kmajor_desc(sa + A_BYTES);
#pragma unroll
            for (int k = 0; k < BK / 16; ++k) {
              // +32 bytes along K inside the 128-byte swizzled row = +2 in the address field
              umma_bf16(d_tmem, adesc + 2u * k, bdesc + 2u * k, IDESC, (kb | k) != 0);
            }
            umma_commit(smem_u32(&ctl->empty[stage]));
          }
          __syncwarp();
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        if (leader) umma_commit(smem_u32(&ctl->tfull[acc]));
        __syncwarp();
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1u;
        }
      }
    }
    // All MMAs issued by the elected thread have completed once `drain` flips.
    if (leader) {
      umma_commit(smem_u32(&ctl->drain));
      mbar_drain(smem_u32(&ctl->drain), 0);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------ epilogue
    const int quarter = warp & 3;
    const int row_in_tile = quarter * 32 + lane;
    const uint32_t lane_addr = static_cast<uint32_t>(quarter * 32) << 16;
    uint32_t acc = 0, acc_phase = 0;
    TileIter it;
    it.init(a.plan, a.n_rows);
    bool ok = true;
    while (ok && it.next_unit()) {
      float m = -INFINITY, s = 0.f;
      int arg = 0x7fffffff;
      float t = 0.f, lx = -INFINITY;  // VERIFY only
      int xd = -1;
      if constexpr (VERIFY) {
        const int row = it.m_tile * BM + row_in_tile;
        if (row < n_rows) xd = a.draft_row[row];
      }
      for (int vt = it.vt; vt < it.vt_end; ++vt) {
        if (!mbar_wait_warp(smem_u32(&ctl->tfull[acc]), acc_phase, abort_flag, a.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const int col_tile = vt * BN;
        // a tile needs per-column masking only at the vocabulary end or where it holds the mask token
        const bool tile_edge = (col_tile + BN > a.V) || (static_cast<unsigned>(a.mask_id - col_tile) < static_cast<unsigned>(BN));
#pragma unroll 1
        for (int c = 0; c < BN / 32; ++c) {
          float v[32];
          tmem_ld32(tmem_base + lane_addr + acc * BN + c * 32, v);
          const int col0 = col_tile + c * 32;
          if (a.wscale != nullptr) {
#pragma unroll
            for (int j = 0; j < 32; ++j) {
              const int col = col0 + j < a.V ? col0 + j : a.V - 1;
              v[j] *= __ldg(a.wscale + col);
            }
          }
          if (tile_edge) {
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (col0 + j >= a.V || col0 + j == a.mask_id) v[j] = -INFINITY;
          }
          if constexpr (VERIFY) {
            if (static_cast<unsigned>(xd - col0) < 32u) {
#pragma unroll
              for (int j = 0; j < 32; ++j)
                if (col0 + j == xd) lx = v[j];
            }
          }
          float cm = v[0];
#pragma unroll
          for (int j = 1; j < 32; ++j) cm = fmaxf(cm, v[j]);
          if (cm > m) {
            int jj = 31;
#pragma unroll
            for (int j = 31; j >= 0; --j)
              if (v[j] == cm) jj = j;
            arg = col0 + jj;
            if constexpr (VERIFY) {
              if (m == -INFINITY) {
                s = 0.f;
                t = 0.f;
              } else {
                const float dm = (m - cm) * LOG2E;
                const float f = ex2_approx(dm);
                t = f * fmaf(dm, s, t);
                s *= f;
              }
            } else {
              s = (m == -INFINITY) ? 0.f : s * ex2_approx((m - cm) * LOG2E);
            }
            m = cm;
          }
          if (m != -INFINITY) {
            const float mc = m * LOG2E;
            const bool wide = !(fabsf(mc) < FUSED_SHIFT_LIMIT);  // take v - m first (see common.cuh)
            if constexpr (VERIFY) {
              float s0 = 0.f, s1 = 0.f, t0 = 0.f, t1 = 0.f;
#pragma unroll
              for (int j = 0; j < 32; j += 2) {
                const float u0 = wide ? (v[j] - m) * LOG2E : fmaf(v[j], LOG2E, -mc);
                const float u1 = wide ? (v[j + 1] - m) * LOG2E : fmaf(v[j + 1], LOG2E, -mc);
                const float e0 = ex2_approx(u0), e1 = ex2_approx(u1);
                s0 += e0;
                s1 += e1;
                t0 = fmaf(e0, fmaxf(u0, -256.f), t0);
                t1 = fmaf(e1, fmaxf(u1, -256.f), t1);
              }
              s += s0 + s1;
              t += t0 + t1;
            } else {
              float s0 = 0.f, s1 = 0.f;
              if (!wide) {
#pragma unroll
                for (int j = 0; j < 32; j += 2) {
                  s0 += ex2_approx(fmaf(v[j], LOG2E, -mc));
                  s1 += ex2_approx(fmaf(v[j + 1], LOG2E, -mc));
                }
              } else {
#pragma unroll
                for (int j = 0; j < 32; j += 2) {
                  s0 += ex2_approx((v[j] - m) * LOG2E);
                  s1 += ex2_approx((v[j + 1] - m) * LOG2E);
                }
              }
              s += s0 + s1;
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&ctl->tempty[acc]));
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1u;
        }
      }
      if (!ok) break;
      const int row = it.m_tile * BM + row_in_tile;
      if (row < n_rows) {
        const int64_t o = static_cast<int64_t>(it.part) * a.P + row;
        a.part_m[o] = m;
        a.part_s[o] = s;
        a.part_a[o] = arg;
        if constexpr (VERIFY) {
          a.part_t[o] = t;
          a.part_x[o] = lx;
        }
      }
    }
  }

  __syncwarp();
  griddep_launch_dependents();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, TMEM_COLS);
}

size_t tc_smem_bytes(int stages) { return static_cast<size_t>(stages) * STAGE_BYTES + sizeof(Ctl) + 1024; }

template <int STAGES, bool VERIFY>
static cudaError_t launch_stages(const CUtensorMap& tmA, const CUtensorMap& tmB, const TcArgs& a,
                                 cudaStream_t st) {
  const size_t smem = tc_smem_bytes(STAGES);
  static_assert(STAGES <= 8, "Ctl holds 8 stages");
  // the shared-memory opt-in is set once per device (not again inside a graph capture)
  static std::atomic<uint64_t> opted_in{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if ((opted_in.load() & bit) == 0) {
    e = cudaFuncSetAttribute(lmhead_tc_kernel<STAGES, VERIFY>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    opted_in.fetch_or(bit);
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.plan.G, 1, 1);
  cfg.blockDim = dim3(TC_THREADS, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, lmhead_tc_kernel<STAGES, VERIFY>, tmA, tmB, a);
}

cudaError_t launch_lmhead_tc(const CUtensorMap& tmA, const CUtensorMap& tmB, const TcArgs& a, int stages,
                             cudaStream_t st) {
  const bool verify = a.part_t != nullptr;
  switch (stages) {
    case 3:
      return verify ? launch_stages<3, true>(tmA, tmB, a, st) : launch_stages<3, false>(tmA, tmB, a, st);
    default:
      return verify ? launch_stages<4, true>(tmA, tmB, a, st) : launch_stages<4, false>(tmA, tmB, a, st);
  }
}

}  // namespace bd
