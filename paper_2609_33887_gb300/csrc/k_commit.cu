// Merge of the per-part softmax partials and the threshold commit with the
// per-block top-1 fallback, for every tau of the grid in one pass.
//
// One CTA (8 warps) per block of the window. Threads split the partial slots
// of each masked position, warp 0 finishes the merge and then applies, for
// every tau_k, the rule
//   commit(p, k) = masked(p) && active(block) && conf(p) >= tau_k           (Sec. 3.1, App. B.1)
//                  || the block is fallback-eligible, holds a masked position,
//                     no position cleared tau_k, and p is the masked position of
//                     highest confidence (lowest position on ties)         (App. B.2)
// with one warp ballot per tau (two for blocks longer than 32).
#include "checks.h"
#include "kernels.h"

namespace bd {

namespace {
constexpr int THREADS = 256;
constexpr int MAX_L = 64;
constexpr int MAX_GROUPS = THREADS / 32;
}  // namespace

__global__ void __launch_bounds__(THREADS) merge_commit_kernel(CommitArgs a) {
  __shared__ float sm_m[MAX_GROUPS][MAX_L], sm_s[MAX_GROUPS][MAX_L];
  __shared__ int sm_a[MAX_GROUPS][MAX_L];
  const int blk = blockIdx.x;
  const int L = a.block_len;
  const int64_t base = static_cast<int64_t>(blk) * L;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  griddep_wait();  // the partials come from the LM-head kernel
  const int n_rows = *a.n_rows;

  // ---- a3: merge of the partial slots. Thread t takes position t % Lp of the
  // block and every groups-th slot starting at t / Lp; loads are issued four
  // slots at a time so their latencies overlap.
  const int Lp = L <= 32 ? 32 : 64;
  const int groups = THREADS / Lp;
  {
    const int jj = threadIdx.x % Lp;
    const int g = threadIdx.x / Lp;
    float m = -INFINITY, s = 0.f;
    int arg = 0x7fffffff;
    // partial slots the workspace holds (index checks of the bounds-checked build)
    const int64_t part_n = static_cast<int64_t>(a.plan.cpu) * (a.plan.G < a.plan.n_vt ? a.plan.G : a.plan.n_vt) * a.P;
    const int r = jj < L && index_ok(base + jj, a.P, a.status) ? a.rowpos[base + jj] : -1;
    if (r >= 0 && index_ok(r, a.P, a.status)) {
      const int ns = slots_of_row(a.plan, n_rows, r);
      int slot = g;
      for (; slot + 3 * groups < ns; slot += 4 * groups) {
        float pm[4], ps[4];
        int pa[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int64_t o = static_cast<int64_t>(slot + u * groups) * a.P + r;
          const bool in = index_ok(o, part_n, a.status);
          pm[u] = in ? a.part_m[o] : -INFINITY;
          ps[u] = in ? a.part_s[o] : 0.f;
          pa[u] = in ? a.part_a[o] : 0x7fffffff;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) softmax_combine(m, s, arg, pm[u], ps[u], pa[u]);
      }
      for (; slot < ns; slot += groups) {
        const int64_t o = static_cast<int64_t>(slot) * a.P + r;
        if (index_ok(o, part_n, a.status)) softmax_combine(m, s, arg, a.part_m[o], a.part_s[o], a.part_a[o]);
      }
    }
    if (jj < L) {
      sm_m[g][jj] = m;
      sm_s[g][jj] = s;
      sm_a[g][jj] = arg;
    }
  }
  __syncthreads();
  if (warp != 0) return;

  const uint32_t flags = a.block_flags[blk];
  const bool eligible = (flags & 2u) != 0;
  bool live[2];
  float conf[2];
  int tok[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int jj = lane + 32 * h;
    live[h] = jj < L && a.rowpos[base + jj] >= 0;
    conf[h] = 0.f;
    tok[h] = -1;
    if (live[h]) {
      float m = sm_m[0][jj], s = sm_s[0][jj];
      int arg = sm_a[0][jj];
      for (int g = 1; g < groups; ++g) softmax_combine(m, s, arg, sm_m[g][jj], sm_s[g][jj], sm_a[g][jj]);
      conf[h] = 1.f / s;  // s >= 1: the maximum contributes exp(0)
      tok[h] = arg;
    }
  }

  // fallback candidate: highest confidence among masked positions, lowest position on ties
  float best_c = -1.f;
  int best_j = 0x7fffffff;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int jj = lane + 32 * h;
    if (live[h] && (conf[h] > best_c || (conf[h] == best_c && jj < best_j))) {
      best_c = conf[h];
      best_j = jj;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float c2 = __shfl_xor_sync(0xffffffffu, best_c, o);
    const int j2 = __shfl_xor_sync(0xffffffffu, best_j, o);
    if (c2 > best_c || (c2 == best_c && j2 < best_j)) {
      best_c = c2;
      best_j = j2;
    }
  }
  const bool any_live = __any_sync(0xffffffffu, live[0] || live[1]);
  const bool take_fallback = eligible && any_live;

  const int seq = blk / a.n_slots;
  uint32_t bits[2] = {0u, 0u};
  for (int k = 0; k < a.taus.T; ++k) {
    const float tau = a.taus.tau[k];
    bool c0 = live[0] && conf[0] >= tau;
    bool c1 = live[1] && conf[1] >= tau;
    uint32_t b0 = __ballot_sync(0xffffffffu, c0);
    uint32_t b1 = __ballot_sync(0xffffffffu, c1);
    if ((b0 | b1) == 0u && take_fallback) {
      if (best_j < 32) {
        b0 = 1u << best_j;
        c0 = (lane == best_j);
      } else {
        b1 = 1u << (best_j - 32);
        c1 = (lane == best_j - 32);
      }
    }
    bits[0] |= static_cast<uint32_t>(c0) << k;
    bits[1] |= static_cast<uint32_t>(c1) << k;
    if (a.out_counts != nullptr && lane == 0) {
      const int cnt = __popc(b0) + __popc(b1);
      if (cnt) atomicAdd(a.out_counts + static_cast<int64_t>(seq) * a.taus.T + k, cnt);
    }
  }

#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int jj = lane + 32 * h;
    if (jj < L) {
      a.out_tokens[base + jj] = tok[h];
      a.out_conf[base + jj] = conf[h];
      a.out_commit[base + jj] = bits[h];
    }
  }
}

cudaError_t launch_merge_commit(const CommitArgs& a, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.n_blocks, 1, 1);
  cfg.blockDim = dim3(THREADS, 1, 1);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, merge_commit_kernel, a);
}

}  // namespace bd
