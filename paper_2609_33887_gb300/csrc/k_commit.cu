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
//
// Vocabulary-parallel split (one head shard per rank): MERGE_EMIT merges the
// slots of each position of this shard's LM head into one partial per window
// position (global token ids: the shard's offset added) instead of
// committing; MERGE_GATHERED merges the n_parts such per-position partials
// gathered from every shard ([n_parts, P] arrays) and commits.
#include "checks.h"
#include "kernels.h"

namespace bd {

namespace {
constexpr int THREADS = 256;
constexpr int MAX_L = 64;
constexpr int MAX_GROUPS = THREADS / 32;
}  // namespace

template <int MODE>
__global__ void __launch_bounds__(THREADS) merge_commit_kernel(CommitArgs a) {
  __shared__ float sm_m[MAX_GROUPS][MAX_L], sm_s[MAX_GROUPS][MAX_L];
  __shared__ int sm_a[MAX_GROUPS][MAX_L];
  __shared__ bool sm_live[MAX_L];  // the position has a compacted row (read once, in the merge stage)
  const int blk = blockIdx.x;
  const int L = a.block_len;
  const int64_t base = static_cast<int64_t>(blk) * L;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  griddep_wait();  // the partials come from the LM-head kernel
  // partial slots per row over the plan's launches (header word)
  const int slots = MODE == MERGE_GATHERED ? a.n_parts : a.n_rows[HDR_SLOTS];

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
    const int64_t part_n = MODE == MERGE_GATHERED
                               ? static_cast<int64_t>(a.n_parts) * a.P
                               : static_cast<int64_t>(plan_max_slots(a.plan)) * a.P;
    int r = -1;  // the slot index of this position: its compacted row, or (gathered) the position itself
    if (jj < L && index_ok(base + jj, a.P, a.status)) {
      if constexpr (MODE == MERGE_GATHERED)
        r = (a.pos_masked[base + jj] != 0 && (a.block_flags[blk] & 1u)) ? static_cast<int>(base + jj) : -1;
      else
        r = a.rowpos[base + jj];
    }
    if (r >= 0 && index_ok(r, a.P, a.status)) {
      const int ns = slots;
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
      if (g == 0) sm_live[jj] = r >= 0;
    }
  }
  __syncthreads();
  if (warp != 0) return;

  if constexpr (MODE == MERGE_EMIT) {
    // one partial per window position, token ids of the whole vocabulary
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int jj = lane + 32 * h;
      if (jj < L) {
        float m = -INFINITY, s = 0.f;
        int arg = -1;
        if (sm_live[jj]) {
          m = sm_m[0][jj];
          s = sm_s[0][jj];
          arg = sm_a[0][jj];
          for (int g = 1; g < groups; ++g) softmax_combine(m, s, arg, sm_m[g][jj], sm_s[g][jj], sm_a[g][jj]);
          arg = m == -INFINITY ? -1 : arg + a.vocab_offset;  // a shard holding only the mask token: nothing
        }
        a.emit_m[base + jj] = m;
        a.emit_s[base + jj] = s;
        a.emit_a[base + jj] = arg;
      }
    }
    return;
  }

  const uint32_t flags = a.block_flags[blk];
  const bool eligible = (flags & 2u) != 0;
  bool live[2];
  float conf[2];
  int tok[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int jj = lane + 32 * h;
    live[h] = jj < L && sm_live[jj];
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

cudaError_t launch_merge_commit(const CommitArgs& a, cudaStream_t st, int mode) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.n_blocks, 1, 1);
  cfg.blockDim = dim3(THREADS, 1, 1);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  switch (mode) {
    case MERGE_EMIT:
      return cudaLaunchKernelEx(&cfg, merge_commit_kernel<MERGE_EMIT>, a);
    case MERGE_GATHERED:
      return cudaLaunchKernelEx(&cfg, merge_commit_kernel<MERGE_GATHERED>, a);
    default:
      return cudaLaunchKernelEx(&cfg, merge_commit_kernel<MERGE_ROWS>, a);
  }
}

}  // namespace bd
