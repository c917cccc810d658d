// The commit sweep and block-buffer update that follow the commit step
// (engine appendix: slot states; maximal-exact-commit appendix, proof parts
// 1 and 2), and its C entry point bd_commit_sweep.
//
// One CTA owns one sequence's window (n_slots <= 64, n_slots * block_len <=
// 4096 positions): it stages the window in shared memory with the step's
// resolutions applied, counts the masked positions per block, takes the
// leading run of active, complete blocks as the committed chain, writes those
// blocks to the cache output and writes the window back shifted by the
// chain's length.
#include <atomic>

#include "bdcommit.h"
#include "common.cuh"
#include "trace.h"

namespace {

constexpr int SWEEP_THREADS = 256;
constexpr int MAX_WINDOW = 4096;  // positions of one sequence's window
constexpr int MAX_SLOTS = 64;     // slots per sequence (per-slot shared arrays, one thread per slot)

struct SweepArgs {
  int32_t* tokens;
  uint8_t* pos_masked;
  uint8_t* block_flags;
  const int32_t* step_tokens;
  const uint32_t* step_commit;
  int32_t* out_cache;
  int32_t* out_n_committed;
  int32_t* out_n_resolved;
  int n_slots, block_len, tau_index, fill;
  uint32_t options;
};

__global__ void __launch_bounds__(SWEEP_THREADS) commit_sweep_kernel(SweepArgs a) {
  __shared__ int32_t tok[MAX_WINDOW];
  __shared__ uint8_t msk[MAX_WINDOW];
  __shared__ int n_masked[MAX_SLOTS];
  __shared__ uint8_t flg[MAX_SLOTS];
  __shared__ uint8_t new_flg[MAX_SLOTS];
  __shared__ int n_res, chain;

  const int tid = threadIdx.x, B = a.n_slots, L = a.block_len, W = B * L;
  const int64_t base = static_cast<int64_t>(blockIdx.x) * W;
  bd::griddep_wait();  // step_tokens / step_commit / the window come from the commit step

  if (tid < B) {
    n_masked[tid] = 0;
    flg[tid] = a.block_flags[static_cast<int64_t>(blockIdx.x) * B + tid];
  }
  if (tid == 0) n_res = 0;
  __syncthreads();

  // 1. resolutions at the deployed threshold, staged with the window
  for (int i = tid; i < W; i += SWEEP_THREADS) {
    const int b = i / L;
    int32_t t = a.tokens[base + i];
    uint8_t m = a.pos_masked[base + i];
    if (m && (flg[b] & BD_BLOCK_ACTIVE) && ((a.step_commit[base + i] >> a.tau_index) & 1u)) {
      t = a.step_tokens[base + i];
      m = 0;
      atomicAdd(&n_res, 1);
    }
    tok[i] = t;
    msk[i] = m;
    if (m) atomicAdd(&n_masked[b], 1);
  }
  __syncthreads();

  // 2. the sweep: the leading run of active, complete blocks commits
  if (tid == 0) {
    int c = 0;
    while (c < B && (flg[c] & BD_BLOCK_ACTIVE) && n_masked[c] == 0) ++c;
    chain = c;
    a.out_n_committed[blockIdx.x] = c;
    if (a.out_n_resolved) a.out_n_resolved[blockIdx.x] = n_res;
  }
  __syncthreads();
  const int c = chain;

  // 3. committed blocks to the cache output
  for (int i = tid; i < c * L; i += SWEEP_THREADS) a.out_cache[base + i] = tok[i];

  // 4. the window shifted left by c blocks, vacated slots refilled
  const int shift = c * L;
  for (int i = tid; i < W; i += SWEEP_THREADS) {
    const int src = i + shift;
    a.tokens[base + i] = src < W ? tok[src] : a.fill;
    a.pos_masked[base + i] = src < W ? msk[src] : uint8_t{1};
  }
  if (tid < B) new_flg[tid] = tid + c < B ? flg[tid + c] : ((a.options & BD_SWEEP_ADMIT) ? BD_BLOCK_ACTIVE : 0);
  __syncthreads();
  if ((a.options & BD_SWEEP_ELIGIBLE_OLDEST) && tid == 0) {
    bool first = true;
    for (int b = 0; b < B; ++b) {
      uint8_t f = new_flg[b] & static_cast<uint8_t>(~BD_BLOCK_FALLBACK_ELIGIBLE);
      if (first && (f & BD_BLOCK_ACTIVE)) {
        f |= BD_BLOCK_FALLBACK_ELIGIBLE;
        first = false;
      }
      new_flg[b] = f;
    }
  }
  __syncthreads();
  if (tid < B) a.block_flags[static_cast<int64_t>(blockIdx.x) * B + tid] = new_flg[tid];
  bd::griddep_launch_dependents();
}

// Compute capability check per device, cached (0 = unknown, 1 = sm_103, 2 = other).
std::atomic<int> g_dev_ok[64];

int check_device() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return BD_ERR_CUDA;
  if (dev < 0 || dev >= 64) return BD_ERR_DEVICE;
  int s = g_dev_ok[dev].load(std::memory_order_relaxed);
  if (s == 0) {
    int maj = 0, mnr = 0;
    if (cudaDeviceGetAttribute(&maj, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&mnr, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
      return BD_ERR_CUDA;
    s = (maj == 10 && mnr == 3) ? 1 : 2;
    g_dev_ok[dev].store(s, std::memory_order_relaxed);
  }
  return s == 1 ? BD_OK : BD_ERR_DEVICE;
}

}  // namespace

extern "C" int bd_commit_sweep(const bd_window* window, const int32_t* step_tokens, const uint32_t* step_commit,
                               int32_t tau_index, uint32_t options, int32_t* out_cache_tokens,
                               int32_t* out_n_committed, int32_t* out_n_resolved, void* stream) {
  bd::TraceRange trace("bd_commit_sweep");
  if (window == nullptr) return BD_ERR_NULL;
  const bd_window& w = *window;
  if (w.n_seq < 0 || w.n_slots < 1 || w.n_slots > MAX_SLOTS || w.block_len < 1 || w.block_len > 64)
    return BD_ERR_SHAPE;
  if (int64_t(w.n_slots) * w.block_len > MAX_WINDOW) return BD_ERR_SHAPE;
  if (int64_t(w.n_seq) * w.n_slots * w.block_len > (int64_t(1) << 24)) return BD_ERR_SHAPE;
  if (tau_index < 0 || tau_index > 31) return BD_ERR_ARG;
  if (options & ~(BD_SWEEP_ADMIT | BD_SWEEP_ELIGIBLE_OLDEST)) return BD_ERR_ARG;
  if (w.n_seq > 0 && (w.tokens == nullptr || w.pos_masked == nullptr || w.block_flags == nullptr ||
                      step_tokens == nullptr || step_commit == nullptr || out_cache_tokens == nullptr ||
                      out_n_committed == nullptr))
    return BD_ERR_NULL;
  if (w.n_seq == 0) return BD_OK;  // nothing to update, no CUDA call
  if (const int rc = check_device()) return rc;

  SweepArgs a;
  a.tokens = w.tokens;
  a.pos_masked = w.pos_masked;
  a.block_flags = w.block_flags;
  a.step_tokens = step_tokens;
  a.step_commit = step_commit;
  a.out_cache = out_cache_tokens;
  a.out_n_committed = out_n_committed;
  a.out_n_resolved = out_n_resolved;
  a.n_slots = w.n_slots;
  a.block_len = w.block_len;
  a.tau_index = tau_index;
  a.fill = w.mask_token_id >= 0 ? w.mask_token_id : -1;
  a.options = options;

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(w.n_seq), 1, 1);
  cfg.blockDim = dim3(SWEEP_THREADS, 1, 1);
  cfg.stream = static_cast<cudaStream_t>(stream);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, commit_sweep_kernel, a);
  if (e == cudaErrorNoKernelImageForDevice || e == cudaErrorInvalidDeviceFunction) return BD_ERR_DEVICE;
  return e == cudaSuccess ? BD_OK : BD_ERR_CUDA;
}
