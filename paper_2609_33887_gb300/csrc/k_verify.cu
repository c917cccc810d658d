// Merge of the verification partials and the acceptance rules of speculative
// decoding (typical-acceptance and lossless-reference appendices), for a whole
// grid of eps settings in one pass.
//
// One CTA (4 warps) per request. A warp merges the partial slots of one row
// (lanes split the slots, then a shuffle tree) into the row's softmax state
// (max M, sum S, argmax A, first moment T in log2 units) and draft logit; lane
// 0 then derives
//   p(x) = exp(l_x - M) / S,   H = ln S - T / (S log2 e)
// and sets bit k when p(x) > min(eps_k, sqrt(eps_k) exp(-H)) and bit 31 when
// the draft equals the argmax. The CTA finally counts, per setting, the
// accepted prefix of the request's draft rows.
#include "kernels.h"

namespace bd {

namespace {
constexpr int THREADS = 128;
constexpr int MAX_ROWS = 33;  // n_draft <= 32 drafts + the bonus row
}  // namespace

__global__ void __launch_bounds__(THREADS) merge_verify_kernel(VerifyArgs a) {
  __shared__ uint32_t bits_s[MAX_ROWS];
  const int q = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int D = a.n_draft, Rq = D + 1;
  griddep_wait();  // the partials come from the LM-head kernel
  // partial slots per row over the plan's launches (header word)
  const int ns = a.n_rows[HDR_SLOTS];

  for (int i = warp; i < Rq; i += THREADS / 32) {
    const int r = q * Rq + i;
    float m = -INFINITY, s = 0.f, t = 0.f, lx = -INFINITY;
    int arg = 0x7fffffff;
    for (int slot = lane; slot < ns; slot += 32) {
      const int64_t o = static_cast<int64_t>(slot) * a.P + r;
      softmax_combine_t(m, s, arg, t, a.part_m[o], a.part_s[o], a.part_a[o], a.part_t[o]);
      lx = fmaxf(lx, a.part_x[o]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
      const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
      const int a2 = __shfl_xor_sync(0xffffffffu, arg, o);
      const float t2 = __shfl_xor_sync(0xffffffffu, t, o);
      softmax_combine_t(m, s, arg, t, m2, s2, a2, t2);
      lx = fmaxf(lx, __shfl_xor_sync(0xffffffffu, lx, o));
    }
    if (lane == 0) {
      const int x = a.draft_row[r];
      const float H = logf(s) - t / (s * LOG2E);
      const float px = (x >= 0 && lx != -INFINITY) ? ex2_approx((lx - m) * LOG2E) / s : 0.f;
      uint32_t bits = 0;
      if (x >= 0) {
        const float eh = expf(-H);
        for (int k = 0; k < a.E; ++k)
          if (px > fminf(a.eps[k], a.sqrt_eps[k] * eh)) bits |= 1u << k;
        if (x == arg) bits |= 1u << 31;
      }
      a.out_tokens[r] = arg;
      a.out_p_draft[r] = px;
      a.out_entropy[r] = H;
      a.out_accept[r] = bits;
      bits_s[i] = bits;
    }
  }
  __syncthreads();
  if (threadIdx.x <= a.E) {
    const int k = threadIdx.x;
    const int bit = k == a.E ? 31 : k;
    int n = 0;
    while (n < D && ((bits_s[n] >> bit) & 1u)) ++n;
    a.out_accepted[static_cast<int64_t>(q) * (a.E + 1) + k] = n;
  }
}

cudaError_t launch_merge_verify(const VerifyArgs& a, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(a.n_req), 1, 1);
  cfg.blockDim = dim3(THREADS, 1, 1);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, merge_verify_kernel, a);
}

}  // namespace bd
