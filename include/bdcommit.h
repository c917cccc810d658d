/*
 * bdcommit: the per-forward commit step of a multi-block diffusion LM engine
 * on one GB300 (sm_103a).
 *
 * One call takes the final hidden state of every position in the engine's
 * window of block slots, and for every still-masked position of every active
 * block:
 *   1. projects it through the LM head          logits = W_head . h
 *   2. reads the mask-suppressed softmax         conf = max_v softmax(logits)_v,
 *      that the engine commits from                token = argmax_v (lowest v on ties)
 *      (App. B.1, "Entropy of the deeper blocks")
 *   3. applies the accept threshold              commit when conf >= tau
 *      ("at or above the accept threshold", Sec. 3.1 and App. B.1), with the
 *      per-block top-1 fallback when no position clears it (App. B.2,
 *      self-distillation protocol), once for every tau of a grid, so one
 *      forward scores a whole grid of operating points (App. F.3).
 * Logits never reach device memory: the LM-head kernel reduces each row to a
 * running (max, sum of exponentials, argmax) while it multiplies.
 *
 * Conventions for every entry point below
 *   - All tensors are caller-owned. Device pointers must stay valid until the
 *     work queued on the stream has finished; the library keeps no reference.
 *   - Calls are asynchronous on the given stream and never synchronise the
 *     host, except bd_get_device_status (documented there).
 *   - Return value: 0 (BD_OK) or a negative bd_status. Argument checks happen
 *     before any CUDA call, so a rejected call has queued nothing. The library
 *     never traps, aborts or exits.
 *   - Position p of the window is p = (s * n_slots + b) * block_len + j for
 *     sequence s, slot b and offset j in the block.
 */
#ifndef BDCOMMIT_H
#define BDCOMMIT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---------------------------------------------------------------- status */
typedef enum {
  BD_OK = 0,
  BD_ERR_NULL = -1,      /* a required pointer is NULL */
  BD_ERR_SHAPE = -2,     /* sizes disagree or are out of range */
  BD_ERR_DTYPE = -3,     /* unsupported dtype or dtype combination */
  BD_ERR_ALIGN = -4,     /* pointer or row stride misaligned (see bd_weight) */
  BD_ERR_TAU = -5,       /* T outside 1..32, NULL grid, or a NaN threshold */
  BD_ERR_WORKSPACE = -6, /* caller workspace smaller than bd_workspace_size */
  BD_ERR_CUDA = -7,      /* a CUDA runtime call or kernel launch failed */
  BD_ERR_TIMEOUT = -8,   /* a bounded device-side wait gave up (see bd_get_device_status) */
  BD_ERR_DEVICE = -9,    /* the current device cannot run this library (needs sm_103) */
  BD_ERR_ARG = -10,      /* other invalid argument (mask_token_id, variant, flags) */
  BD_ERR_BOUNDS = -11    /* a device-side index check failed: only the bounds-checked build
                            (libbdcommit_checks.so, -DBD_CHECKS) checks indices */
} bd_status;

/* ----------------------------------------------------------------- dtypes */
typedef enum {
  BD_F32 = 0,  /* IEEE binary32 */
  BD_BF16 = 1, /* bfloat16 */
  BD_E4M3 = 2, /* FP8 E4M3 (OCP "fn" variant: no infinities), weights only */
  BD_NVFP4 = 3 /* 4-bit E2M1 codes with an E4M3 scale per 16 elements (NVFP4), weights only */
} bd_dtype;

/* bd_exec.flags bits. */
#define BD_EXEC_FP8_ACTIVATIONS 1

/* Block flag bits (bd_mask_state.block_flags). */
#define BD_BLOCK_ACTIVE 1u            /* the slot holds an active block (App. F) */
#define BD_BLOCK_FALLBACK_ELIGIBLE 2u /* the block may take the top-1 fallback (App. B.2) */

/* Hidden states of the whole window: [rows, cols] row-major, device memory.
 *   rows  = P = n_seq * n_slots * block_len (every slot, placeholders too:
 *           the engine forwards the whole window, App. F)
 *   cols  = d, the model width
 *   ld    = elements between consecutive rows (>= cols)
 *   dtype = BD_F32 or BD_BF16. With BD_BF16 the pointer must be 16-byte
 *           aligned and ld * 2 a multiple of 16. */
typedef struct {
  const void* data;
  int32_t dtype;
  int64_t rows;
  int64_t cols;
  int64_t ld;
} bd_hidden;

/* LM-head weights [vocab, dim] row-major (one row per vocabulary entry, the
 * K-major layout of an nn.Linear head), device memory.
 *   dtype BD_F32  : with BD_F32 hidden states (exact fp32 SIMT path).
 *   dtype BD_BF16 : with BD_BF16 hidden states (tensor-core path).
 *   dtype BD_E4M3 : with BD_BF16 hidden states; `scale` is a device float32
 *                   array [vocab] and the weight of row v is code * scale[v]
 *                   (per-output-channel scaling, the FP8 precision lever).
 *   dtype BD_NVFP4: with BD_BF16 hidden states (the 4-bit weight lever).
 *                   `data` holds E2M1 codes, two per byte: element k of a row
 *                   is the low nibble of byte k / 2 for even k, the high
 *                   nibble for odd k; `ld` counts BYTES (>= ceil(dim / 2));
 *                   `block_scale` [vocab, block_ld] holds E4M3 codes, element
 *                   k using block_scale[v * block_ld + k / 16] (block_ld >=
 *                   ceil(dim / 16)); `scale` is an optional float32 [vocab]
 *                   per-row scale (NULL = 1). Weight (v, k) =
 *                   e2m1(code) * e4m3(block scale) * scale[v].
 *   For BD_BF16 / BD_E4M3 / BD_NVFP4 the pointer must be 16-byte aligned and
 *   ld * element size (bytes for BD_NVFP4) a multiple of 16.
 *   Both quantised formats decode exactly to bf16. A BD_E4M3 head on the
 *   commit step is read as it is by the 8-bit tensor path of the CTA-pair
 *   kernel at every window size (see bd_exec.variant), with no copy. For the
 *   other cases, on the CTA-pair kernel (windows up to 8192 positions) the
 *   codes are decoded inside the kernel, so the workspace holds no bf16 copy
 *   of the head, when a row holds at least 16 bytes of codes and, for
 *   BD_NVFP4, `block_scale` is 16-byte aligned with block_ld a multiple of
 *   16; otherwise the head is first decoded into a bf16 copy in the
 *   workspace (bd_workspace_size accounts for it). The environment variables
 *   BD_E4M3_SPLIT=0 (no 8-bit path) and BD_FUSED_DECODE=0 (no decode in the
 *   kernel) select the other paths. */
typedef struct {
  const void* data;
  int32_t dtype;
  int64_t vocab;
  int64_t dim;
  int64_t ld;
  const float* scale;         /* required for BD_E4M3, optional for BD_NVFP4, else ignored */
  const uint8_t* block_scale; /* BD_NVFP4 only */
  int64_t block_ld;           /* BD_NVFP4 only */
} bd_weight;

/* Which positions are still masked and which slots hold active blocks
 * (the engine's fixed-slot block buffer, App. F). Device memory.
 *   pos_masked [n_seq * n_slots * block_len] : 1 = still masked, 0 = resolved
 *   block_flags[n_seq * n_slots]             : BD_BLOCK_* bits
 *   block_len in 1..64 (the paper's engine uses 32)
 *   mask_token_id: -1 = no suppression; else in [0, vocab): that entry is
 *                  removed from the softmax and can never be the token. */
typedef struct {
  int32_t n_seq;
  int32_t n_slots;
  int32_t block_len;
  int32_t mask_token_id;
  const uint8_t* pos_masked;
  const uint8_t* block_flags;
} bd_mask_state;

/* Threshold grid: HOST array tau[0..T-1], 1 <= T <= 32, no NaN. Bit k of a
 * position's commit mask answers "does this position commit at tau[k]". The
 * values are copied at call time; the array may be reused immediately. */
typedef struct {
  const float* tau;
  int32_t T;
} bd_tau_grid;

/* Execution options.
 *   stream          : a cudaStream_t (NULL = the legacy default stream).
 *   workspace       : device scratch of at least bd_workspace_size bytes,
 *                     256-byte aligned; NULL = a library-owned buffer for the
 *                     current device, grown with cudaMalloc on demand (not
 *                     allowed inside CUDA graph capture: pass your own then).
 *                     One workspace must not be used by two calls that can
 *                     run at the same time.
 *   out_counts      : optional device int32 [n_seq * T]; receives, per
 *                     sequence and threshold, the number of committed
 *                     positions (the numerator of tokens per forward, Sec. 2.1).
 *   lmhead_event_begin / lmhead_event_end : optional cudaEvent_t recorded on
 *                     the stream right before and after the LM-head kernel,
 *                     for timing it alone.
 *   variant         : 0 = automatic: the CTA-pair tensor-core kernel for BF16
 *                     heads at every window size and for E4M3 heads with
 *                     16-byte aligned rows (see below); NVFP4 heads (and E4M3
 *                     heads the 8-bit path cannot read) on the CTA-pair kernel
 *                     up to 8192 window positions and the one-CTA kernel on a
 *                     decoded bf16 copy above; the fp32 SIMT kernel for F32
 *                     heads. 1 = force the fp32-FMA SIMT LM-head kernel; 2 =
 *                     force the one-CTA tensor-core kernel (tokens on the MMA M
 *                     side); 3 = force the CTA-pair tensor-core kernel
 *                     (vocabulary on the M side). 2 and 3 need BF16 hidden
 *                     states.
 *                     E4M3 heads on the CTA-pair kernel (variant 0 or 3, code
 *                     rows 16-byte aligned, dim >= 16) run on the 8-bit tensor
 *                     path with the BF16 hidden states unchanged in value: each
 *                     packed row is scaled by a power of two 2^s so that its
 *                     largest magnitude lies in [128, 256) and written as two
 *                     E4M3 terms hi = e4m3(h 2^s), lo = e4m3(h 2^s - hi); the
 *                     head's codes multiply both terms (tcgen05.mma
 *                     kind::f8f6f4, exact products, fp32 accumulation) and the
 *                     logits are scaled by 2^-s and the head's row scale.
 *                     hi + lo equals h 2^s exactly for every element of at
 *                     least 2^-10 of its row's largest; a smaller one is off
 *                     by at most 2^-17 of the row's largest.
 *   flags           : 0, or BD_EXEC_FP8_ACTIVATIONS (commit step only): the
 *                     W8A8 variant of the precision lever. Needs a BD_E4M3 head
 *                     (16-byte aligned, ld a multiple of 16, dim >= 16), BF16
 *                     hidden states and the CTA-pair kernel (variant 0 or 3);
 *                     else BD_ERR_ARG / ALIGN.
 *                     Each packed hidden row is quantised to E4M3 with one
 *                     scale per row (a = max |h|, code = e4m3(h * fl32(448 /
 *                     a)) rounding to nearest even and saturating, scale =
 *                     fl32(a / 448); an all-zero row gets scale 0) and the LM
 *                     head multiplies the E4M3 codes on the 8-bit tensor path
 *                     (tcgen05.mma kind::f8f6f4), applying the head's row scale
 *                     and the token's scale to each fp32 logit. Lossy: results
 *                     are those of the quantised activations. */
typedef struct {
  void* stream;
  void* workspace;
  size_t workspace_bytes;
  int32_t* out_counts;
  void* lmhead_event_begin;
  void* lmhead_event_end;
  int32_t variant;
  int32_t flags;
} bd_exec;

/* The commit step (Sec. 3.1, App. B.1, B.2, F) on the default stream with the
 * library-owned workspace. Outputs, all device arrays of P entries and all
 * fully written:
 *   out_tokens[p] : argmax token of a masked position of an active block, else -1
 *   out_conf[p]   : its confidence (max softmax probability, in (0, 1]), else 0
 *   out_commit[p] : bit k set <=> the position commits at tau[k], else 0 */
int bd_commit_step(const bd_hidden* hidden, const bd_weight* weight,
                   const bd_mask_state* mask_state, const bd_tau_grid* tau_grid,
                   int32_t* out_tokens, float* out_conf, uint32_t* out_commit);

/* Same as bd_commit_step with explicit execution options (exec may be NULL). */
int bd_commit_step_ex(const bd_hidden* hidden, const bd_weight* weight,
                      const bd_mask_state* mask_state, const bd_tau_grid* tau_grid,
                      int32_t* out_tokens, float* out_conf, uint32_t* out_commit,
                      const bd_exec* exec);

/* Bytes of device workspace a call with these arguments needs (0 if the
 * arguments are invalid), for bd_exec.variant 0 (automatic) with flags 0 or
 * BD_EXEC_FP8_ACTIVATIONS. Depends on sizes, dtypes and the current device's
 * SM count only, not on the data. A forced variant 1 or 2 can need more (more
 * partial slots; a decoded copy of a quantised head); such a call with a
 * smaller caller workspace returns BD_ERR_WORKSPACE without launching. */
size_t bd_workspace_size(const bd_hidden* hidden, const bd_weight* weight,
                         const bd_mask_state* mask_state, const bd_tau_grid* tau_grid);

/* Kernels one bd_commit_step_ex call with these arguments queues (the
 * per-threshold counts' reset is a memset, not a kernel): compaction + row
 * packing, the decode of a quantised head where the LM head reads a bf16
 * copy, the LM head (two launches where spill pairs run beside clusters of
 * two CTA pairs, see BD_PAIR_SPILL), merge + commit; 0 for an empty window.
 * Arguments as for bd_commit_step_ex (exec may be NULL; only its variant and
 * flags are read). Returns a negative bd_status if the arguments are
 * invalid or the device cannot run the library. Host-only: queues nothing. */
int bd_step_kernels(const bd_hidden* hidden, const bd_weight* weight, const bd_mask_state* mask_state,
                    const bd_tau_grid* tau_grid, const bd_exec* exec);

/* The work plan the LM head takes for a window of n_rows compacted rows
 * (masked positions of active blocks), as the compaction kernel computes it
 * on the device once N is known; host-only, for inspection and tests.
 * Writes min(n_out, 8) int32 words to `out` (host memory): N, the partial
 * slots per row over both LM-head launches (vocabulary parts times the CTAs
 * that write a partial per unit), the main launch's band size (runner
 * m-tiles) and parts, the spill launch's band size and parts (0, 0 without
 * one), the v-tile where the spill launch's range begins (the v-tile count
 * without one) and the spill launch's first slot. Arguments as for
 * bd_step_kernels; n_rows in 0..window positions. Returns the number of
 * words of the plan (8), or a negative bd_status. The plan never changes what
 * is computed. */
int bd_plan_header(const bd_hidden* hidden, const bd_weight* weight, const bd_mask_state* mask_state,
                   const bd_tau_grid* tau_grid, const bd_exec* exec, int32_t n_rows, int32_t* out, int32_t n_out);

/* ------------------------------------------------------------ tuning knobs --
 * Environment variables read at every call (none is needed; each changes how
 * the work is done, never what is computed):
 *   BD_E4M3_SPLIT=0      E4M3 heads not on the 8-bit path (see bd_exec.variant)
 *   BD_FUSED_DECODE=0    quantised heads decoded to a bf16 copy, not in the kernel
 *   BD_PAIR_MAX_P=n      the automatic choice takes the CTA-pair kernel for NVFP4
 *                        heads up to n window positions (default 8192)
 *   BD_PAIR_MC=1|2       single CTA pairs, or clusters of two pairs sharing each
 *                        head tile by multicast (default: clusters for windows of
 *                        at most 512 positions or more than 256 MiB of packed rows)
 *   BD_PAIR_SHARE=0|1    the two pairs of a cluster share head tiles (two token
 *                        groups, one v-tile at a time; default) or token rows (one
 *                        token group, two v-tiles at a time)
 *   BD_PAIR_SPILL=0|1    with clusters of two pairs, the CTA pairs that still fit
 *                        on the SMs the clusters leave free (4 on a 152-SM GB300)
 *                        take the last v-tiles in a second, concurrent launch
 *                        (default: on for more than 256 MiB of packed rows). The
 *                        split assumes those SMs are free: where other work holds
 *                        them, the spill launch runs after the clusters and the
 *                        LM head takes about twice as long; set 0 there
 *   BD_SPILL_PCT=n       a spill pair's time per v-tile against a cluster pair's,
 *                        in percent (default 100): sets the vocabulary split
 *   BD_PLAN_GM=n, BD_PLAN_GV=n   fix the work plan's band size (runner m-tiles)
 *                        or vocabulary part count; BD_PLAN_RR=1 takes its units
 *                        round-robin instead of in packed rounds
 *   BD_L2_HEAD, BD_L2_ROWS = 0|1|2   L2 eviction priority (first, normal, last) of
 *                        the head tiles and token rows (default 0 and 2)
 *   BD_TC_STAGES=3|4     pipeline stages of the one-CTA tensor-core kernel */

/* ------------------------------------------------ vocabulary-parallel split --
 * The head split by vocabulary rows over G ranks (or G calls on one device):
 * rank g holds rows [offset_g, offset_g + V_g) of W. The only exchange is
 * 12 bytes per position and rank: each rank's (max m, sum of exp(l - m),
 * lowest argmax a) over its rows, which combine exactly as the kernels'
 * vocabulary parts do: (m, s, a) + (m', s', a') = (M, s e^(m - M) + s' e^(m' - M),
 * the lowest id among the maxima), with M = max(m, m'); conf = 1 / s, token = a
 * (App. B.1: the mask-suppressed softmax over the whole vocabulary).
 *
 * Per-position partials, device arrays of P = n_seq * n_slots * block_len
 * entries each (or [n_parts, P] when gathered, part g at g * P):
 *   m : float32 max logit, -inf where the position has no prediction
 *   s : float32 sum of exp(l - m) over the shard's rows (0 there)
 *   a : int32 global vocabulary id of the lowest argmax (-1 there) */
typedef struct {
  float* m;
  float* s;
  int32_t* a;
} bd_partials;

/* Part 1: the LM head and its softmax statistics over one head shard. `shard`
 * holds vocabulary rows [vocab_offset, vocab_offset + shard->vocab) of the
 * head (any dtype bd_commit_step accepts; an E4M3 shard's scale covers its own
 * rows); mask_state->mask_token_id is a GLOBAL id (-1 = none), suppressed by
 * the shard that holds it. Writes `out` for every window position: the
 * partial of the masked positions of active blocks, (-inf, 0, -1) elsewhere.
 * exec: stream, workspace (bd_workspace_size with the shard as the head and
 * mask_token_id -1), variant; flags, out_counts and events must be 0 / NULL.
 * Errors as bd_commit_step_ex, plus BD_ERR_ARG for a negative offset or an
 * offset + vocab beyond 2^30; a shard whose only row is the mask token has
 * nothing to predict (BD_ERR_SHAPE): leave it out of the split. */
int bd_lmhead_partials(const bd_hidden* hidden, const bd_weight* shard, int64_t vocab_offset,
                       const bd_mask_state* mask_state, const bd_partials* out, const bd_exec* exec);

/* Part 2: merges the n_parts (1..4096) shards' partials of every position,
 * gathered as [n_parts, P] arrays (e.g. by an all-gather), and applies the
 * commit rule of bd_commit_step for the whole threshold grid; outputs as
 * bd_commit_step (tokens are global ids). Equal maxima in two shards go to
 * the lower id, as in one pass. exec: stream and out_counts; workspace,
 * flags and events must be NULL / 0. Needs no workspace. */
int bd_merge_commit(const bd_partials* gathered, int32_t n_parts, const bd_mask_state* mask_state,
                    const bd_tau_grid* tau_grid, int32_t* out_tokens, float* out_conf, uint32_t* out_commit,
                    const bd_exec* exec);

/* Synchronises `stream` (a cudaStream_t, NULL = legacy default), then returns
 * and clears the device-side status of the current device: BD_OK, or
 * BD_ERR_TIMEOUT if a kernel's bounded wait gave up since the last call (its
 * outputs are then invalid), or BD_ERR_CUDA if the synchronisation failed. */
int bd_get_device_status(void* stream);

/* Failure-detection self-test (the paper has no counterpart). Queues on
 * `stream` one small kernel that waits, through the same bounded wait the
 * tensor-core kernels use, on a barrier that nothing ever completes; after the
 * wait limit (about 1 s) it records the timeout in the device status word of
 * the current device and returns. The next bd_get_device_status then returns
 * BD_ERR_TIMEOUT and clears the word; the context stays usable. No fault, trap
 * or hang is involved. Returns BD_OK once queued (or BD_ERR_DEVICE / BD_ERR_CUDA). */
int bd_selftest_timeout(void* stream);

/* Static English text for a status code. Never NULL. */
const char* bd_status_string(int status);

/* Frees the library-owned workspaces and status words of every device, and
 * forgets the cached device address of bd_commit_step_static's array (the
 * next such call looks it up again, so the library stays usable after a
 * cudaDeviceReset that follows this call). No call may be in flight. */
int bd_shutdown(void);

/* Size of the device scratch array that bd_commit_step_static works in. */
#define BD_STATIC_SCRATCH_BYTES (32u * 1024u * 1024u)

/* The commit step without any allocation. The paper has no counterpart: this
 * is a service for callers that must not allocate device memory, such as code
 * running inside an allocator or memory-pool callback (cudaMalloc there would
 * re-enter the allocator), a process whose device memory is fully reserved by
 * a framework's caching allocator, or a latency-critical serving loop that
 * cannot afford cudaMalloc's implicit device-wide synchronisation.
 *
 * Same arguments and outputs as bd_commit_step, plus `stream` (a cudaStream_t,
 * NULL = legacy default stream). Instead of a workspace, the call works in one
 * file-scope device array of BD_STATIC_SCRATCH_BYTES (32 MiB) that every GPU
 * which loads the library holds until the process exits. It calls no
 * cudaMalloc, cudaFree or other allocating routine.
 *   - Size limit: a call whose workspace (bd_workspace_size) would exceed
 *     BD_STATIC_SCRATCH_BYTES returns BD_ERR_WORKSPACE before queuing anything
 *     (the 8 x 2 x 32, d = 2048, V = 151936 bf16 window needs about 3 MiB).
 *   - First call on a device: it looks up the array's device address with
 *     cudaGetSymbolAddress (the device must be current) and caches it; make
 *     that first call before any stream capture.
 *   - Sharing: every call on a device uses the same array, which keeps the
 *     previous call's contents (everything a call reads there it writes
 *     first). Calls that can overlap on the GPU (different streams, or
 *     different host threads) race on the array: serialise them.
 *   - Failures on the device: a bounded device-side wait that gives up is
 *     recorded in a status word inside the array (not in the word
 *     bd_get_device_status reads) and stays recorded, across later calls,
 *     until bd_static_device_status reads and clears it. */
int bd_commit_step_static(const bd_hidden* hidden, const bd_weight* weight,
                          const bd_mask_state* mask_state, const bd_tau_grid* tau_grid,
                          int32_t* out_tokens, float* out_conf, uint32_t* out_commit,
                          void* stream);

/* The device status of bd_commit_step_static on the current device (no paper
 * counterpart; allocates nothing either). Synchronises `stream`, then returns
 * and clears the status word in the array: BD_OK, BD_ERR_TIMEOUT if a bounded
 * wait of any static call gave up since the last read (that call's outputs
 * are invalid), BD_ERR_BOUNDS (bounds-checked build), or BD_ERR_CUDA.
 * Read it after the static calls whose outputs you use. */
int bd_static_device_status(void* stream);

/* The failure-detection self-test of bd_selftest_timeout aimed at the status
 * word of bd_commit_step_static's array (no paper counterpart): one small
 * kernel on `stream` waits about 1 s on a barrier nothing completes and
 * records the timeout there; the next bd_static_device_status returns
 * BD_ERR_TIMEOUT. No fault, trap or hang is involved. */
int bd_static_selftest_timeout(void* stream);

/* ---------------------------------------------- speculative verification --
 * The same LM head and fused softmax serve the verification step of
 * speculative decoding with the lossy typical-acceptance rule the paper tests
 * (typical-acceptance appendix): a draft token x is accepted when the target's
 * probability of it exceeds min(eps, sqrt(eps) * exp(-H)), H the entropy of the
 * target's next-token distribution; the lossless reference accepts x only when
 * it is the target's argmax (lossless-reference appendix). A request accepts
 * the longest prefix of its drafts that pass.
 *
 * Draft tokens of a verification batch, device memory:
 *   n_req    requests (>= 0)
 *   n_draft  draft tokens per request, 1..32
 *   draft    [n_req * n_draft] int32: draft token i of request q at
 *            q * n_draft + i; an entry outside [0, vocab) has probability 0
 * The hidden states then hold n_req * (n_draft + 1) rows: row
 * q * (n_draft + 1) + i is the target state whose next-token distribution
 * verifies draft token i (i < n_draft); the last row of a request gives the
 * token the target adds after the accepted prefix when every draft passes. */
typedef struct {
  int32_t n_req;
  int32_t n_draft;
  const int32_t* draft;
} bd_draft;

/* Typical-acceptance settings: HOST array eps[0..E-1], 1 <= E <= 31, each in
 * (0, 1] (a lower eps accepts more). Copied at call time. */
typedef struct {
  const float* eps;
  int32_t E;
} bd_eps_grid;

#define BD_ACCEPT_LOSSLESS_BIT 31 /* bit of out_accept set when the draft is the target's argmax */

/* One verification step, asynchronous on exec->stream (exec may be NULL).
 * Outputs, device arrays, all fully written (R = n_req * (n_draft + 1)):
 *   out_tokens   [R] int32  : the target's argmax (lowest index on ties)
 *   out_p_draft  [R] float  : target probability of the row's draft token (0 on
 *                             the last row of a request)
 *   out_entropy  [R] float  : entropy of the target distribution, in nats
 *   out_accept   [R] uint32 : bit k = accepted at eps[k]; bit 31 = lossless
 *                             (0 on the last row of a request)
 *   out_accepted [n_req * (E + 1)] int32 : accepted prefix length of request q
 *                             at eps[k] at q * (E + 1) + k, the lossless rule at
 *                             column E; accepted tokens for the target forward
 *                             are that length + 1
 * Same hidden / weight dtypes, alignment rules, variants and workspace rules
 * as bd_commit_step_ex (size from bd_verify_workspace_size); exec->out_counts
 * must be NULL. Errors: as bd_commit_step_ex, with BD_ERR_TAU for a bad eps
 * grid and BD_ERR_SHAPE for n_draft outside 1..32 or hidden->rows != R. */
int bd_verify_step(const bd_hidden* hidden, const bd_weight* weight, const bd_draft* draft,
                   const bd_eps_grid* eps, int32_t* out_tokens, float* out_p_draft, float* out_entropy,
                   uint32_t* out_accept, int32_t* out_accepted, const bd_exec* exec);

/* Bytes of device workspace bd_verify_step needs for these arguments (0 if invalid). */
size_t bd_verify_workspace_size(const bd_hidden* hidden, const bd_weight* weight, const bd_draft* draft,
                                const bd_eps_grid* eps);

/* ------------------------------------------------------- commit sweep --
 * The block-buffer update that follows the commit step in every decode step
 * (engine appendix: slot states; maximal-exact-commit appendix, proof part 1).
 *
 * The window's own state, updated in place, device memory:
 *   tokens      [P] int32 : the token each position holds (its content at
 *                           masked positions is irrelevant)
 *   pos_masked  [P] uint8 : 1 = still masked (the commit step's pos_masked)
 *   block_flags [n_seq * n_slots] : BD_BLOCK_* bits; BD_BLOCK_ACTIVE set =
 *                           an admitted block, clear = a placeholder slot
 *   n_seq, n_slots, block_len, mask_token_id as in bd_mask_state, with
 *   n_slots <= 64 and n_slots * block_len <= 4096 (block_len <= 64). */
typedef struct {
  int32_t n_seq;
  int32_t n_slots;
  int32_t block_len;
  int32_t mask_token_id;
  int32_t* tokens;
  uint8_t* pos_masked;
  uint8_t* block_flags;
} bd_window;

#define BD_SWEEP_ADMIT 1u           /* vacated slots return as admitted, all-masked blocks (else placeholders) */
#define BD_SWEEP_ELIGIBLE_OLDEST 2u /* afterwards only the oldest active block of a sequence is fallback-eligible */

/* One decode step's state update at the deployed threshold tau_index, on
 * `stream` (a cudaStream_t, NULL = legacy default), after the commit step on
 * the same stream (it may start while that step finishes and waits for it):
 *   1. every position that is masked, in an active block and has bit
 *      tau_index set in step_commit takes step_tokens[p] and is unmasked
 *      (other bits are ignored);
 *   2. the sweep visits each sequence's slots left to right and commits a
 *      block when it is active, has no masked position (complete, hence
 *      commit-ready under the default commit semantics) and its predecessor
 *      was committed (or it is the first slot), so chains commit at once;
 *   3. the c committed blocks leave the window for the cache: their tokens go
 *      to out_cache_tokens [P] at blocks (s * n_slots + j), j < c (the rest of
 *      that array is left untouched); out_n_committed[s] = c;
 *   4. the remaining slots shift left by c with their tokens, masks and flags;
 *      the c vacated slots at the end are mask-filled (tokens = mask_token_id,
 *      or -1 when it is -1) and get flags 0, or BD_BLOCK_ACTIVE with
 *      BD_SWEEP_ADMIT; with BD_SWEEP_ELIGIBLE_OLDEST the fallback bit is then
 *      moved to the first active slot of each sequence.
 * out_n_resolved [n_seq] (optional, may be NULL) receives the positions step 1
 * resolved. step_tokens / step_commit are the commit step's out_tokens /
 * out_commit. Afterwards no window block is active, complete and preceded
 * only by committed blocks (the paper's zero exact-committable but
 * uncommitted blocks).
 * With n_seq == 0 the call does nothing and every array may be NULL.
 * Errors (nothing queued): BD_ERR_NULL for a missing pointer; BD_ERR_SHAPE for
 * n_seq < 0, n_slots outside 1..64, block_len outside 1..64, n_slots * block_len > 4096,
 * or more than 2^24 positions; BD_ERR_ARG for tau_index outside 0..31 or
 * unknown option bits; BD_ERR_DEVICE off sm_103; BD_ERR_CUDA if the launch
 * fails. No allocation; calls on one window must be serialised. */
int bd_commit_sweep(const bd_window* window, const int32_t* step_tokens, const uint32_t* step_commit,
                    int32_t tau_index, uint32_t options, int32_t* out_cache_tokens, int32_t* out_n_committed,
                    int32_t* out_n_resolved, void* stream);

/* Library version as MAJOR*10000 + MINOR*100 + PATCH. */
int bd_version(void);

#ifdef __cplusplus
}
#endif

#endif /* BDCOMMIT_H */
