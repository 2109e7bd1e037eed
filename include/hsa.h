/*
 * hsa.h -- C ABI of libhsa, the GB300 (sm_103a) hot path of Heterogeneous Step
 * Allocation (HSA), a training-free step-skipping scheme for video diffusion
 * transformers (arXiv 2605.06892).
 *
 * One denoising iteration i of an HSA layer runs, in order:
 *   hsa_partition_active   active set A_i from the token groups     (Sec. 2.2, 2.5)
 *   hsa_gather_active      rows of A_i entering the block            (Sec. 2.3, step 1)
 *   hsa_kv_sync_scatter    fresh K/V of A_i into the layer's cache   (Sec. 2.3, step 2)
 *   hsa_active_attention   |A_i| queries against all N cached keys   (Sec. 2.3, step 3)
 *   hsa_cached_euler       all N latents advanced by one Euler step  (Sec. 2.4, Eq. 6)
 * and, once per sample, hsa_partition assigns tokens to step-budget groups
 * from a per-token statistic (Sec. 2.2 Eq. 3, Eq. 5; App. B, Eq. 7).
 *
 * Conventions for every call below:
 *  - Pointers named as device pointers must be device (or managed) memory of
 *    the current CUDA device; the caller owns all memory.  Host pointers are
 *    read before the call returns.  The library allocates nothing.
 *  - Work is enqueued on `stream` (NULL = the legacy default stream) and the
 *    call returns without waiting for it.  Argument checks happen on the host
 *    before any launch; a failed check launches nothing.
 *  - Errors that only the GPU can see (an index out of range, a non-finite
 *    statistic, a pipeline wait that ran out) do not fault the GPU: the kernel
 *    skips the offending access, records the error in a per-device word, and
 *    hsa_get_device_error() reports it.
 *  - Return values are hsa_status codes (0 = success, negative = error), or a
 *    documented non-negative count.
 *  - Token tensors are row-major with the token index outermost: a [N, H, D]
 *    tensor stores element (n, h, d) at offset (n*H + h)*D + d.
 */
#ifndef HSA_H
#define HSA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t. */
struct CUstream_st;
typedef struct CUstream_st *hsa_stream_t;

typedef enum {
    HSA_BF16 = 0,   /* bfloat16 storage, fp32 accumulation */
    HSA_F32 = 1     /* fp32 storage and arithmetic */
} hsa_dtype;

typedef enum {
    HSA_OK = 0,
    HSA_ERR_INVALID_ARG = -1,   /* null pointer, bad size, misaligned pointer */
    HSA_ERR_NOT_DIVISOR = -2,   /* a step budget does not divide T (Eq. 5) */
    HSA_ERR_BAD_COUNTS = -3,    /* group sizes negative or not summing to N */
    HSA_ERR_UNSUPPORTED = -4,   /* shape outside the supported set */
    HSA_ERR_NONFINITE = -5,     /* NaN or infinite statistic (device-side) */
    HSA_ERR_INDEX = -6,         /* index or group id out of range (device-side) */
    HSA_ERR_TIMEOUT = -7,       /* a bounded pipeline wait ran out (device-side) */
    HSA_ERR_CUDA = -8,          /* a CUDA runtime call or launch failed */
    HSA_ERR_WORKSPACE = -9      /* workspace missing, too small or misaligned */
} hsa_status;

/* Static string for a status code. */
const char *hsa_status_string(int status);

/* Library ABI version, currently 1. */
int hsa_version(void);

/* ------------------------------------------------------------ host helpers */

/* Checks step budgets and group sizes against Sec. 2.2: budgets[0] == T (the
 * baseline group G_1), budgets non-increasing, each a positive divisor of T
 * (Eq. 5); counts[k] >= 0 with sum N (counts may be NULL to skip that part).
 * Host only.  Returns HSA_OK, HSA_ERR_INVALID_ARG, HSA_ERR_NOT_DIVISOR or
 * HSA_ERR_BAD_COUNTS. */
int hsa_check_budgets(int T, const int *budgets, const int *counts, int K, int N);

/* Margin m = floor((1 - k) T / 2) of the phase-aware caching window (Sec. 2.5)
 * for k = window_pct / 100, in integer arithmetic.  Iterations i < m and
 * i > T - m - 1 run every token.  Returns m, or HSA_ERR_INVALID_ARG when
 * window_pct is outside [0, 100] or T < 1.  Host only. */
int hsa_window_margin(int T, int window_pct);

/* |A_i| from the group sizes: the sum of counts[k] over the groups active at
 * iteration iter (group k is active iff iter mod (T / budgets[k]) == 0, or
 * iter lies outside the caching window).  Host only, no device access, so a
 * caller can size buffers without synchronising.  Negative on bad input. */
int hsa_active_count(const int *budgets, const int *counts, int K, int T,
                     int iter, int window_pct);

/* Noise levels sigma_0 = 1 > sigma_1 > ... > sigma_T = 0 of the Euler solver
 * (Sec. 2.1, Eq. 2), computed in fp64 into the host array sigma[T + 1]:
 * t_i = 1 - i/T and sigma_i = shift*t_i / (1 + (shift - 1) t_i); shift = 1
 * gives the linear schedule.  The step of iteration i is sigma_{i+1} - sigma_i
 * (negative).  Host only. */
int hsa_sigma_schedule(int T, double shift, double *sigma);

/* ------------------------------------------------------------- a1 partition */

/* Bytes of device workspace hsa_partition needs for N tokens (0 for N == 0). */
size_t hsa_partition_workspace_bytes(int N);

/* Token partition (Sec. 2.2 Eq. 3) by the dynamic selection rule (App. B,
 * Eq. 7): tokens are ranked by stat ascending, ties broken by the lower token
 * index (-0 and +0 are equal); the counts[K-1] lowest go to group K-1 (the
 * smallest budget), the next counts[K-2] to group K-2, ..., the counts[0]
 * highest to group 0, the baseline group with budgets[0] == T.
 *   stat       device, fp32 [N]: per-token statistic (e.g. the mean L1
 *              relative change of the velocity, Eq. 7, or any score).
 *   budgets,   host, int [K]: step budget s_k and size |G_k| of each group,
 *   counts     checked as hsa_check_budgets does; 1 <= K <= 32.
 *   group_of   device, int32 [N], written: group id in [0, K) per token.
 *   workspace  device, >= hsa_partition_workspace_bytes(N) bytes, 256-byte
 *              aligned; overwritten.  Must not overlap stat or group_of.
 * A NaN or infinite statistic is reported as HSA_ERR_NONFINITE by
 * hsa_get_device_error; group_of is then unspecified. */
int hsa_partition(const float *stat, int N, int T, const int *budgets,
                  const int *counts, int K, int32_t *group_of, void *workspace,
                  size_t workspace_bytes, hsa_stream_t stream);

/* Largest N accepted by hsa_partition_static. */
#define HSA_PARTITION_STATIC_MAX_TOKENS 524288

/* hsa_partition without a workspace argument, for callers that cannot
 * allocate device memory for one: a plugin inside a host framework that owns
 * all device memory and offers it no allocator, or a latency-critical loop
 * that must not call cudaMalloc/cudaFree (they may synchronise the device).
 * The paper has no counterpart; the ranking and group assignment are exactly
 * those of hsa_partition (same arguments, same results).
 * Scratch: a fixed device array inside the library, about 8.5 MB, sized for
 * N <= HSA_PARTITION_STATIC_MAX_TOKENS (the sort that partitions layers of more
 * than 360448 tokens uses it; smaller layers take paths that need no scratch);
 * every GPU that loads the library's
 * partition module holds it until the process exits.  The CUDA runtime
 * reserves it when that module is loaded on a device: when the library is
 * loaded if CUDA_MODULE_LOADING=EAGER, otherwise (lazy loading, the default)
 * at the first partition call or symbol query on that device.  A host
 * framework that claims all device memory up front should therefore make one
 * call early, before it does.  Larger N returns HSA_ERR_UNSUPPORTED before any
 * launch.  Nothing is allocated: no cudaMalloc, cudaFree or allocating
 * library call is made.
 * The first call on a device looks up the array's device address (a CUDA
 * runtime query) for that device, so make that first call before any stream
 * capture.  Every call on a device shares the one array and finds the last
 * call's contents there (none need to start at zero); calls whose work
 * overlaps on the GPU (other streams, or other host threads) race on it and
 * must be serialised by the caller. */
int hsa_partition_static(const float *stat, int N, int T, const int *budgets,
                         const int *counts, int K, int32_t *group_of,
                         hsa_stream_t stream);

/* Statistics for the other token allocation strategies of App. B, to be
 * ranked by hsa_partition (the random strategy R ranks any random statistic
 * the caller draws):
 *  - uniform allocation (U): stat[n] = top 24 bits of (n+1) * 2654435769 mod
 *    2^32 (golden-ratio sequence), an exact integer in fp32.  Each group then
 *    holds the tokens of one interval of the sequence, which are spaced by at
 *    most three distinct gaps over the whole token range ("maximally spread").
 *  - first-frame reservation (F): stat[n] = FLT_MAX for n < frame_tokens (the
 *    first latent frame, (H_l/2)*(W_l/2) tokens in row-major order), applied
 *    on top of a random statistic; with counts[0] >= frame_tokens every
 *    first-frame token lands in the baseline group.
 *   stat  device, fp32 [N], written (U) or updated in place (F). */
int hsa_uniform_stat(float *stat, int N, hsa_stream_t stream);
int hsa_reserve_first_frame(float *stat, int N, int frame_tokens, hsa_stream_t stream);

/* Token reordering (Sec. 2.5), applied once before the denoising loop: new
 * position r holds old token order[r]; the tokens of groups 1..K-1 come first
 * in token order, then the n_baseline tokens of the baseline group (group 0),
 * also in token order.  The KV cache then only needs the prefix of
 * M = N - n_baseline rows, because the baseline group is active at every
 * iteration (see hsa_active_attention_prefix).
 *   group_of   device, int32 [N]; exactly n_baseline entries are 0.
 *   order      device, int32 [N], written (new -> old).  Reorder a per-token
 *              tensor with hsa_gather_active(src, .., order, N, dst).
 *   where      device, int32 [N] or NULL, written (old -> new); undo the
 *              reordering with hsa_gather_active(.., where, N, ..).
 *   group_new  device, int32 [N] or NULL, written: group_of[order[r]].
 * A group_of that disagrees with n_baseline is reported as HSA_ERR_INDEX. */
int hsa_reorder_tokens(const int32_t *group_of, int N, int n_baseline, int32_t *order,
                       int32_t *where, int32_t *group_new, hsa_stream_t stream);

/* ---------------------------------------------------- a2 active set per step */

/* Active set A_i (Sec. 2.3; Fig. 1): token n is active at iteration iter iff
 * iter mod (T / budgets[group_of[n]]) == 0 (Sec. 2.2) or iter is outside the
 * caching window of window_pct percent (Sec. 2.5; 100 = no window).
 *   group_of  device, int32 [N] in [0, K).
 *   idx       device, int32 [>= |A_i|], written: active token ids ascending.
 *   pos       device, int32 [N] or NULL, written: rank of n in idx, or -1.
 * |A_i| is hsa_active_count(...) of the same groups, known on the host.  A
 * group id outside [0, K) is reported as HSA_ERR_INDEX (that token is then
 * treated as skipped). */
int hsa_partition_active(const int32_t *group_of, int N, int T,
                         const int *budgets, int K, int iter, int window_pct,
                         int32_t *idx, int32_t *pos, hsa_stream_t stream);

/* --------------------------------------------------------------- a3 gather */

/* dst[j, :] = src[idx[j], :] for j < n_active: the rows of the active tokens
 * that enter the transformer block (Sec. 2.3, step 1).
 *   src       device, [N, row_bytes] (any element type).
 *   row_bytes row size in bytes, a positive multiple of 16; src and dst
 *             16-byte aligned.
 *   idx       device, int32 [n_active], values in [0, N).
 *   dst       device, [n_active, row_bytes], written.
 * An index outside [0, N) leaves its dst row untouched (HSA_ERR_INDEX). */
int hsa_gather_active(const void *src, size_t row_bytes, int N,
                      const int32_t *idx, int n_active, void *dst,
                      hsa_stream_t stream);

/* ------------------------------------------------------ a4 KV-cache scatter */

/* KV-cache synchronisation (Sec. 2.3, step 2): k_cache[idx[j]] = k_fresh[j]
 * and v_cache[idx[j]] = v_fresh[j] for j < n_active, one launch for both;
 * rows of skipped tokens are left untouched.
 *   k_cache, v_cache  device, [N, H, D] of dtype, updated in place.
 *   k_fresh, v_fresh  device, [n_active, H, D] of dtype (K/V of A_i).
 *   idx               device, int32 [n_active], distinct values in [0, N)
 *                     (A_i never repeats a token; repeated ids race, and
 *                     hsa_check_indices detects them).
 * H*D*sizeof(dtype) must be a multiple of 16 bytes and every pointer 16-byte
 * aligned.  An index outside [0, N) skips its row (HSA_ERR_INDEX). */
int hsa_kv_sync_scatter(void *k_cache, void *v_cache, const void *k_fresh,
                        const void *v_fresh, const int32_t *idx, int n_active,
                        int N, int H, int D, hsa_dtype dtype,
                        hsa_stream_t stream);

/* Opt-in check of an index array, for debugging (Sec. 2.2: the groups are
 * disjoint, so an active set never names a token twice, and the KV scatter
 * above relies on that).  Reports HSA_ERR_INDEX through hsa_get_device_error
 * when an entry of idx lies outside [0, N) or a value appears more than once;
 * the hot-path calls do not make this check themselves.
 *   idx        device, int32 [n], any order.
 *   workspace  device, >= hsa_check_indices_workspace_bytes(N) bytes (one
 *              bit per token), 256-byte aligned; overwritten.  Calls sharing
 *              one workspace must not overlap on the GPU.
 * Two launches (clear the bitmap, then mark); returns HSA_ERR_WORKSPACE when
 * the workspace is missing, too small or misaligned. */
size_t hsa_check_indices_workspace_bytes(int N);
int hsa_check_indices(const int32_t *idx, int n, int N, void *workspace,
                      size_t workspace_bytes, hsa_stream_t stream);

/* Rotary position embedding of the active rows (Sec. 2.3: the positional
 * frequencies are subsampled to match A_i).  The table holds, for every token
 * n of the grid and rotation pair i, (cos, sin) of its angle; the calls below
 * rotate an active row j by the table row of its token idx[j], pair (x0, x1)
 * of each head becoming (fma(x0, c, -(x1 s)), fma(x0, s, x1 c)) in fp32,
 * rounded to bf16.
 *
 * hsa_rope_table: host-side table of a (F, Hh, Ww) grid, tokens row-major:
 * the D/2 pairs form three bands, p_t = D/2 - 2 floor(D/6) pairs for the
 * frame, then floor(D/6) each for the row and the column; pair i of a band
 * of p pairs turns by pos * theta^(-i/p).  table: host, fp32 [N, D/2, 2]
 * written (fp64 math, rounded once).  D a multiple of 8.
 *
 * hsa_rope_rows: x device bf16 [n, H, D], rotated in place (e.g. Q[A_i]).
 * hsa_kv_sync_scatter_rope: hsa_kv_sync_scatter (bf16) with the fresh K rows
 * rotated on their way into the cache; V is copied unchanged.
 *   table  device, fp32 [N, D/2, 2], 16-byte aligned.
 * An idx entry outside [0, N) skips its row (HSA_ERR_INDEX). */
int hsa_rope_table(int F, int Hh, int Ww, int D, double theta, float *table);
int hsa_rope_rows(void *x, const int32_t *idx, int n, int H, int D, const float *table, int N,
                  hsa_stream_t stream);
int hsa_kv_sync_scatter_rope(void *k_cache, void *v_cache, const void *k_fresh,
                             const void *v_fresh, const int32_t *idx, int n_active, int N,
                             int H, int D, const float *table, hsa_stream_t stream);

/* -------------------------------------------------- a5 active attention */

/* Full-context attention of the active queries (Sec. 2.3, step 3; Sec. 2.1
 * "Self-attention"), per head h and active row j:
 *   out[j, h, :] = sum_n softmax_n(scale * <q_{r,h}, k_{n,h}>) v_{n,h}
 * over all N cached keys, with r = q_idx[j] when q_idx is given (q is then
 * [N, H, D] and rows are read by index) or r = j (q is compact
 * [n_active, H, D]).  No mask; scale <= 0 selects 1/sqrt(D).  The cost is
 * O(|A_i| N) instead of O(N^2).
 *   k_cache, v_cache  device, [N, H, D] of dtype.
 *   out               device, [n_active, H, D] of dtype, written.
 *   workspace         device, optional (NULL = none), 16-byte aligned; see
 *                     hsa_active_attention_workspace_bytes.  With it, the
 *                     (query block, head) units of the last, partly filled
 *                     wave of CTAs are split along the keys and merged
 *                     afterwards, so that the last wave finishes sooner;
 *                     without it the result is the same up to rounding order.
 *                     Overwritten; calls using one workspace must not overlap.
 * Supported: D in {64, 128}; H >= 1; 1 <= N < 2^31; 0 <= n_active.
 * HSA_BF16 runs on the tensor cores (tcgen05, fp32 accumulation); HSA_F32
 * runs in fp32 on the CUDA cores and ignores the workspace.  Pointers must be
 * 16-byte aligned.  A q_idx entry outside [0, N) yields a zero query row
 * (HSA_ERR_INDEX). */
int hsa_active_attention(const void *q, const int32_t *q_idx, int n_active,
                         const void *k_cache, const void *v_cache, int N, int H,
                         int D, float scale, void *out, hsa_dtype dtype,
                         void *workspace, size_t workspace_bytes,
                         hsa_stream_t stream);

/* hsa_active_attention over keys held in two sources, read in order: the M
 * rows of k_cache / v_cache ([M, H, D], the cache of the non-baseline prefix
 * after token reordering, Sec. 2.5) followed by the B rows of k_base /
 * v_base ([B, H, D], the fresh K/V of the baseline group, which is active at
 * every iteration).  Keys total M + B >= 1; either source may be empty.
 * q_idx, when given, indexes a [M + B, H, D] query tensor.  Everything else
 * as hsa_active_attention (which is this call with B = 0). */
int hsa_active_attention_prefix(const void *q, const int32_t *q_idx, int n_active,
                                const void *k_cache, const void *v_cache, int M,
                                const void *k_base, const void *v_base, int B, int H, int D,
                                float scale, void *out, hsa_dtype dtype, void *workspace,
                                size_t workspace_bytes, hsa_stream_t stream);

/* Workspace bytes that let hsa_active_attention balance its last wave (0 when
 * the dtype or shape takes none).  Depends only on the device's SM count and
 * D, so one buffer serves every call of a given D on that device. */
size_t hsa_active_attention_workspace_bytes(int n_active, int N, int H, int D,
                                            hsa_dtype dtype);

/* ------------------------------------------------------- a6 cached Euler */

/* Cached Euler update (Sec. 2.4, Eq. 6) of all N tokens in one pass: when
 * pos[n] >= 0 the velocity cache takes the fresh velocity,
 * v_cache[n] = v_fresh[pos[n]]; then x[n] = fma(v_cache[n], dsigma, x[n])
 * (fp32, one rounding per element), dsigma = sigma_{i+1} - sigma_i.
 *   x, v_cache  device, fp32 [N, C], updated in place.
 *   v_fresh     device, fp32 [n_active, C] (velocities of A_i) or NULL.
 *   pos         device, int32 [N] (as written by hsa_partition_active) or
 *               NULL; both NULL = no refresh.
 *   n_fresh     rows of v_fresh; a pos value outside [-1, n_fresh) (above
 *               the range, or any negative value other than -1) is treated
 *               as -1 and reported as HSA_ERR_INDEX.
 * C must be a positive multiple of 4 and the pointers 16-byte aligned. */
int hsa_cached_euler(float *x, float *v_cache, const float *v_fresh,
                     const int32_t *pos, int n_fresh, int N, int C, float dsigma,
                     hsa_stream_t stream);

/* Cached Euler update fused with the velocity statistic of the dynamic token
 * selection (App. B, Eq. 7), for the initial full-budget iterations whose
 * velocities rank the tokens.  For every token with pos[n] >= 0 it first adds
 *   weight * ||v_fresh[pos[n]] - v_cache[n]||_1 / ||v_fresh[pos[n]]||_1
 * to stat[n] (v_cache[n] still holds the previous step's velocity; a zero
 * denominator adds 0 when the numerator is 0 and weight * FLT_MAX otherwise),
 * then performs exactly hsa_cached_euler.  With weight = 1/(number of steps
 * averaged) stat ends as the mean relative change, ready for hsa_partition.
 *   stat  device, fp32 [N], accumulated in place (fp32 fma).
 * pos and v_fresh are required; other arguments as for hsa_cached_euler. */
int hsa_cached_euler_l1rel(float *x, float *v_cache, const float *v_fresh,
                           const int32_t *pos, int n_fresh, int N, int C, float dsigma,
                           float *stat, float weight, hsa_stream_t stream);

/* ------------------------------------------------------------------ errors */

/* Waits for `stream`, then reports and clears the device-side errors recorded
 * on the current device since the last call: HSA_ERR_TIMEOUT if a bounded wait
 * ran out, else HSA_ERR_NONFINITE, else HSA_ERR_INDEX, else HSA_OK; or
 * HSA_ERR_CUDA if the wait itself failed.  The word is per device, shared by
 * every stream and thread. */
int hsa_get_device_error(hsa_stream_t stream);

/* Number of kernels this library has launched in this process, on any device
 * or stream, since it was loaded (a host-side counter, incremented when a
 * launch is enqueued; a call that fails its argument checks adds nothing).
 * A call captured into a CUDA graph counts once, at capture; replays of the
 * graph are not counted.  Never fails; takes no GPU. */
unsigned long long hsa_launch_count(void);

#ifdef __cplusplus
}
#endif

#endif /* HSA_H */
