/*
 * libtula_ags -- the data-parallel optimizer step of Adaptive Gradient
 * Scaling (AGS) from Tula (arXiv 2603.18112), on one NVIDIA GB300 (sm_103a).
 *
 * One step, per the paper:
 *   1. the mean of K replica gradient buffers (Eq. 1c: synchronous data-
 *      parallel SGD averages the N workers' gradients; here the K replicas
 *      sit in one GPU's HBM and the all-reduce becomes an in-place mean);
 *   2. per-layer squared norms of the mean gradient (and of the weights);
 *   3. the gradient-variability metric Delta(G) = |(|G_i|^2 - |G_{i-1}|^2) /
 *      |G_{i-1}|^2| (Eq. 5) and the branch of Algorithm 1: scaled when
 *      Delta < delta, unscaled (sensitive phase) otherwise;
 *   4. the scaled update (Eq. 7b, Algorithm 1) applied through the wrapped
 *      SGD optimizer with momentum and weight decay (Sec. IV-A, IV-B).
 *
 * Conventions for every entry point:
 *   - Tensors are fp32, in caller-owned DEVICE memory, 4-byte aligned; the
 *     fast path wants them 16-byte aligned (misaligned tensors take a scalar
 *     path with the same results).
 *   - Arrays of pointers (param_ptrs, grad_ptrs, ...) and numels are HOST
 *     arrays, read during the call only.
 *   - Calls are asynchronous on `stream` (a cudaStream_t; NULL = the legacy
 *     default stream).  They allocate nothing, never synchronize the host,
 *     and perform no host<->device copy, so they can be captured into a CUDA
 *     graph.  Results are bitwise reproducible run to run, and independent of
 *     the grid size (the reduction order depends on the numels only).
 *   - The workspace is caller-owned device memory of at least
 *     tula_ags_workspace_size() bytes, ZERO-FILLED before its first use; the
 *     library leaves it re-usable (its counters back at zero) after every
 *     call.  Calls that share a workspace must be ordered (one stream).
 *   - Return value: TULA_OK (0) or a negative TULA_ERR_* code.  Argument
 *     errors are detected on the host before anything is enqueued.  After
 *     TULA_ERR_CUDA (a launch failed part way) or a nonzero
 *     tula_ags_workspace_error() (a bounded wait inside a kernel ran out), the
 *     step may be partly applied: zero the workspace again before reusing it.
 *   - Element-wise arithmetic is IEEE fp32, one rounding per operation, in the
 *     order written below (no fused multiply-add).  Squared norms are fp32 sums
 *     within a tile (<= 9216 elements; relative error below ~4e-6) added across
 *     tiles exactly, in integers (fixed point from 2^-352 to 2^320, by L2
 *     atomics, so the order tiles land in cannot change a bit), then rounded
 *     once to fp64.  A tile whose fp32 sums would overflow (a lane sum above
 *     2^120) or lose precision to underflow (every lane sum below 2^-100, zero
 *     included) is summed again with its elements scaled by an exact power of two,
 *     and elements loaded one by one (tails, misaligned tensors) are squared in
 *     fp64, so these norms hold over the whole fp32 range.  Norms that feed a
 *     coefficient (gradscale refresh, LARS) split every square exactly into two
 *     fp32 parts, add them as float-float pairs per lane and in fp64 across lanes
 *     (relative error ~1e-14), then exactly across tiles; a tile whose pairs cannot hold that (a
 *     square that overflows, or sums below 2^-77) is redone with exact fp64
 *     squares, so these norms keep that precision over the whole fp32 range.
 */
#ifndef TULA_AGS_H
#define TULA_AGS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define TULA_AGS_VERSION 1

#define TULA_OK 0
#define TULA_ERR_ARG (-1)         /* NULL where a pointer is required, n_tensors < 1, K outside
                                     [1, TULA_MAX_K], numel < 0, a tensor above the size limit
                                     (see tula_ags_step), unaligned fp32 pointer, bad enum,
                                     mom_ptrs NULL with momentum != 0, refresh with K == 1 */
#define TULA_ERR_WORKSPACE (-2)   /* workspace NULL or smaller than tula_ags_workspace_size() */
#define TULA_ERR_CUDA (-3)        /* a kernel launch failed; see tula_ags_last_cuda_error() */
#define TULA_ERR_UNSUPPORTED (-4) /* a valid but unimplemented combination of options */
#define TULA_ERR_SCRATCH_LIMIT (-5) /* tula_ags_step_static_scratch: the tensor list needs more
                                       scratch than TULA_STATIC_SCRATCH_BYTES */
#define TULA_ERR_NO_MEMORY (-6)   /* host memory for launch tables or a plan could not be
                                     allocated; nothing was enqueued */

#define TULA_MAX_K 16

/* How the per-tensor coefficient c_p on the gradient is chosen. */
#define TULA_RULE_AGS 0    /* Algorithm 1: c_p = gradscale_p when Delta < delta, else 1 */
#define TULA_RULE_NONE 1   /* vanilla large-batch training (LBT): c_p = 1 */
#define TULA_RULE_LARS 2   /* prior art named in Sec. V-B: c_p = lars_trust * |w_p| / |g_p|,
                              every step (1 when either norm is 0) */
#define TULA_RULE_STATIC 3 /* static scaling U(s) of Eq. 8: c_p = static_s when Delta < delta */

/* Granularity of gradscale (Algorithm 1 keeps one entry per parameter). */
#define TULA_SCALE_PER_TENSOR 0  /* one factor per tensor: hp->scale[p] */
#define TULA_SCALE_PER_ELEMENT 1 /* one factor per element: hp->scale_elem[p][j] */

#define TULA_BRANCH_AUTO 0     /* Algorithm 1's test Delta < delta */
#define TULA_BRANCH_SCALED 1   /* force the scaled branch (tests) */
#define TULA_BRANCH_UNSCALED 2 /* force the unscaled branch (tests) */

/* hp->state, device fp64 [TULA_STATE_LEN]; zero-filled = before the first step. */
#define TULA_STATE_G2_PREV 0 /* |G_{i-1}|^2 of Eq. 5 (after a step: that step's |G|^2) */
#define TULA_STATE_STEPS 1   /* steps done */
#define TULA_STATE_DELTA 2   /* Delta of the last step (+inf at the first step) */
#define TULA_STATE_SCALED 3  /* 1 if the last step took the scaled branch, else 0 */
#define TULA_STATE_LEN 4

/* Per-layer statistics rows, device fp64 [n_tensors][TULA_STATS_LEN]. */
#define TULA_STAT_W_SQ 0      /* |w_p|^2 before the update */
#define TULA_STAT_G_SQ 1      /* |gbar_p|^2, gbar = mean of the K replicas */
#define TULA_STAT_G0_SQ 2     /* |g_{0,p}|^2, replica 0 before averaging */
#define TULA_STAT_W_NORM 3    /* |w_p| */
#define TULA_STAT_G_NORM 4    /* |gbar_p| */
#define TULA_STAT_RATIO 5     /* |w_p| / |gbar_p|: the per-layer ratio LARS scales the learning
                                 rate by (Sec. V-B); 0 when |gbar_p| = 0 */
#define TULA_STAT_COEF 6      /* c_p applied to the gradient this step (NaN: per-element scale) */
#define TULA_STAT_SCALE 7     /* gradscale_p after the step (0 without a per-tensor scale) */
#define TULA_STATS_LEN 8

typedef struct tula_ags_hparams {
    int K;             /* replica gradient buffers, 1 .. TULA_MAX_K */
    int rule;          /* TULA_RULE_* (default AGS) */
    int granularity;   /* TULA_SCALE_* (default PER_TENSOR) */
    int force_branch;  /* TULA_BRANCH_* (default AUTO) */
    int refresh_scale; /* 1: after this step's update, run UpdateGradScale of Algorithm 1 with
                          g_small = replica 0 (a sub-batch of the large batch, same weights) and
                          g_large = the mean: gradscale_p = min(|g_0p| / (|gbar_p| + eps), s_max).
                          Needs K > 1 and PER_TENSOR; the step itself uses the old gradscale. */
    float delta;       /* threshold on Delta (default 0.5, Sec. III-C and IV-B) */
    float eps;         /* stability term of UpdateGradScale (default 1e-8, Algorithm 1) */
    float s_max;       /* bound on gradscale, sqrt(b_large / b_small) (default sqrt(K)) */
    float static_s;    /* s of Eq. 8 for TULA_RULE_STATIC (default 1) */
    float lars_trust;  /* trust coefficient for TULA_RULE_LARS (default 1).  c_p is about
                          lars_trust * |w_p| / |gbar_p|, so a step moves w by roughly
                          lr * lars_trust * |w| / (1 - momentum): with lr 0.1 and momentum 0.9,
                          a trust of 1 doubles |w| per step.  Values near 1e-3 keep it small. */
    float *scale;                 /* device fp32 [n_tensors]: gradscale per tensor (AGS, PER_TENSOR);
                                     written when refresh_scale is set */
    float *const *scale_elem;     /* HOST array of n_tensors device fp32 pointers: gradscale per
                                     element (AGS, PER_ELEMENT); read only when scaled */
    double *state;                /* device fp64 [TULA_STATE_LEN], read and written */
    double *layer_stats;          /* device fp64 [n_tensors][TULA_STATS_LEN], or NULL */
    void *workspace;              /* device, >= tula_ags_workspace_size(), zero before first use */
    size_t workspace_bytes;
    int grid_ctas;                /* CTAs per launch; 0 = one wave of resident CTAs (results do
                                     not depend on it) */
    void *trace_events[5];        /* optional cudaEvent_t (NULL = none), recorded on `stream`:
                                     [0] before the reduction kernel(s), [1] after them,
                                     [2] after the pass-1 finish (before the update kernel),
                                     [3] after the update kernel(s), [4] the end of the step
                                     (after the finish that follows the update, when the step
                                     has statistics or refreshes the gradscale).  A recorded
                                     event keeps the next kernel from starting early, so steps
                                     that record events run slightly slower. */
} tula_ags_hparams;

/* Fills *hp with the paper's defaults for K replicas: AGS, per tensor, automatic branch,
 * delta 0.5, eps 1e-8, s_max sqrt(K) (b_small = one replica's share of the large batch),
 * static_s 1, lars_trust 1; all pointers NULL, grid_ctas 0. */
void tula_ags_default_hparams(tula_ags_hparams *hp, int K);

/* Bytes of workspace needed for this list of tensor sizes and K replicas (host only): about
 * 1.6 KB per tensor (accumulators and per-tensor sums), whatever the tensors' sizes. */
int tula_ags_workspace_size(const int64_t *numels, int n_tensors, int K, size_t *bytes);

/*
 * One AGS optimizer step over n_tensors tensors (the whole model).
 *   param_ptrs[p]          w_p, device fp32 [numels[p]], updated in place
 *   grad_ptrs[k*n + p]     replica k of the gradient of tensor p, device fp32; when K > 1
 *                          grad_ptrs[0*n + p] receives the mean gbar_p (an in-place all-reduce);
 *                          the other replicas are only read
 *   mom_ptrs[p]            momentum buffer m_p, device fp32, updated in place; mom_ptrs may be
 *                          NULL only when momentum == 0 (then w <- w - lr * d)
 *   numels[p] >= 0         element counts (0 = skipped); all tensors together may span
 *                          fewer than 2^31 tiles of min(tula_ags_chunk_elems(1, K + 1),
 *                          tula_ags_chunk_elems(2, 4)) elements (K + 2 in place of K + 1
 *                          when K = 1; an empty tensor counts as one tile): about 3.3e12
 *                          elements for K <= 4, 1.9e12 at K = 8, 8.2e11 at K = 16, more
 *                          than any GB300 holds; a longer list gives TULA_ERR_ARG
 * Per element, with c the coefficient of the rule (Algorithm 1, Eq. 8):
 *   gbar = (((g_0 + g_1) + ...) + g_{K-1}) / K
 *   d    = c * gbar + weight_decay * w
 *   m    = momentum * m + d            (zero-filled m = torch.optim.SGD's first step)
 *   w    = w - lr * m
 * Also updates hp->state and, when given, hp->layer_stats and (refresh) hp->scale.
 */
int tula_ags_step(float *const *param_ptrs, float *const *grad_ptrs, float *const *mom_ptrs,
                  const int64_t *numels, int n_tensors, float lr, float momentum,
                  float weight_decay, const tula_ags_hparams *hp, void *stream);

/*
 * A plan: the same step as tula_ags_step for a training loop that steps one fixed set of tensors
 * again and again.  tula_ags_plan_create checks the sizes and pointers once and copies them;
 * each tula_ags_plan_step then checks only hp and the scalars, and the launch tables (sizes and
 * pointers of up to ~31 KB per kernel launch) are built by the first step of each kernel variant
 * and reused by every later one.  Results are those of tula_ags_step bit for bit.
 *   tula_ags_plan_create: arguments as tula_ags_step.  Of hp only K and scale_elem are read:
 *     the per-element gradscale buffers, when given, are copied with the rest and are the ones
 *     every step of the plan uses (a step with PER_ELEMENT needs them).  The arrays and hp may
 *     be freed on return; the tensors must stay allocated until the plan is destroyed.  Binds
 *     the plan to the current CUDA device.  *plan_out receives the plan (NULL on error).
 *     Errors: TULA_ERR_ARG (as tula_ags_step, or plan_out NULL), TULA_ERR_CUDA (no current
 *     device), TULA_ERR_NO_MEMORY.  Allocates host memory only.
 *   tula_ags_plan_step: lr, momentum, weight_decay and hp as tula_ags_step; hp->K must be the
 *     plan's, and hp->scale_elem is ignored.  Every other field (rule, granularity, branch,
 *     refresh, scale, state, layer_stats, workspace, grid_ctas, trace_events) may change from
 *     one call to the next.  Momentum != 0 needs a plan created with momentum buffers.  Errors
 *     as tula_ags_step, and TULA_ERR_ARG when the current device is not the plan's.
 *   tula_ags_plan_destroy: frees the plan (NULL is a no-op).  Launches already issued do not
 *     use it, so it may be destroyed as soon as the last tula_ags_plan_step has returned.
 * A plan is not thread-safe: one host thread at a time may call tula_ags_plan_step on it.
 */
typedef struct tula_ags_plan tula_ags_plan;
int tula_ags_plan_create(float *const *param_ptrs, float *const *grad_ptrs,
                         float *const *mom_ptrs, const int64_t *numels, int n_tensors,
                         const tula_ags_hparams *hp, tula_ags_plan **plan_out);
int tula_ags_plan_step(tula_ags_plan *plan, float lr, float momentum, float weight_decay,
                       const tula_ags_hparams *hp, void *stream);
int tula_ags_plan_destroy(tula_ags_plan *plan);

/*
 * A step sharded over ranks (one rank per GPU; the paper trains data-parallel with DDP, Sec.
 * IV-A).  Each rank owns whole tensors and calls, with its own tensors only:
 *   1. tula_ags_shard_reduce: pass 1 on its tensors -- the mean of its K replicas (Eq. 1c) and
 *      their norms, kept in its workspace -- and its share of |G|^2 (Eq. 5) into g2_share;
 *   2. an exchange of the shares that the caller makes (e.g. an all-reduce of the
 *      TULA_G2_SHARE_WORDS uint64 words with an integer SUM over the ranks, in any order);
 *   3. tula_ags_shard_update with the summed shares: Delta and the branch of Algorithm 1 from the
 *      whole model's |G|^2, then the coefficients and the update of its tensors.
 * A share is an exact integer: words 0-20 the 32-bit digits (from 2^-352) of the sum of this
 * rank's tile partials of |gbar|^2 with carries in their high halves, word 21 the number of inf
 * partials, word 22 the number of NaN partials, word 23 zero.  Integer addition has no order, so
 * every rank takes the same |G|^2, Delta and branch, equal bit for bit to those of one
 * tula_ags_step over all tensors (tiles are cut per tensor, so each tensor's norms are the same
 * wherever it lives); the ranks together may span fewer than 2^31 pass-1 tiles.
 * Arguments as tula_ags_step, with the rank's tensors; hp (workspace sized for the rank's
 * tensors, state, scale, layer_stats) must be the same in both calls, and no other call may use
 * the workspace between them.  g2_share, g2_total: device uint64 [TULA_G2_SHARE_WORDS], 8-byte
 * aligned (TULA_ERR_ARG otherwise); g2_share is written, g2_total read.  Asynchronous on
 * `stream`; the exchange must be ordered between the two calls.
 */
#define TULA_G2_SHARE_WORDS 24
int tula_ags_shard_reduce(float *const *param_ptrs, float *const *grad_ptrs,
                          float *const *mom_ptrs, const int64_t *numels, int n_tensors,
                          float momentum, const tula_ags_hparams *hp, uint64_t *g2_share,
                          void *stream);
int tula_ags_shard_update(float *const *param_ptrs, float *const *grad_ptrs,
                          float *const *mom_ptrs, const int64_t *numels, int n_tensors, float lr,
                          float momentum, float weight_decay, const tula_ags_hparams *hp,
                          const uint64_t *g2_total, void *stream);

/*
 * Per-layer statistics without an update (read-only on every tensor): rows of
 * TULA_STATS_LEN fp64 as above, columns TULA_STAT_COEF and TULA_STAT_SCALE set to 0.
 * grad_ptrs[k*n + p] as in tula_ags_step.  stats_out: device fp64 [n_tensors][8].
 * Paper: TulaOptimizer wraps the training optimizer and tracks the gradient norm of every
 * parameter tensor (Sec. IV-A); the squared norms of the mean gradient are the per-layer terms
 * of |G|^2 in Eq. 5, those of replica 0 (a small-batch gradient at the same weights) are the
 * small-batch norms of Algorithm 1's UpdateGradScale, and |w_p| / |gbar_p| is the per-layer ratio
 * by which LARS scales the learning rate (Sec. V-B).
 */
int tula_layer_stats(const float *const *param_ptrs, const float *const *grad_ptrs, int K,
                     const int64_t *numels, int n_tensors, double *stats_out, void *workspace,
                     size_t workspace_bytes, void *stream);

/*
 * UpdateGradScale of Algorithm 1 from a small-batch gradient g_small[p] and the large-batch
 * gradient g_large[p] (device fp32), with hp->eps and hp->s_max:
 *   PER_TENSOR  (hp->scale[p]):       min(|g_small_p| / (|g_large_p| + eps), s_max), fp64, rounded
 *   PER_ELEMENT (hp->scale_elem[p][j]): fminf(|g_small / (g_large + eps)|, s_max), fp32
 * Uses hp->workspace (PER_TENSOR); hp->state is not touched.
 */
int tula_ags_update_scale(const float *const *g_small, const float *const *g_large,
                          const int64_t *numels, int n_tensors, const tula_ags_hparams *hp,
                          void *stream);

/*
 * tula_ags_step_static_scratch -- the same optimizer step as tula_ags_step, for callers that
 * cannot allocate device memory. (The paper has no counterpart; this is a deployment aid.)
 *
 * Who needs it: code that runs inside a host framework which owns every device allocation and
 * forbids foreign ones, code on a latency-critical path where cudaMalloc's implicit device-wide
 * synchronization is not acceptable, and plain C callers whose fixed call signature leaves no
 * place to keep a workspace between calls.  Such a caller still passes every input and output
 * (tensors, hp->scale, hp->state, hp->layer_stats); only the scratch moves.
 *
 * The scratch that tula_ags_step takes from hp->workspace (chunk partial sums, per-tensor sums,
 * counters, coefficients) lives instead in one file-scope __device__ array of
 * TULA_STATIC_SCRATCH_BYTES (16 MiB) inside this library.  Every GPU that loads the library holds
 * that array until the process exits.  hp->workspace and hp->workspace_bytes are ignored.
 *
 * Limit: the scratch a tensor list needs (tula_ags_workspace_size) is about 1.6 KB per tensor,
 * whatever the tensors' sizes and K: up to 10,670 tensors.  A longer list is rejected with
 * TULA_ERR_SCRATCH_LIMIT before anything is enqueued.
 *
 * Set-up: every call looks up the array's device address in the current device's context
 * (cudaGetSymbolAddress, a host-side lookup), so the address never goes stale, also after
 * cudaDeviceReset.  The first call on a device also loads the library's device code there: make
 * it, with that device current, before any stream capture.
 * Sharing: every call on a device uses the same array.  Each call clears the counters it needs
 * zeroed (two asynchronous memsets on `stream`, enqueued only once every argument has been
 * accepted) and otherwise overwrites what the previous call left, so calls that overlap on the
 * GPU (different streams, or different host threads) race and must not be issued.  Allocates
 * nothing: no cudaMalloc, no cudaFree, no allocating library call.
 * Errors: as tula_ags_step, plus TULA_ERR_SCRATCH_LIMIT.  A bounded wait that runs out inside a
 * kernel sets the array's error word, which no later call clears: read it (and clear it) with
 * tula_ags_static_scratch_error.  While it is set, the steps since it was last read are not
 * valid.
 */
#define TULA_STATIC_SCRATCH_BYTES (16u << 20)
int tula_ags_step_static_scratch(float *const *param_ptrs, float *const *grad_ptrs,
                                 float *const *mom_ptrs, const int64_t *numels, int n_tensors,
                                 float lr, float momentum, float weight_decay,
                                 const tula_ags_hparams *hp, void *stream);

/*
 * The error word of the static scratch on the current device, read after the work already
 * enqueued on `stream` (the call waits for that stream), then cleared: *error_out = 0 when every
 * bounded wait of the static-scratch steps since the last read completed, bit 0 set when one ran
 * out.  The counterpart of tula_ags_workspace_error for tula_ags_step_static_scratch (no
 * counterpart in the paper).  TULA_ERR_ARG when error_out is NULL; TULA_ERR_CUDA when a CUDA
 * call fails.
 */
int tula_ags_static_scratch_error(void *stream, int *error_out);

/*
 * Failure-detection check on the static scratch: as tula_ags_check_wait_timeout, with the error
 * word of the static array on the current device in place of a workspace's.  Asynchronous on
 * `stream`; about two seconds of GPU time.  No counterpart in the paper.
 */
int tula_ags_static_scratch_check_wait_timeout(void *stream);

/* Human-readable text for a TULA_* status code. */
const char *tula_ags_error_string(int code);

/* The cudaError_t of the last failed launch on this thread (0 if none). */
int tula_ags_last_cuda_error(void);

/* Number of kernels this process has launched through the library. */
uint64_t tula_ags_launch_count(void);

/*
 * Elements per tile (work item) of a pass that streams `streams` tensors through shared memory:
 * pass 1, the reduction (K replicas [+ g_small]; one tile of every stream fills a 36 KB stage),
 * pass 2, the update (gbar, w [+ m] [+ per-element scale]; a 24 KB stage), or pass 3, the
 * reduction when it also reads w (K replicas + w: LARS steps and tula_layer_stats; a 45 KB
 * stage).  A multiple of 128; TULA_ERR_ARG for another pass or when streams is outside
 * [1, TULA_MAX_K + 2] (passes 1 and 3) or [1, 4] (pass 2).
 */
int tula_ags_chunk_elems(int pass, int streams);

/*
 * Host-only view of the work decomposition: tensor p is split into
 * max(1, ceil(numels[p] / chunk_elems)) tiles; chunk_start_out[p] is the index of its first tile
 * and chunk_start_out[n_tensors] the total (n_tensors + 1 entries).
 */
int tula_ags_plan_chunks(const int64_t *numels, int n_tensors, int chunk_elems,
                         int64_t *chunk_start_out);

/*
 * Failure-detection check: launches, on `stream`, one warp that makes the library's bounded
 * mbarrier wait run out (it waits on an mbarrier that nothing arrives on; about two seconds) and
 * records it in the workspace's error word exactly as a streaming kernel records a stage that
 * never fills.  tula_ags_workspace_error() then reports bit 0; the CUDA context stays usable.
 * No counterpart in the paper.  TULA_ERR_WORKSPACE when workspace is NULL, misaligned or smaller
 * than the error word's offset + 4 bytes.
 */
int tula_ags_check_wait_timeout(void *workspace, size_t workspace_bytes, void *stream);

/*
 * Reads (synchronously, with cudaMemcpy) and clears the workspace's error word: 0 when every
 * wait of the kernels that used this workspace completed; bit 0 set when a bounded wait inside a
 * kernel ran out (the step's results are then not valid).  numels, n_tensors and K are those the
 * workspace was sized for.
 */
int tula_ags_workspace_error(const void *workspace, size_t workspace_bytes,
                             const int64_t *numels, int n_tensors, int K, int *error_out);

#ifdef __cplusplus
}
#endif

#endif /* TULA_AGS_H */
