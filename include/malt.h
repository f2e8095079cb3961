/*
 * malt.h -- C ABI of the GB300 MALT / MALTER optimizer step.
 *
 * One call updates every 2-D weight matrix of a model by the MALT update
 * (Algorithm 1 of "MALT: Lightweight Curvature-Aware Muon via Diagonal
 * Preconditioning") or the MALTER update (Algorithm 2).  Per matrix W (m x n)
 * with gradient G, momentum M, row statistics l (m) and column statistics
 * r (n), one step computes
 *
 *   M <- mu1 M + (1 - mu1) G                          (Alg. 1, M_t line)
 *   l <- mu2 l + (1 - mu2) [||G[i,:]||^2]_i           (Alg. 1, l_t line; eq. dp_preconditioner)
 *   r <- mu2 r + (1 - mu2) [||G[:,j]||^2]_j           (Alg. 1, r_t line)
 *   L = Diag((l + eps)^(-1/8)),  R = Diag((r + eps)^(-1/8))
 *   Mt = L M R,  O = NS_k(Mt),  D = L O R             (Alg. 1; Section 3.2 eq. final-update)
 *   W <- W - lr * s * ||O||_F / (||D||_F + eps) * D   (Alg. 1 W_t line: s = 1)
 *
 * and for MALTER additionally (Algorithm 2 and the alpha_t equation of
 * Section 3.5)
 *
 *   nu    <- mu2 nu + (1 - mu2) ||L G R||_F^2
 *   alpha  = sqrt(1 - mu2^t) / (1 - mu1^t + eps) * ||Mt||_F / (sqrt(nu) + eps),  s = alpha
 *
 * with t the 1-based step count.  NS_k is the quintic Newton-Schulz iteration
 * (the paper names it, Section 3.1, without its constants): on the wide
 * orientation of Mt (transposed when m > n), X = Mt / (||Mt||_F + ns_eps),
 * then k times A = X X^T, B = b A + c A A, X = a X + B X.
 *
 * Every call is asynchronous on the given CUDA stream (a cudaStream_t passed
 * as void*; NULL is the legacy default stream) and returns a status code
 * immediately; only malt_check, malt_get_scalars, malt_set_scalars,
 * malt_debug_scalars, malt_profile_read and malt_debug_wait_timeout wait for
 * the stream.  Only malt_init_state allocates device memory (the workspace,
 * with the persistent schedule's work table for every ns_steps value);
 * malt_debug_wait_timeout allocates one word for its probe, and the first
 * malt_step_host call on a state creates its two copy streams and their
 * events.  All device pointers passed in stay owned by the caller.
 *
 * Steps of one state share its workspace (operand buffers, partial sums,
 * scalars, counters).  Enqueue them on one stream, or order their streams
 * with events, so that no two steps of the same state run at once on the
 * GPU; a step switched to another stream with no such ordering races the
 * previous one.  A state is not thread-safe: calls on one state from several
 * host threads must be serialised by the caller.  Separate states share
 * nothing and may run concurrently.
 */
#ifndef MALT_H
#define MALT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ------------------------------------------------------ */
#define MALT_OK                   0
#define MALT_ERR_INVALID_ARG     -1  /* null pointer, n < 0, bad hyperparameter */
#define MALT_ERR_UNSUPPORTED     -2  /* rows or cols < 1, rows*cols >= 2^31 after
                                        rounding each up to a multiple of 8, bad dtype */
#define MALT_ERR_MISALIGNED      -3  /* a device pointer is not 16-byte aligned */
#define MALT_ERR_SHAPE_CHANGED   -4  /* step called with shapes/dtypes other than at init */
#define MALT_ERR_CUDA            -5  /* a CUDA runtime call failed (see malt_status_string) */
#define MALT_ERR_TIMEOUT         -6  /* a device-side wait ran out of its time budget
                                        (1 s plus 66 ns per column of the launch's
                                        longest Newton-Schulz reduction) */
#define MALT_ERR_OUT_OF_MEMORY   -7  /* workspace allocation failed at init */

/* ---- element types ----------------------------------------------------- */
#define MALT_F32   0
#define MALT_BF16  1

/* One 2-D parameter.  All pointers are DEVICE pointers owned by the caller,
 * 16-byte aligned, row-major and densely packed (leading dimension = cols).
 *   w       W, rows x cols, MALT_F32 or MALT_BF16, updated in place (bf16
 *           results are rounded to nearest even)
 *   g       G, rows x cols, MALT_F32 or MALT_BF16, read only
 *   m       momentum M, rows x cols fp32, updated in place
 *   l, r    row statistics (rows fp32) and column statistics (cols fp32),
 *           updated in place
 * rows and cols may be any positive sizes, with rows*cols < 2^31 after rounding
 * each up to a multiple of 8 (the kernels index a matrix's elements with
 * 32-bit offsets).  A matrix whose rows or cols are not multiples of 8 runs on
 * zero-padded copies in the library's workspace: each step copies its W, G,
 * M, l, r in and W, M, l, r back out (two extra passes over that matrix
 * only), with the same results.  W, G and M must not overlap each other or
 * another parameter's buffers. */
typedef struct {
    void*        w;
    int32_t      w_dtype;
    const void*  g;
    int32_t      g_dtype;
    float*       m;
    float*       l;
    float*       r;
    int64_t      rows;
    int64_t      cols;
} malt_param_t;

/* Hyperparameters (the Require line of Algorithms 1 and 2, plus the
 * Newton-Schulz settings).  Suggested defaults: mu1 0.95, mu2 0.99,
 * eps 1e-8 (the paper's appendix table), weight_decay 0, ns_steps 5,
 * (ns_a, ns_b, ns_c) = (3.4445, -4.7750, 2.0315), ns_eps 1e-7.
 * weight_decay, when non-zero, applies W <- (1 - lr*weight_decay) W before
 * the update (decoupled; the paper's table lists 0.1 but its algorithms
 * leave it out).  Constraints: 0 <= mu1, mu2 < 1; eps >= 0; 1 <= ns_steps <= 64. */
typedef struct {
    float   lr;
    float   mu1;
    float   mu2;
    float   eps;
    float   weight_decay;
    int32_t ns_steps;
    float   ns_a;
    float   ns_b;
    float   ns_c;
    float   ns_eps;
} malt_hparams_t;

/* Opaque per-model state: the library-owned workspace (Newton-Schulz operand
 * buffers grouped by shape, statistics partials, L and R, the per-matrix
 * MALTER scalar nu, the step counter t, the device status word). */
typedef struct malt_state malt_state_t;

/* Plan the step for these n parameters (their shapes and dtypes are fixed
 * from here on), allocate the workspace on the current CUDA device, and
 * zero M, l, r of every parameter on `stream` (Algorithm 1 INITIALIZE line;
 * nu_0 = 0 and t = 0 as in Algorithm 2).  W is left untouched.
 * n = 0 is allowed (every later step is a no-op).
 * On success *out receives a state the caller frees with malt_destroy_state;
 * on failure *out is NULL and nothing stays allocated. */
int malt_init_state(malt_state_t** out, const malt_param_t* params, int32_t n, void* stream);

/* One MALT step (Algorithm 1) of all n parameters, enqueued on `stream`.
 * params must describe the same shapes and dtypes, in the same order, as at
 * init (MALT_ERR_SHAPE_CHANGED otherwise); the pointers may differ. */
int malt_step(malt_state_t* st, const malt_param_t* params, int32_t n,
              const malt_hparams_t* hp, void* stream);

/* One MALTER step (Algorithm 2): as malt_step plus the nu / alpha scalars.
 * MALT and MALTER steps may be mixed on one state; nu only advances on
 * MALTER steps while t advances on both. */
int malter_step(malt_state_t* st, const malt_param_t* params, int32_t n,
                const malt_hparams_t* hp, void* stream);

/* One Muon step through the same engine, for comparison with MALT: the
 * update of Section 3.1 (eq. muon-update) with the momentum of Algorithm 1,
 *   M <- mu1 M + (1 - mu1) G,  O = NS_k(M),  W <- W - lr ||O||/(||O|| + eps) O,
 * i.e. MALT with L = R = I (the graft then only rescales by ||O||/(||O||+eps)).
 * The row / column statistics l, r are neither read nor updated (their
 * pointers must still be valid); t advances.  Same arguments and errors as
 * malt_step. */
int muon_step(malt_state_t* st, const malt_param_t* params, int32_t n,
              const malt_hparams_t* hp, void* stream);

/* One MALT (malter = 0) or MALTER (malter != 0) step whose gradients arrive
 * in HOST memory and whose updated weights are copied back to HOST memory.
 * g_host[i] holds rows*cols elements of params[i].g_dtype and is copied into
 * the device buffer params[i].g (which the library overwrites); after the
 * update, params[i].w is copied to w_host[i] (rows*cols elements of
 * params[i].w_dtype).  Host buffers should be page-locked (cudaHostAlloc /
 * pinned) for the copies to overlap.  The copies run on two library-owned
 * streams ordered by events against `stream`: the next call's gradient copy
 * waits only until the last step that read the same device G buffers (same
 * params[0].g) has consumed them (for a set other than the last two used, until
 * the latest step has consumed its gradients, which on one stream follows
 * every earlier step) -- so a caller that alternates two device
 * gradient sets gets the copy-in of step i+1 fully overlapped with step i,
 * and a caller with one set still overlaps it with step i's Newton-Schulz
 * work -- and this step's weight copy overlaps the next step, whose weight
 * update waits for it.  Returns immediately; w_host is valid
 * once malt_check (which waits for all three streams) returns.  The host
 * buffers must stay untouched until then.  Same validation and errors as
 * malt_step, plus MALT_ERR_INVALID_ARG for a null host pointer. */
int malt_step_host(malt_state_t* st, const malt_param_t* params, int32_t n,
                   const malt_hparams_t* hp, int32_t malter, const void* const* g_host,
                   void* const* w_host, void* stream);

/* Checkpoint support: copy the n per-matrix nu values and the step counter t
 * to host memory (get) or from host memory (set).  Both synchronise with the
 * stream of the state's last call.  M, l, r and W are caller-owned and are
 * saved by the caller. */
int malt_get_scalars(malt_state_t* st, float* nu_host, int32_t n, int64_t* t_host);
int malt_set_scalars(malt_state_t* st, const float* nu_host, int32_t n, int64_t t_host);

/* Wait for the stream of the state's last call (and the copy streams of
 * malt_step_host), then return (and clear) the
 * device-side status word: MALT_OK, or MALT_ERR_TIMEOUT when a kernel gave up
 * on a bounded wait, or MALT_ERR_CUDA when the stream reported an error. */
int malt_check(malt_state_t* st);

/* Test hooks.
 * malt_debug_direction: enqueue on `stream` a copy of the last step's
 *   orthogonalised direction O of parameter idx (rows x cols, bf16,
 *   row-major, same orientation as W) into the device buffer out.
 * malt_debug_precond: enqueue on `stream` copies of the last step's diagonal
 *   preconditioners of parameter idx, L = (l + eps)^(-1/8) (rows floats) and
 *   R = (r + eps)^(-1/8) (cols floats), as the step computed and used them
 *   (Algorithm 1, L_t / R_t line), into the device buffers L_out and R_out
 *   (fp32, caller-owned).  Muon steps leave L = R = 1.
 * malt_debug_scalars: synchronise, then write 8 floats per parameter to host
 *   memory: ||O||_F, ||D||_F, ||Mt||_F, ||L G R||_F^2 (MALTER steps, else 0),
 *   nu, alpha (1 on MALT steps), the applied scale lr*alpha*||O||/(||D||+eps),
 *   and 1/(||Mt||_F + ns_eps). */
int malt_debug_direction(malt_state_t* st, int32_t idx, void* out, void* stream);
int malt_debug_precond(malt_state_t* st, int32_t idx, float* L_out, float* R_out, void* stream);
/* malt_debug_timeout_site: where the first device-side wait gave up in the
 *   work that the last MALT_ERR_TIMEOUT from malt_check covered, 5 int32 to
 *   out5 (host memory): site code (1 claim a ring slot, 2 producer waits for
 *   the previous product, 3 free operand stage, 4 / 20 / 36 next item in the
 *   ring (odd producer / MMA / epilogue), 5 free accumulator, 6 stage
 *   operands, 7 finished accumulator, 8 epilogue waits for the Gram product,
 *   9 MMA drain; 0 when nothing timed out), work item, sequence number or
 *   reduction slice, block and thread index. */
int malt_debug_timeout_site(const malt_state_t* st, int32_t* out5);
int malt_debug_scalars(malt_state_t* st, float* out_host, int32_t n);
/* malt_debug_check_guards: every buffer of the state's workspace is followed
 *   by a 256-byte guard region filled with a fixed pattern at init.  Counts,
 *   after the state's last stream has finished, the guard bytes that no
 *   longer hold the pattern, into *bad_bytes (host): 0 unless a kernel wrote
 *   past one of its buffers.  Synchronises. */
int malt_debug_check_guards(malt_state_t* st, int64_t* bad_bytes);

/* Exercise the bounded device-side wait used by the kernels: launch one
 * block that waits on a flag nothing ever sets, for at most budget_ns
 * nanoseconds, then synchronise.  Returns MALT_ERR_TIMEOUT when the wait gave
 * up as designed (the expected result), MALT_OK if it somehow completed. */
int malt_debug_wait_timeout(int64_t budget_ns, void* stream);

/* Per-kernel timing.  While enabled, every kernel launch of a step is
 * bracketed by CUDA events recorded on the step's stream; malt_profile_read
 * synchronises, adds the elapsed device time (milliseconds) and the launch
 * count of each kernel kind into ms_out[kind] / launches_out[kind]
 * (nkinds entries, up to MALT_NUM_KINDS) and resets the accumulators.
 * Profiling only adds event records; it changes no result. */
#define MALT_KIND_BIND      0
#define MALT_KIND_STATS     1
#define MALT_KIND_FINALIZE  2
#define MALT_KIND_PRESCALE  3
#define MALT_KIND_NORMS     4
#define MALT_KIND_NS_GRAM   5
#define MALT_KIND_NS_POLY   6
#define MALT_KIND_NS_BX     7
#define MALT_KIND_SCALARS   8
#define MALT_KIND_APPLY     9
#define MALT_KIND_NS_PERSISTENT 10   /* all Newton-Schulz products, persistent schedule */
#define MALT_KIND_PAD      11   /* copies of matrices with rows or cols not a multiple of 8 */
#define MALT_NUM_KINDS     12
int malt_profile_enable(malt_state_t* st, int32_t enable);
int malt_profile_read(malt_state_t* st, double* ms_out, int64_t* launches_out, int32_t nkinds);

/* Schedule of a state's steps (the Orth step of Algorithm 1 is k iterations
 * of A = X X^T, B' = aI + bA + cA^2, X <- B' X per matrix).
 *   MALT_NS_PHASED: one launch per HBM-bound stage (statistics, finalize,
 *     prescale, norms, scalars, apply) and one per Newton-Schulz product (3 k
 *     launches per group of up to 8 shape classes), each product over all
 *     matrices finished before the next starts.
 *   MALT_NS_PERSISTENT: the same HBM-bound launches; one persistent launch
 *     per class group runs every product of every iteration.  Tiles are
 *     claimed dynamically in product order; a tile of matrix j waits on the
 *     device (bounded) only until the previous product of matrix j is stored,
 *     so one matrix's next product overlaps another matrix's current one and
 *     there is no launch gap or wave tail between products.
 *   MALT_NS_AUTO (default): per class group, persistent when a Gram product
 *     has fewer tiles than 16 waves of the resident CTA pairs, phased otherwise.
 * Both compute every tile with the same arithmetic: results are bitwise
 * identical.  Takes effect at the next step.  The persistent launches claim
 * from a work table that malt_init_state builds once for up to 64 iterations,
 * so no step uploads anything.  MALT_ERR_INVALID_ARG for a null state or an
 * unknown schedule. */
#define MALT_NS_PHASED     0
#define MALT_NS_PERSISTENT 1
#define MALT_NS_AUTO       2
int malt_set_ns_schedule(malt_state_t* st, int32_t schedule);

/* Host only (no GPU, no CUDA call): the work table of the persistent schedule
 * for these parameter shapes (only rows and cols are read) and ns_steps
 * iterations, in claim order, 8 int32 per item: launch group, stage (3 i +
 * kind for iteration i), kind (0 Gram, 1 Poly, 2 B*X), matrix index, local
 * index (the 256 x 256 tile of the NS frame; Gram and Poly list the upper
 * triangle only), the index of the counter the item waits for
 * ((stage - 1) * n + matrix, or -1), the count that counter must reach (16
 * signals per tile of the previous product), and the number of tiles of
 * (stage, matrix).  Writes min(capacity, total) items to out (capacity * 8
 * int32, caller-owned) and the total to *count; call with capacity 0 to size
 * out.  MALT_ERR_INVALID_ARG for bad arguments or ns_steps outside [1, 64],
 * MALT_ERR_UNSUPPORTED for a shape malt_init_state would reject. */
int malt_ns_schedule(const malt_param_t* params, int32_t n, int32_t ns_steps, int32_t* out,
                     int64_t capacity, int64_t* count);

/* Statistics stage of ONE matrix without any device allocation.
 * The paper has no counterpart: this exists for callers that cannot allocate
 * device memory when they need the work done -- code under a framework
 * allocator that owns all device memory, code in a latency-critical loop that
 * must not risk the device synchronisation an allocation may cause, services
 * that reserve all their memory at start-up.  It runs the momentum and
 * statistics updates and writes the two diagonal preconditioners with the
 * same kernels' arithmetic as a MALT step for that matrix (bitwise the same
 * m, l, r, and L, R as malt_debug_precond returns):
 *   m <- mu1 m + (1 - mu1) g;  l, r <- EMAs of the row / column sums of g^2;
 *   L_out = (l + eps)^(-1/8) (rows floats), R_out = (r + eps)^(-1/8) (cols floats).
 * All pointers are caller-owned device buffers laid out as in malt_param_t
 * (g rows x cols in g_dtype, m rows x cols fp32, l and L_out rows fp32, r and
 * R_out cols fp32), 16-byte aligned; rows and cols positive multiples of 8.
 * Its scratch (per-tile partial sums) lives in a fixed array inside the
 * library, MALT_NOALLOC_SCRATCH_FLOATS floats (4 MiB) on every GPU that loads
 * the library, held until the process exits.  A matrix that needs more --
 * ceil(cols/256)*rows rounded up to 64, plus ceil(rows/64)*cols floats -- is
 * rejected with MALT_ERR_UNSUPPORTED (and a message on stderr).
 * The first call on a device looks up the array's device address (with that
 * device current), so make that first call before any stream capture.  All
 * calls share the one array: calls that overlap on the GPU (other streams,
 * other threads) race and must be serialised by the caller.  Nothing in the
 * array needs to start at zero; every partial sum is written before it is
 * read.  Enqueued on `stream`; does not synchronise. */
#define MALT_NOALLOC_SCRATCH_FLOATS 1048576
int malt_stats_noalloc(const void* g, int32_t g_dtype, float* m, float* l, float* r,
                       float* L_out, float* R_out, int64_t rows, int64_t cols,
                       float mu1, float mu2, float eps, void* stream);

/* Whole-optimizer step, 2-D matrices: register bf16 copies of fp32 master
 * weights.  copies[i] is a caller-owned device buffer of rows x cols bf16
 * (16-byte aligned) that every later step's weight update fills with the
 * round-to-nearest-even of the updated fp32 W of parameter i (the weights a
 * bf16 model computes with), or NULL for none; copies = NULL clears all.
 * Only parameters with w_dtype MALT_F32 may have a copy
 * (MALT_ERR_UNSUPPORTED otherwise).  n must equal the state's parameter
 * count.  Takes effect at the next step. */
int malt_set_weight_copies(malt_state_t* st, void* const* copies, int32_t n);

/* ---- Whole-optimizer step: AdamW for the other parameters --------------
 * The paper updates only the 2-D weight matrices with MALT / MALTER and hands
 * the vectors, scalars, embeddings and output head to AdamW (Section 5.1,
 * parameter grouping; appendix table: betas (0.9, 0.95), weight decay 0.1).
 * Per tensor at step t (1-based, counted on the device):
 *   m <- beta1 m + (1 - beta1) g,  v <- beta2 v + (1 - beta2) g^2,
 *   w <- (1 - lr wd) w - lr (m / (1 - beta1^t)) / (sqrt(v / (1 - beta2^t)) + eps),
 * decoupled weight decay wd per tensor.  One grouped streaming launch (plus
 * a pointer-binding launch) covers every tensor.  A whole-optimizer step is
 * malt_step (or malter_step) on the matrices and malt_adamw_step on the rest,
 * enqueued on the same stream. */
typedef struct {
    float*       w;             /* fp32 master weights, numel, updated in place     */
    void*        w_copy;        /* bf16 copy of the updated w (numel), or NULL      */
    const void*  g;             /* gradient, numel, MALT_F32 or MALT_BF16, read only */
    int32_t      g_dtype;
    float*       m;             /* first moment, numel fp32, in place               */
    float*       v;             /* second moment, numel fp32, in place              */
    int64_t      numel;         /* elements (any positive count)                   */
    float        weight_decay;  /* decoupled decay of this tensor (0 for none)      */
} malt_adamw_param_t;
/* All pointers are caller-owned DEVICE pointers, 16-byte aligned, not
 * overlapping one another or another tensor's. */

typedef struct {
    float lr;      /* learning rate                                     */
    float beta1;   /* first-moment EMA, 0 <= beta1 < 1 (table: 0.9)      */
    float beta2;   /* second-moment EMA, 0 <= beta2 < 1 (table: 0.95)    */
    float eps;     /* added to sqrt(v_hat), >= 0 (1e-8 suggested)        */
} malt_adamw_hparams_t;

/* Opaque: the tensor table, block-prefix table and step counter t. */
typedef struct malt_adamw_state malt_adamw_state_t;

/* Plan the launches for these n tensors (sizes and gradient types fixed from
 * here on), allocate the small state on the current device and zero m and v
 * of every tensor on `stream` (m_0 = v_0 = 0, t = 0).  n = 0 is allowed.
 * Errors: MALT_ERR_INVALID_ARG (null pointer, n < 0, NaN decay),
 * MALT_ERR_UNSUPPORTED (numel <= 0, bad g_dtype), MALT_ERR_MISALIGNED,
 * MALT_ERR_OUT_OF_MEMORY; on failure *out is NULL. */
int malt_adamw_init_state(malt_adamw_state_t** out, const malt_adamw_param_t* params, int32_t n,
                          void* stream);

/* One AdamW step of all n tensors, enqueued on `stream` (no host
 * synchronisation).  The tensors must have the sizes and gradient types of
 * init, in the same order (MALT_ERR_SHAPE_CHANGED); pointers, w_copy and
 * weight_decay may change.  MALT_ERR_INVALID_ARG for hyperparameters out of
 * range. */
int malt_adamw_step(malt_adamw_state_t* st, const malt_adamw_param_t* params, int32_t n,
                    const malt_adamw_hparams_t* hp, void* stream);

/* Checkpoint support: read or set the step counter t (both synchronise with
 * the stream of the state's last call).  m, v and w are caller-owned. */
int malt_adamw_get_step(malt_adamw_state_t* st, int64_t* t_host);
int malt_adamw_set_step(malt_adamw_state_t* st, int64_t t_host);

/* Free the state (synchronises with its last stream first). */
void malt_adamw_destroy_state(malt_adamw_state_t* st);

/* Bytes of device workspace the state holds. */
size_t malt_workspace_bytes(const malt_state_t* st);

/* Static text for a status code. */
const char* malt_status_string(int code);

/* Free the workspace (synchronises with the state's last stream first). */
void malt_destroy_state(malt_state_t* st);

#ifdef __cplusplus
}
#endif

#endif /* MALT_H */
