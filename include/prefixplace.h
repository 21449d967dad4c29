/*
 * prefixplace.h -- C ABI of libprefixplace.so, the GB300 (sm_103a) planner
 * hot path of PrefixPlace (arXiv 2608.01655).
 *
 * The library plans prefix-complete KV-cache targets for W workers over a
 * prefix tree of n chunks.  Its hot path is the per-worker exact update of
 * coordinate refinement: node marginals against the other workers' current
 * targets (Eq. 10 requester-side, Eq. 7 source-dependent), then the exact
 * capacity-k rooted-tree DP (Eq. 9, Theorem 1) and its traceback, batched over
 * workers and order-diverse starts (Algorithm 1).
 *
 * Conventions shared by every entry point
 *   - Node ids are the caller's (0..n-1).  The preorder used internally
 *     (roots, then children, each in ascending node id) is never exposed
 *     except through pp_instance_preorder().
 *   - Integers only: costs are int64 microseconds, demand int64 counts.  The
 *     paper's floating-point tolerance epsilon is therefore 0: a refinement
 *     update is accepted only on a strict improvement.
 *   - Every function returns a pp_status and never aborts; pp_last_error()
 *     gives a thread-local message for the last failure in the calling
 *     thread.  Kernels report device-side problems (a budget above the
 *     declared bound, a wait that ran out) through a status word of the
 *     instance; pp_instance_sync() and pp_plan_run() read and clear it.
 *   - "device" pointers are CUDA global-memory pointers of the instance's
 *     device (for example torch tensors' data_ptr()); "host" pointers are
 *     ordinary CPU memory.  The caller owns every buffer it passes; the
 *     library owns the instance and its internal scratch.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  Calls that
 *     take device buffers are asynchronous and stream-ordered.
 *   - Limits: 1 <= W <= 32 workers (holder sets are 32-bit masks), the
 *     largest useful budget min(k, total chunk weight) <= 32768 slots, and a
 *     skip-row stack depth (bounded by the tree depth) <= 65533.
 */
#ifndef PREFIXPLACE_H
#define PREFIXPLACE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct pp_instance pp_instance;   /* opaque, library-owned */

typedef enum {
    PP_OK = 0,
    PP_EINVAL = 1,      /* bad argument: size, mode, null pointer, weight < 1, negative data */
    PP_ENOTTREE = 2,    /* parent[] out of range, self-parent, or a cycle */
    PP_EOVERFLOW = 3,   /* sum of demand * recompute, of demand or of recompute exceeds 2^62 */
    PP_ENOMEM = 4,      /* device or host allocation failed */
    PP_ECUDA = 5,       /* a CUDA runtime call failed */
    PP_ETIMEOUT = 6,    /* a bounded device-side wait ran out (device status word) */
    PP_EBOUNDS = 7      /* a device-side bounds check failed (device status word) */
} pp_status;

enum { PP_TRANSFER_REQUESTER = 0, PP_TRANSFER_SOURCE = 1 };

/* Optional inputs and outputs of pp_plan_run / pp_replan.  Zero-initialise it:
 * every "in" field's zero is the default.  Array members may be NULL. */
typedef struct {
    int64_t *per_start_objective;  /* [n_starts] host, out: objective of each candidate */
    int32_t *per_start_sweeps;     /* [n_starts] host, out: refinement sweeps run */
    int32_t *per_start_accepted;   /* [n_starts] host, out: accepted refinement updates */
    int32_t *orders_used;          /* [n_starts][W] host, out: the start orders */
    int32_t best_start;            /* out: index of the returned candidate (>= n_starts:
                                      safeguard best_start - n_starts) */
    int32_t dp_count;              /* out: tree DPs executed (inactive starts excluded; with
                                      default orders and n_starts > 1 every start's first
                                      greedy update walks the standalone-score DP of its
                                      worker, which is the same DP, so it is not run again) */
    int64_t dp_cells;              /* out: sum over executed DPs of n * k_h (Eq. 9 cells) */
    int32_t kernel_launches;       /* out: kernels launched by this call */
    int64_t dp_rows_swept;         /* out: rows the DPs actually swept (pruned sweep), summed */
    int32_t time_phases;           /* in: nonzero = time the phases below with CUDA events */
    float phase_ms[3];             /* out (if time_phases): device time of the marginal,
                                      tree-DP (with its row pruning) and traceback launches,
                                      summed over the plan's steps (per-start streams: the
                                      mean over starts of each start's sum) */
    int32_t dp_launches;           /* out: tree-DP steps (lock step: batched launches; per-start
                                      streams: the mean over starts of executed updates),
                                      the standalone-score launch included */
    int32_t no_safeguards;         /* in: nonzero = leave out the safeguard candidates */
    int64_t safeguard_objective[3];/* out: Independent, Popularity, LocalDedup objectives
                                      (requester-side only; else 0) */
    int32_t marginals;             /* in, source-dependent only: 0 automatic, 1 scan each
                                      chunk's holders, 2 keep top-2 holder tables per start
                                      (Section IV-C); results are identical */
    int32_t used_top2;             /* out: 1 if the top-2 tables were used */
    int32_t schedule;              /* in: 0 automatic, 1 lock step (all starts advance together,
                                      one batched launch per step), 2 per-start streams (each
                                      start on its own stream, never waiting for a slower
                                      one).  Automatic takes per-start streams when S > 1 and
                                      CUDA_DEVICE_MAX_CONNECTIONS (read at the call; it acts
                                      when the CUDA context is created) gives every stream its
                                      own hardware queue, min(S, 32), else lock step.
                                      out: the schedule used (1 or 2).  Results are identical */
    int32_t hw_queues;             /* out: the hardware queue count the automatic schedule assumed
                                      (CUDA_DEVICE_MAX_CONNECTIONS as read at the call, 8 when
                                      unset).  The driver reads that variable only when the CUDA
                                      context is created, so a context created before it was set
                                      may have fewer queues: the per-start schedule then runs
                                      slower, with the same results */
} pp_plan_stats;

/*
 * pp_instance_create -- validate a planner instance, upload it and build the
 * per-instance tables (preorder, next(i), the DP's row metadata, and the
 * gains of Eq. 2-3 or Eq. 5).
 *
 *   n, W          chunks (n >= 0) and workers (1..32)
 *   parent        host [n]: parent node id, or -1 for a child of the implicit
 *                 no-cost dummy root (Section III-A)
 *   weight        host [n]: budget slots per chunk, >= 1 (1 = the paper's
 *                 equal-sized chunks)
 *   demand        host [W][n]: Lambda_m(b) >= 0, already counted on every
 *                 chunk of each request's prefix path (Section III-A)
 *   recompute     host [W][n]: w_m(b) >= 0 in microseconds
 *   transfer      host, >= 0 microseconds: mode PP_TRANSFER_REQUESTER
 *                 [W][n] f_m(b) (Eq. 1); mode PP_TRANSFER_SOURCE [W][W][n],
 *                 element [h][m][b] = f_{m<-h}(b) (Section III-C); the
 *                 diagonal h == m is never read
 *   budget        host [W]: k_m >= 0 slots
 *   stream        stream for the uploads and precompute kernels
 *   out           receives the instance (NULL on failure)
 * Errors: PP_EINVAL, PP_ENOTTREE, PP_EOVERFLOW (one of three exact sums
 * over all (m, b) above 2^62: Lambda * w, which bounds every objective,
 * marginal and DP value of the planner; Lambda, which bounds the Popularity
 * safeguard's DP values; w, which bounds the epoch update's one-time cost),
 * PP_ENOMEM, PP_ECUDA.
 * The call synchronises `stream` before returning; the inputs are not retained.
 */
pp_status pp_instance_create(int32_t n, int32_t W, const int32_t *parent, const int32_t *weight,
                             const int64_t *demand, const int64_t *recompute,
                             const int64_t *transfer, int32_t transfer_mode,
                             const int32_t *budget, void *stream, pp_instance **out);

/* Frees the instance and its device memory.  NULL is accepted. */
pp_status pp_instance_destroy(pp_instance *inst);

/*
 * pp_instance_preorder -- the internal preorder (Section IV-A, "number nodes
 * in preorder and compute next(i)"): order[i] = node at 0-based position i,
 * next[i] = first position after that node's subtree.  Host [n] outputs.
 * Also reports the depth of the DP's skip-row stack (may be NULL).
 */
pp_status pp_instance_preorder(const pp_instance *inst, int32_t *order, int32_t *next,
                               int32_t *stack_depth);

/*
 * pp_row_plan -- host-only (no CUDA call): the preorder and the DP's row plan
 * for a parent array, as pp_instance_create builds them.  Positions are swept
 * from n-1 down to 0; the skip branch of Eq. 9 at position i reads row
 * next(i), which is the row just computed when next(i) == i + 1 (skip_code
 * -1), the zero boundary row when next(i) == n (skip_code -2), and otherwise
 * a row saved on the skip-row stack at level skip_code >= 0.  push_level[i]
 * >= 0 saves row i at that level; -1 saves nothing.
 *   order, next, skip_code, push_level   host [n] out
 *   stack_depth                          host out: levels used
 * Errors: PP_EINVAL, PP_ENOTTREE.
 */
pp_status pp_row_plan(int32_t n, const int32_t *parent, int32_t *order, int32_t *next,
                      int32_t *skip_code, int32_t *push_level, int32_t *stack_depth);

/*
 * pp_row_plan_registers -- host-only: the per-row codes of the register-
 * resident variant of the same row plan (the wavefront DP kernel keeps the
 * top of the skip-row stack in registers; the zero row is the top of the
 * empty stack).  code[i], i a preorder position (host [n] out):
 *   bits 0-2   w_i - 1 (weights above 8 read as 8)
 *   bits 3-4   0: the skip row is row i+1 (next(i) = i + 1); 2: the stack top
 *   bit 5      after row i, reload the top from level `level`
 *   bit 6      after row i, save row i at level `level`; it becomes the top
 *   bit 7      after row i, the stack is empty: the top is the zero row
 *   bits 16-31 level
 * Errors: PP_EINVAL, PP_ENOTTREE.
 */
pp_status pp_row_plan_registers(int32_t n, const int32_t *parent, const int32_t *weight,
                                int32_t *code);

/*
 * pp_instance_sync -- synchronise `stream`, then read and clear the device
 * status word.  Returns PP_OK, PP_ETIMEOUT, PP_EBOUNDS or PP_ECUDA.
 */
pp_status pp_instance_sync(pp_instance *inst, void *stream);

/*
 * pp_marginals -- exact node marginals of one worker per batch item against
 * the other workers' targets (Prop. 1).
 *   requester-side: p_h(b) = a_h(b) + 1{no worker l != h holds b} Delta(b)   (Eq. 10)
 *   source-dependent: p_h(b) = sum_m Lambda_m(b) [q_{m<-h}(b) - v_m^{(-h)}(b)]_+ (Eq. 7)
 *     with v_m^{(-h)}(b) the best q_{m<-l}(b) over holders l != h (0 if none).
 *   batch         items (>= 0)
 *   worker        device [batch]: h per item, 0..W-1
 *   holder_mask   device [batch][n] by node id: bit l set = worker l holds the
 *                 chunk; bit h itself is ignored
 *   profit        device [batch][n] by node id, out
 * Errors: PP_EINVAL (host-side argument checks).  A worker id out of range
 * sets PP_EBOUNDS in the status word and leaves that item's profits at 0.
 */
pp_status pp_marginals(pp_instance *inst, int32_t batch, const int32_t *worker,
                       const uint32_t *holder_mask, int64_t *profit, void *stream);

/*
 * pp_dp_bits_size -- bytes of the workspace that pp_tree_dp writes and
 * pp_traceback reads for `batch` items whose budgets are at most
 * `max_budget`: the decision bits plus the rows of the pruned sweep (rows
 * strictly below a chunk whose strict descendants all have profit <= 0 never
 * change a kept row's value or decision, so the DP skips them).  Returns 0 for
 * batch <= 0 or an invalid max_budget.
 */
size_t pp_dp_bits_size(const pp_instance *inst, int32_t batch, int32_t max_budget);

/*
 * pp_tree_dp -- the exact capacity-k prefix-complete tree knapsack (Eq. 9,
 * Theorem 1) for each batch item:
 *   D[i][0] = 0, D[n][j] = 0,
 *   D[i][j] = max{ D[next(i)][j], p(b_i) + D[i+1][j - w_i] }  (take needs j >= w_i)
 * over preorder positions i, recording "take" only on a strict improvement.
 *   profit        device [batch][n] by node id; any int64 values whose
 *                 absolute sum stays below 2^62 (not checked)
 *   budget        device [batch]: k per item, 0 <= k <= max_budget
 *   max_budget    host: upper bound of budget[]; fixes the bit layout
 *   best          device [batch], out: D[0][k]
 *   bits          device workspace of pp_dp_bits_size(inst, batch, max_budget)
 *                 bytes, out: decision bits for pp_traceback
 * A budget outside [0, max_budget] sets PP_EBOUNDS and that item's best to 0.
 * The call may allocate instance-owned device scratch for the skip-row stack
 * on first use (or when a larger batch needs more).  A batch that pp_dp_split
 * splits runs as two launches on two streams of the instance (created on the
 * first such call, with three events), forked from and joined back to
 * `stream`, so the work stays ordered on `stream`; calls on one instance use
 * its scratch and must not overlap on the GPU.
 */
pp_status pp_tree_dp(pp_instance *inst, int32_t batch, const int64_t *profit,
                     const int32_t *budget, int32_t max_budget, int64_t *best,
                     uint32_t *bits, void *stream);

/*
 * pp_tree_dp_noalloc -- pp_tree_dp for callers that must not allocate device
 * memory while they plan.  The paper has no counterpart: it is a library
 * convenience.  pp_tree_dp may call cudaMalloc on first use, for skip-row
 * stack levels that do not fit in shared memory.  Some callers cannot allow
 * that: cudaMalloc can wait until the whole device is idle, which a serving
 * loop with a latency budget cannot afford, and a process whose device memory
 * is already handed out by its own caching allocator may not get a raw
 * allocation at all.  This variant keeps those levels in a fixed 16 MiB array
 * of the library's device memory (every GPU that loads the library holds it
 * until the process exits) and calls no allocating routine.
 * Arguments, results and bit layout are exactly those of pp_tree_dp, and
 * pp_traceback reads the bits as usual.
 * Limit: batch * (stack levels beyond shared memory) * padded columns * 8
 * bytes must be at most 16 MiB (pp_dp_geometry gives the levels held in
 * shared memory and the padded columns, pp_instance_preorder the stack
 * depth); a larger launch is rejected with PP_EINVAL and nothing runs.
 * The instance's device must be the current device.  The first call on a
 * device looks up the array's device address (a one-time set-up); make that
 * first call before any stream capture.  All calls on a device share the
 * array and leave their contents in it.  Nothing in it needs to start at
 * zero, since a call writes every stack level before reading it.  But calls
 * that overlap on the GPU (other streams, other host threads) race on it and
 * give wrong results: keep them ordered.
 */
pp_status pp_tree_dp_noalloc(pp_instance *inst, int32_t batch, const int64_t *profit,
                             const int32_t *budget, int32_t max_budget, int64_t *best,
                             uint32_t *bits, void *stream);

/*
 * pp_dp_rows_swept -- for the last pp_tree_dp / pp_tree_dp_noalloc on
 * `workspace` (same batch and max_budget), the number of rows each item's DP
 * actually swept after pruning (host [batch] out).  Synchronises `stream`.
 * Errors: PP_EINVAL, PP_ECUDA.
 */
pp_status pp_dp_rows_swept(const pp_instance *inst, int32_t batch, int32_t max_budget,
                           const uint32_t *workspace, int32_t *rows, void *stream);

/*
 * pp_traceback -- recover each item's optimal parent-closed set from the
 * decision bits (Algorithm 1's backtracking, from the cell of the first row
 * and the full budget): start at position 0
 * with j = k; "take" marks the chunk, j -= w_i and moves to i+1; "skip" moves
 * to next(i).  Among optimal sets this returns the lexicographically smallest
 * preorder indicator.
 *   bits, budget, max_budget   exactly as given to pp_tree_dp
 *   chosen        device [batch][n] by node id, out: 1 = selected, else 0
 */
pp_status pp_traceback(pp_instance *inst, int32_t batch, const uint32_t *bits,
                       const int32_t *budget, int32_t max_budget, uint8_t *chosen,
                       void *stream);

/*
 * pp_objective -- the planner objective of each batch item's placement:
 * F (Lemma 1, Eq. 4) for requester-side instances, F_pair (Eq. 6) for
 * source-dependent ones.  Placements need not be feasible.
 *   chosen        device [batch][W][n] by node id: nonzero = worker holds chunk
 *   obj           device [batch], out
 */
pp_status pp_objective(pp_instance *inst, int32_t batch, const uint8_t *chosen, int64_t *obj,
                       void *stream);

/*
 * pp_plan_run -- Algorithm 1 (procedure PrefixPlace): for each start order,
 * one WorkerGreedy pass (Theorem 3), then at most max_rounds refinement
 * sweeps; a sweep with no accepted update ends that start.  Starts run
 * batched in lock step, or each on its own stream (stats->schedule).  With the requester-side objective the Independent, Popularity
 * and LocalDedup placements (pp_safeguards) join the candidates as indices
 * S, S+1, S+2 unless stats->no_safeguards is set.
 *   n_starts      S >= 1
 *   orders        host [S][W] permutations of 0..W-1, or NULL for the default:
 *                 S == 1 the identity; otherwise start 0 = standalone-score
 *                 order (descending, ties to the lower id), start 1 its
 *                 reverse, start s >= 2 a Fisher-Yates shuffle driven by
 *                 SplitMix64 seeded with s (j = next() mod (i + 1), i = W-1..1)
 *   max_rounds    R >= 0 refinement sweeps
 *   placement     host [W][n] out: the best candidate (highest objective,
 *                 ties to the lowest candidate index), 1 = resident
 *   objective     host out: its objective (Eq. 4 or Eq. 6)
 *   stats         optional (NULL) extra outputs
 * Synchronous: returns after the result is on the host.  Errors: PP_EINVAL,
 * PP_ENOMEM, PP_ECUDA, and any device status (PP_ETIMEOUT, PP_EBOUNDS).
 */
pp_status pp_plan_run(pp_instance *inst, int32_t n_starts, const int32_t *orders,
                      int32_t max_rounds, uint8_t *placement, int64_t *objective,
                      pp_plan_stats *stats, void *stream);

/*
 * pp_test_inject -- testing hook for the failure path of the DP kernel's
 * bounded waits; it makes no GPU fault.  kind 1: from the next launch on, the
 * chain warp with index `value` (-1 = none, the default) stops publishing
 * its ring counter, so the warp to its right waits until its time limit
 * (0.5 s) runs out, every warp of the launch leaves its loop, and
 * pp_instance_sync() reports PP_ETIMEOUT with the context still usable.
 * Applies to the current device.  Errors: PP_EINVAL, PP_ECUDA.
 */
pp_status pp_test_inject(int32_t kind, int32_t value);

/*
 * pp_dp_geometry -- the launch shape pp_tree_dp uses for `batch` items with
 * budgets up to `max_budget` (host out[8]): wavefront kernel (1) or one-CTA
 * kernel (0), CTAs per cluster, warps per CTA, columns per thread, warps per
 * DP, skip-row stack levels in shared memory, shared memory bytes per CTA,
 * padded column count.  Errors: PP_EINVAL.
 */
pp_status pp_dp_geometry(const pp_instance *inst, int32_t batch, int32_t max_budget, int32_t *out);

/*
 * pp_dp_split -- whether pp_tree_dp runs `batch` items with budgets up to
 * `max_budget` as two concurrent launches (host out[5]): items of the wide
 * launch (0 = one launch; its shape is that of pp_dp_geometry), CTAs per
 * cluster and warps per CTA of the narrow launch that takes the other items
 * (the ones with the fewest kept rows), its skip-row stack levels in shared
 * memory, and the wide launch's shared memory bytes per CTA.  A split is
 * used when the batch exceeds, by at most 2, the number of the wide clusters
 * that the device holds at one CTA per SM (15 clusters of 8 CTAs on a
 * 152-SM GB300); results and decision bits do not depend on it.
 * Errors: PP_EINVAL.
 */
pp_status pp_dp_split(const pp_instance *inst, int32_t batch, int32_t max_budget, int32_t *out);

/*
 * pp_dp_stack_bytes -- bytes of skip-row stack scratch the instance holds
 * (no counterpart in the paper; host out).  pp_tree_dp and pp_plan_run
 * allocate it on the first launch whose skip-row stack does not fit in shared
 * memory and keep it until pp_instance_destroy; pp_tree_dp_noalloc never adds
 * to it.  0 before any such launch.  Errors: PP_EINVAL.
 */
pp_status pp_dp_stack_bytes(const pp_instance *inst, size_t *out);

/*
 * pp_tune_dp -- override of this instance's DP launch shape, for tuning
 * sweeps (no counterpart in the paper): CTAs per cluster (1..8, 0 =
 * automatic), columns per thread (power of two up to 16, 0 = automatic),
 * force_flat != 0 selects the one-CTA kernel, no_prune != 0 sweeps every row
 * instead of the pruned sweep (results are the same either way).  Later
 * pp_dp_bits_size / pp_tree_dp / pp_traceback / pp_plan_run calls on this
 * instance use it, so set it before sizing workspaces; other instances are
 * not affected.  Not thread-safe against concurrent calls on the same
 * instance.  Errors: PP_EINVAL.
 */
pp_status pp_tune_dp(pp_instance *inst, int32_t cluster_ctas, int32_t columns_per_thread, int32_t force_flat,
                     int32_t no_prune);

/*
 * pp_default_orders -- the start orders pp_plan_run uses when it is given
 * orders = NULL (Section IV-C: standalone-score order, its reverse, then
 * SplitMix64 shuffles; the identity for one start), written to host
 * [n_starts][W].  Runs the standalone-score DPs on the device when
 * n_starts > 1.  Lets several processes split the starts of one plan: each
 * computes the same orders and runs its share with pp_plan_run.
 * Synchronous.  Errors: PP_EINVAL, PP_ENOMEM, PP_ECUDA.
 */
pp_status pp_default_orders(pp_instance *inst, int32_t n_starts, int32_t *orders, void *stream);

/*
 * pp_safeguards -- the safeguard candidates that Algorithm 1 adds for the
 * requester-side objective (Section IV-C; the comparators of Section V-A):
 * every worker's target is the exact DP of Eq. 9 on
 *   [0] Independent  Lambda_m(b) w_m(b)   (the worker alone)
 *   [1] Popularity   Lambda_m(b)          (local demand alone)
 *   [2] LocalDedup   workers in index order; a_m(b) (Eq. 2) for a chunk an
 *                    earlier worker holds, else Lambda_m(b) w_m(b)
 *   placement   host [3][W][n] out, by node id
 *   objective   host [3] out, Eq. 4
 * Synchronous on `stream`.  Errors: PP_EINVAL (source-dependent instance,
 * null argument, another current device), PP_ENOMEM, PP_ECUDA.
 */
pp_status pp_safeguards(pp_instance *inst, uint8_t *placement, int64_t *objective, void *stream);

/* Outputs of pp_replan. */
typedef struct {
    int64_t incumbent_objective;   /* G(T_old) under the instance's (refreshed) demand */
    int64_t new_objective;         /* G(T_new) of the reoptimised target */
    int64_t materialization_cost;  /* one-time cost of the chunks T_new adds, microseconds */
    int64_t break_even_requests;   /* ceil(cost * epoch_requests / (G_new - G_old)), INT64_MAX when
                                      that does not fit in int64; -1 without a gain */
    int32_t adopted;               /* 1: T_new returned; 0: the incumbent kept */
} pp_replan_result;

/*
 * pp_replan -- epoch update with the amortisation rule (Section IV-D; the
 * break-even requests of RQ5).  `inst` holds the refreshed demand.  The
 * incumbent is scored under it, a reoptimised target is planned exactly as
 * pp_plan_run does (n_starts, orders, max_rounds, stats as there), and the
 * target's one-time cost is, for every chunk a worker holds in the target but
 * not in the incumbent, the cheaper of recomputing it and fetching it from a
 * worker that holds it in the incumbent (recomputing when none does) -- the
 * Section III-A materialisation rule applied to the incumbent.  G is a saving
 * per epoch of `epoch_requests` requests, so the target is adopted iff
 *   (G_new - G_old) * horizon_requests > cost * epoch_requests.
 *   incumbent     host [W][n] by node id, nonzero = resident
 *   placement     host [W][n] out: the target if adopted, else the incumbent
 *   result        host out
 * Synchronous.  Errors: PP_EINVAL (epoch_requests <= 0, horizon_requests < 0,
 * null pointers, and those of pp_plan_run), PP_ENOMEM, PP_ECUDA, device status.
 */
pp_status pp_replan(pp_instance *inst, const uint8_t *incumbent, int32_t n_starts, const int32_t *orders,
                    int32_t max_rounds, int64_t epoch_requests, int64_t horizon_requests,
                    uint8_t *placement, pp_replan_result *result, pp_plan_stats *stats, void *stream);

/* Thread-local description of the last failure in this thread ("" if none). */
const char *pp_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* PREFIXPLACE_H */
