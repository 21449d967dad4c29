// Internal declarations of libprefixplace (not installed, not part of the ABI).
#pragma once

#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>
#include <string>
#include <vector>

#include "prefixplace.h"

namespace pp {

// ---------------------------------------------------------------------------
// DP row metadata.  Rows are preorder positions, swept from n-1 down to 0.
// The skip branch of Eq. 9 reads row next(i):
//   kSkipCur   next(i) == i + 1: the row just computed (kept in registers)
//   kSkipZero  next(i) == n: the boundary row D[n][.] = 0
//   level >= 0 a row saved earlier on the skip-row stack at that level
// A row is pushed only when a position q < r - 1 reads it (next(q) == r),
// so the stack holds one row per pending subtree continuation and its depth
// is bounded by the tree depth.
// Packed in one int32: low 16 bits skip code + 2, high 16 bits push level + 1.
// ---------------------------------------------------------------------------
constexpr int kSkipZero = -2;
constexpr int kSkipCur = -1;
constexpr int kMaxStackLevels = 65533;

__host__ __device__ inline int meta_skip(int32_t m) { return (m & 0xFFFF) - 2; }
__host__ __device__ inline int meta_push(int32_t m) { return ((m >> 16) & 0xFFFF) - 1; }
inline int32_t meta_pack(int skip, int push)
{
    return (int32_t)(((uint32_t)(push + 1) << 16) | (uint32_t)(skip + 2));
}

// Row metadata of the wavefront DP kernel: the skip-row stack top is kept in
// registers (every stack read is of the top, and the zero row D[n][.] is the
// top of the empty stack), so a row needs only: its weight, whether its skip
// row is the row just computed (next(i) = i + 1) or the top, and whether it
// pushes (store the new row at `level`; it becomes the top) or pops (reload
// the new top from `level`, or reset it to the zero row when the stack empties).
// bits 0-2 weight-1 (weights <= 8), 3-4 kind, 5 reload, 6 push, 7 zero top,
// 16-31 level.
constexpr int kWaveCur = 0, kWaveTop = 2;
constexpr int kWaveReload = 1 << 5, kWavePush = 1 << 6, kWaveZeroTop = 1 << 7;
constexpr int kWaveStackOps = kWaveReload | kWavePush | kWaveZeroTop;
__host__ __device__ inline int32_t wave_pack(int w, int kind, int flags, int level)
{
    return (int32_t)((uint32_t)(w - 1) | ((uint32_t)kind << 3) | (uint32_t)flags | ((uint32_t)level << 16));
}

// Column geometry of one DP launch: thread t of the chain owns columns
// t*C + c + 1 (c = 0..C-1); column 0 is the boundary D[.][0] = 0.  Decision
// bits of row i are kpad/32 words; word (t/32)*C + c holds bit (t%32) for the
// column t*C + c + 1, i.e. one __ballot_sync per (warp, c).
struct DpGeom {
    int C = 1;        // columns per thread
    int T = 32;       // threads per chain (all CTAs)
    int kpad = 32;    // T * C columns
    int words = 1;    // decision words per row (kpad / 32)
    int P = 1;        // warps per chain
    int wave = 0;     // 1: wavefront kernel (cluster of CL CTAs x WPC warps)
    int CL = 1;       // CTAs per chain (thread-block cluster)
    int WPC = 1;      // warps per CTA
    int WMAX = 1;     // largest chunk weight the wavefront kernel is built for
    int L_smem = 0;   // skip-row stack levels held in shared memory
    size_t smem = 0;  // dynamic shared memory per CTA
    // Split launch (wavefront kernel, batch just above what clusters of CL
    // CTAs hold at one CTA per SM): the `split` items with the most kept rows
    // run as clusters of CL, the rest concurrently as clusters of CL2 = CL / 2
    // CTAs x WPC2 = 2 * WPC warps on the SMs left over (same P, C and bit
    // layout).  Both launches reserve more than half an SM's shared memory so
    // that no SM hosts two CTAs.  split = 0: one launch.
    int split = 0;
    size_t smem_x = 0;                       // the wide launch's shared memory when split
    int CL2 = 0, WPC2 = 0, L_smem2 = 0;
    size_t smem2 = 0;
};
// Decision bits of every DP kernel, packed by each thread over blocks of 32
// rows in sweep order (row r = n - 1 - i, block r / 32, bit r % 32): for chain
// warp g, lane and column offset c, the word
//   (((item * P + g) * nblk + r / 32) * C + c) * 32 + lane
// holds the take decisions of column (g * 32 + lane) * C + c + 1, with
// nblk = ceil(n / 32).

// Workspace of one batched DP launch (pp_dp_bits_size bytes, carved in this
// order): decision bits, then the pruned sweep (rows kept in sweep order, the
// inverse map position -> kept index or -1, prefix counts of positive
// profits, kept-row counts).  A row is dropped when every strict descendant
// of its parent has a non-positive profit: such a parent's interior is never
// taken and leaves D[parent+1] = D[next(parent)], so dropping those rows
// changes no value and no bit of a kept row (see k_prune).
// For the traceback, per kept row t (kept index, sweep order): skip[t] = kept
// index of next(row t), -1 when next(row t) = n; wsuf[t] = sum of the
// weights of kept rows t..nkept-1.
struct DpWork {
    uint32_t *bits = nullptr;      // [batch][P][nblk][C][32]
    int32_t *rowlist = nullptr;    // [batch][n]
    int32_t *kidx = nullptr;       // [batch][n]
    int32_t *cnt = nullptr;        // [batch][n + 1]
    int32_t *nkept = nullptr;      // [batch]
    int32_t *skip = nullptr;       // [batch][n]
    int32_t *wsuf = nullptr;       // [batch][n + 1]
    int64_t *rowp = nullptr;       // [batch][n] profit of each kept row, sweep order
    int32_t *rowm = nullptr;       // [batch][n] wave-kernel metadata of each kept row
};
size_t dp_work_bytes(int batch, int n, int words);
DpWork dp_work_split(void *base, int batch, int n, int words);
// the same workspace seen as a batch of one: item `item` of `w`
DpWork dp_work_item(const DpWork &w, int item, int n, int words);

// Status word values written by kernels (same numbering as pp_status).
constexpr int32_t kDevOk = PP_OK;

struct Scratch {
    void *ptr = nullptr;
    size_t bytes = 0;
};

}  // namespace pp

struct pp_instance {
    int32_t n = 0;
    int32_t W = 0;
    int32_t mode = 0;
    int device = 0;
    int sm_count = 0;
    int32_t stack_depth = 0;            // skip-row stack levels needed by the DP
    int64_t total_weight = 0;           // sum of chunk weights
    int32_t max_weight = 1;             // largest chunk weight
    int32_t trace_skips = 1;            // skips the traceback speculates per step beyond the first
    // DP launch-shape overrides of this instance (pp_tune_dp; 0 = automatic)
    int32_t tune_cl = 0, tune_c = 0, tune_flat = 0, tune_noprune = 0;
    std::vector<int32_t> h_order, h_next, h_budget, h_wpre, h_meta, h_wave;
    // device tables, preorder-indexed unless noted
    int32_t *d_order = nullptr;         // [n] position -> node id
    int32_t *d_next = nullptr;          // [n]
    int32_t *d_wpre = nullptr;          // [n] chunk weight
    int32_t *d_meta = nullptr;          // [n] packed skip / push codes
    int32_t *d_wave = nullptr;          // [n] wavefront-kernel row metadata
    int2 *d_pspan = nullptr;            // [n] parent x's strict-descendant range (x+1, next(x)); roots -1
    int32_t *d_budget = nullptr;        // [W]
    int64_t *d_a = nullptr;             // mode 0: [W][n] a_m(b)       (Eq. 2)
    int64_t *d_delta = nullptr;         // mode 0: [n]    Delta(b)     (Eq. 3)
    int64_t *d_own = nullptr;           // mode 0: [W][n] Lambda_m(b) [w_m(b) - f_m(b)]_+ (own first-copy gain)
    int64_t *d_pop = nullptr;           // mode 0: [W][n] Lambda_m(b)
    int64_t *d_rec = nullptr;           // [W][n] w_m(b) by node id
    int64_t *d_tr = nullptr;            // by node id: mode 0 [W][n] f_m(b), mode 1 [W][W][n] f_{m<-h}(b)
    int64_t *d_g = nullptr;             // mode 1: [W][W][n] Lambda_m(b) q_{m<-h}(b) at [h][m][i] (Eq. 5)
    int32_t *d_status = nullptr;        // device status word
    pp::Scratch stack;                  // skip-row stack spill of pp_tree_dp
    pp::Scratch plan;                   // pp_plan_run working set
    pp::Scratch plan_bits;              // pp_plan_run decision bits
    pp::Scratch sg;                     // safeguard candidates' working set
    pp::Scratch rp;                     // epoch update working set
    pp::Scratch top2;                   // top-2 holder tables of the planner
    // split DP launches: the two launches run on these streams (higher and
    // lower priority), forked from and joined back to the caller's stream
    cudaStream_t split_hi = nullptr, split_lo = nullptr;
    cudaEvent_t split_fork = nullptr, split_join_hi = nullptr, split_join_lo = nullptr;
    // pp_plan_run without lock step: one stream per start (up to kPlanStreams),
    // forked from and joined back to the caller's stream
    std::vector<cudaStream_t> plan_streams;
    std::vector<cudaEvent_t> plan_join;
    cudaEvent_t plan_fork = nullptr;
    std::vector<cudaEvent_t> phase_events;      // timing events of pp_plan_run, reused across calls
};

namespace pp {

// error reporting (thread-local message)
pp_status fail(pp_status s, const std::string &msg);
pp_status cuda_fail(cudaError_t e, const char *what);
#define PP_CUDA(call)                                                   \
    do {                                                                \
        cudaError_t e_ = (call);                                        \
        if (e_ != cudaSuccess) return ::pp::cuda_fail(e_, #call);       \
    } while (0)

pp_status ensure_scratch(Scratch &s, size_t bytes);
void free_scratch(Scratch &s);

// DP launch geometry for a given largest budget (after clamping to the
// instance's total weight).  Returns false when the budget is too large.
bool dp_geometry(const pp_instance *inst, int32_t max_budget, DpGeom *g, int batch = 1);

// Launchers used by both the ABI calls and the planner.
//   prof_by_node: profits indexed by node id (ABI) instead of preorder
//   item_budget:  [batch] budgets; item_active: [batch] or null (0 = skip item)
// stack_item: the launch's items use skip-row stack scratch from item slot
// stack_item on (launches of disjoint slots may run concurrently)
pp_status launch_tree_dp(pp_instance *inst, int batch, const int64_t *profit, bool prof_by_node,
                         const int32_t *item_budget, const int32_t *item_active,
                         const DpGeom &g, int64_t *best, const DpWork &work, cudaStream_t st,
                         int32_t max_budget, unsigned long long *rows_kept = nullptr, int stack_item = 0);
// scratch for the skip-row stack of `items` item slots of geometry g
pp_status ensure_dp_stack(pp_instance *inst, const DpGeom &g, int items);

pp_status launch_marginals(pp_instance *inst, int batch, const int32_t *worker,
                           const uint32_t *mask, bool by_node, const int32_t *item_active,
                           int64_t *profit, int64_t *oldsum, cudaStream_t st);

pp_status launch_objective(pp_instance *inst, int batch, const uint32_t *mask,
                           const uint8_t *chosen, int64_t *obj, cudaStream_t st);

// Top-2 holder tables of the source-dependent marginals, per start (batch item):
// v1, v2, l1 [batch][W][n] and the pre-update bit of the current worker [batch][n].
struct Top2 {
    int64_t *v1 = nullptr;
    int64_t *v2 = nullptr;
    int8_t *l1 = nullptr;
    uint8_t *oldbit = nullptr;
};
pp_status launch_marginals_top2(pp_instance *inst, int batch, const int32_t *prev_worker, const int32_t *worker,
                                const uint32_t *mask, const int32_t *item_active, const Top2 &t2,
                                int64_t *profit, int64_t *oldsum, cudaStream_t st);


// Traceback of pp_tree_dp's bits.  With mask == nullptr it writes chosen[]
// bytes by node id (ABI); otherwise it is the planner's accept-and-update
// step (see pp_plan.cu) and writes holder-mask bits in preorder.
struct AcceptArgs {
    const int32_t *worker = nullptr;    // [batch] h per item
    const int64_t *best = nullptr;      // [batch] D[0][k]
    const int64_t *oldsum = nullptr;    // [batch] sum of p_h over the current T_h
    int32_t *active = nullptr;          // [batch] start still refining
    int32_t *improved = nullptr;        // [batch] set on an accepted update
    int32_t *accepted = nullptr;        // [batch] accepted-update counter
    uint32_t *mask = nullptr;           // [batch][n] holder masks (preorder)
    int greedy = 0;                     // 1: always accept (WorkerGreedy pass)
    // optional [batch]: item b walks the decision bits (and pruned-sweep data)
    // of DP item bits_item[b] of the workspace instead of item b
    const int32_t *bits_item = nullptr;
};
pp_status launch_traceback(pp_instance *inst, int batch, const DpWork &work, const DpGeom &g,
                           const int32_t *item_budget, uint8_t *chosen, const AcceptArgs *acc,
                           cudaStream_t st);

// Safeguard candidates (requester-side): Independent, Popularity, LocalDedup
// holder masks [3][n] in preorder (device, in inst->sg, valid until the next
// call) and their objectives (host [3]).  Adds its kernel launches and DP
// cells to the counters.
pp_status plan_impl(pp_instance *inst, int32_t S, const int32_t *orders, int32_t R, uint8_t *placement,
                    int64_t *objective, pp_plan_stats *stats, cudaStream_t st, bool orders_only = false);

pp_status safeguards_impl(pp_instance *inst, cudaStream_t st, const uint32_t **masks, int64_t *obj,
                          int *launches, int64_t *cells, int *dp_launches);

}  // namespace pp
