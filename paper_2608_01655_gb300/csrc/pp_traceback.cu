// Traceback of the tree DP's decision bits (Algorithm 1's backtracking,
// Theorem 1: at most n visited states) and, in the planner, the accept-and-
// update step fused into it (Section IV-C, Prop. 1).  The bits are those
// pp_dp.cu's kernels write: for chain warp g, lane and column offset c, the
// word (((item * P + g) * nblk + r / 32) * C + c) * 32 + lane holds the take
// decisions of kept rows r (sweep order) at column (g * 32 + lane) * C + c + 1.
#include "pp_internal.cuh"

namespace pp {

constexpr unsigned kFull = 0xffffffffu;

// ===========================================================================
// Traceback from (0, k) (Algorithm 1, "backtrack"): at a visited row, take ->
// mark b_i, j -= w_i and go to the next kept row; skip -> go to next(i); stop
// at i = n or j = 0.  In kept-row order a take always moves from kept index t
// to t - 1 (the next kept row in preorder, since a pruned interior is all
// "skip"), and a skip moves to skip[t].  The walk is monotone in t and j, so
// one warp reads it tile by tile: a tile is 64 kept rows x 32 columns, whose
// decision bits are 64 words (one word holds 32 rows of one column), loaded
// together with the tile's skip targets, positions and suffix weights in one
// round of independent loads.  Inside the tile every step is register work:
// lane l tests row t - l at the column reached after taking rows t..t-l+1, a
// ballot gives the take-run, and the row that ends it is the skip.  A step
// that leaves the tile (rows below it, or columns left of it) loads the next.
// With unit chunk weights, helper warps of the walking warp's CTA follow its
// position through shared memory and prefetch into L1 the tiles below it in
// its column band (this tile's columns and the next ones to the left); the
// walk itself is unchanged (~4% shorter walks in the paper-scale plan; with
// chunk weights 1-2 the same prefetching made the source-dependent plan's
// walks ~15% longer, so weighted walks go without it).
// Planner mode (acc.mask != nullptr): the update is accepted in the greedy
// pass, or in refinement iff D[0][k] > sum of p_h over the current T_h
// (equivalent to G(T_-h, T'_h) > G(T) by Prop. 1); an accepted update
// replaces bit h of the holder masks by the traced set.
// ===========================================================================
constexpr int kTraceTileRows = 64;       // kept rows per traceback tile (a multiple of 32)
constexpr int kTraceHelpers = 3;         // prefetching warps beside the walking one
constexpr int kTraceAhead = 4;           // tiles below the walker's that they prefetch
constexpr uint32_t kTracePollLimit = 1u << 22;   // polls of the walker's position (~0.4 s)

__device__ __forceinline__ void prefetch_l1(const void *p)
{
    asm volatile("prefetch.global.L1 [%0];" ::"l"(__cvta_generic_to_global(p)));
}

// Helper warps (threads 32 .. 32 * (1 + kTraceHelpers) - 1): while the walker
// works, prefetch the decision-bit lines of the kept-row blocks from its tile
// down to kTraceAhead tiles below, for the 64 columns ending at its column,
// nearest first, and the same rows of the skip targets and positions.  walk[0], walk[1]: the walker's tile (first row, column); walk[2]:
// set when the walk is over.  Every address is inside the item's arrays.
__device__ void trace_prefetch(const uint32_t *Bi, int nblk, int C, int P, int nk, const int32_t *sk,
                               const int32_t *rl, volatile int *walk)
{
    const int ht = threadIdx.x - 32, NH = 32 * kTraceHelpers;
    int last_r0 = -2, last_j0 = -1;
    for (uint32_t it = 0; it < kTracePollLimit; ++it) {
        if (walk[2]) break;
        const int r0 = walk[0], j0 = walk[1];
        if ((r0 == last_r0 && j0 == last_j0) || r0 < 0 || j0 < 1 || nk <= 0) {
            __nanosleep(128);
            continue;
        }
        last_r0 = r0;
        last_j0 = j0;
        const int jl = j0 > 64 ? j0 - 63 : 1;
        const int lgC = __ffs(C) - 1;                             // C is a power of two
        const int tlo = (jl - 1) >> lgC, thi = (j0 - 1) >> lgC;   // chain threads owning those columns
        const int glo = tlo >> 5, ghi = min(thi >> 5, P - 1);
        const int ng = ghi - glo + 1;
        const int b_hi = min((r0 >> 5) + kTraceTileRows / 32 - 1, min(nblk, (nk + 31) >> 5) - 1);
        const int b_lo = max(0, (r0 >> 5) - kTraceAhead * (kTraceTileRows / 32));
        const int nb = b_hi - b_lo + 1;
        const int lines = nb > 0 ? nb * ng * C : 0;
        for (int x = ht; x < lines; x += NH) {
            const int c = x & (C - 1), gb = x >> lgC;
            // 64 columns span at most three chain warps: no run-time division
            const int bq = ng == 1 ? gb : ng == 2 ? gb >> 1 : gb / 3;
            const int gg = glo + (gb - bq * ng), b = b_hi - bq;
            const int ln = gg == glo ? (tlo & 31) : 0;
            prefetch_l1(Bi + (((size_t)gg * nblk + b) * C + c) * 32 + ln);
        }
        const int rlo = b_lo * 32, rhi = min(nk, (b_hi + 1) * 32);
        for (int r = rlo + 32 * ht; r < rhi; r += 32 * NH) {
            prefetch_l1(sk + r);
            prefetch_l1(rl + r);
        }
    }
}

// BYNODE: the ABI mode (chosen bytes by node id, acc.mask == nullptr);
// otherwise the planner's accept-and-update mode.  A template parameter, so
// the planner's walk carries no trace of the ABI mode's node-id loads.
template <int SKIPS, bool BYNODE>
__global__ void __launch_bounds__(256)
k_traceback(int32_t n, DpWork w, int C, int P, int kpad, int unit_weights,
            const int32_t *__restrict__ item_budget, const int32_t *__restrict__ order,
            uint8_t *__restrict__ chosen, AcceptArgs acc)
{
    const int item = blockIdx.x;
    uint32_t hbit = 0;
    uint32_t *M = nullptr;
    if (acc.mask) {
        if (!acc.active[item]) return;
        const bool ok = acc.greedy || acc.best[item] > acc.oldsum[item];
        if (!ok) return;
        const int32_t h = acc.worker[item];
        if (h < 0 || h >= 32) return;
        hbit = 1u << h;
        M = acc.mask + (size_t)item * n;
        // fire-and-forget reductions: no thread waits for the old mask words
        // (in the greedy pass T_h is still empty: nothing to clear)
        if (!acc.greedy)
            for (int32_t x = threadIdx.x; x < n; x += blockDim.x) atomicAnd(M + x, ~hbit);
    } else {
        uint8_t *ch = chosen + (size_t)item * n;
        for (int32_t x = threadIdx.x; x < n; x += blockDim.x) ch[x] = 0;
    }
    __shared__ int s_walk[3];                 // walker's tile row, tile column, done
    if (threadIdx.x == 0) {
        s_walk[0] = -1;
        s_walk[1] = 0;
        s_walk[2] = 0;
    }
    __syncthreads();
    volatile int *walk = s_walk;
    const int32_t kq = item_budget[item];
    const int bi = acc.bits_item ? acc.bits_item[item] : item;   // the DP item whose bits this walks
    const int nblk = (n + 31) / 32;
    const uint32_t *Bi = w.bits + (size_t)bi * P * (size_t)nblk * C * 32;
    const int32_t *rl = w.rowlist + (size_t)bi * n;
    const int32_t *sk = w.skip + (size_t)bi * n;
    const int32_t *ws = w.wsuf + (size_t)bi * (n + 1);
    const int nk = w.nkept[bi];
    if (threadIdx.x >= 32) {
        if (threadIdx.x < 32 * (1 + kTraceHelpers) && kq > 0 && unit_weights)
            trace_prefetch(Bi, nblk, C, P, nk, sk, rl, walk);
        return;
    }
    const int lane = threadIdx.x;
    if (acc.mask && !acc.greedy && lane == 0) {
        acc.improved[item] = 1;
        acc.accepted[item] += 1;
    }
    if (kq <= 0) return;
    int32_t j = kq < kpad ? kq : kpad;
    const int lgC = __ffs(C) - 1;
    auto word_at = [&](int blk, int col) -> uint32_t {       // bits of rows blk*32.. at column col >= 1
        const int q = col - 1;
        const int tt = q >> lgC, c = q & (C - 1);             // C is a power of two
        return Bi[(((size_t)(tt >> 5) * nblk + blk) * C + c) * 32 + (tt & 31)];
    };
    int t = nk - 1;                 // row of position 0 (the first root): swept last
    constexpr int TB = kTraceTileRows / 32;                   // 32-row blocks per tile
    for (int guard = 0; guard <= 2 * n + 2 && t >= 0 && j > 0; ++guard) {
        // ---- load the tile holding (t, j): rows r0..r0+TB*32-1, columns j0-31..j0
        const int r0 = t & ~(kTraceTileRows - 1), j0 = j;
        if (lane == 0) {                      // where the helpers prefetch next
            walk[1] = j0;
            walk[0] = r0;
        }
        const int colx = j0 - lane;
        uint32_t wv[TB];
        int skv[TB], rlv[TB], wsv[TB];
#pragma unroll
        for (int x = 0; x < TB; ++x) {
            const int r = r0 + 32 * x + lane;
            wv[x] = (colx >= 1 && r0 + 32 * x < nk) ? word_at((r0 >> 5) + x, colx) : 0u;
            skv[x] = r < nk ? sk[r] : -1;
            rlv[x] = r < nk ? rl[r] : 0;
            // ABI mode writes chosen[] by node id: fetch the rows' node ids with
            // the tile rather than one dependent load per step
            if (BYNODE && r < nk) rlv[x] = order[rlv[x]];
            wsv[x] = (!unit_weights && r < nk) ? ws[r] : 0;
        }
        const int wstop = unit_weights ? 0 : ws[min(r0 + kTraceTileRows, nk)];
        // a register of block lr / 32 of the lane lr % 32 (every lane calls it)
        auto pick = [&](const auto &v, int lr, int from) {
            int out = 0;
#pragma unroll
            for (int x = 0; x < TB; ++x) {
                const int y = __shfl_sync(kFull, (int)v[x], from);
                out = (lr >> 5) == x ? y : out;
            }
            return out;
        };
        // suffix weight of kept row r in r0..r0+TB*32
        auto wsat = [&](int r) -> int {
            const int lr = r - r0;
            const int y = pick(wsv, lr, lr & 31);
            return lr >= kTraceTileRows ? wstop : y;
        };
        // ---- walk inside the tile
        while (t >= r0 && j > 0 && j > j0 - 32) {
            const int row = t - lane;
            const int lr = (row - r0) & (kTraceTileRows - 1);
            int col, coln;
            if (unit_weights) {
                col = j - lane;
                coln = col - 1;
            } else {
                const int wt = wsat(t + 1), wr = wsat(row + 1), wr0 = wsat(row);
                col = j - (wr - wt);
                coln = j - (wr0 - wt);
            }
            const bool valid = row >= r0 && col >= 1 && col > j0 - 32;
            const uint32_t word = (uint32_t)pick(wv, lr, (j0 - col) & 31);
            const bool take = valid && ((word >> (lr & 31)) & 1u);
            const uint32_t tm = __ballot_sync(kFull, take);
            const int L = tm == kFull ? 32 : __ffs(~tm) - 1;    // rows t..t-L+1 are taken
            const int pos = pick(rlv, lr, lr & 31);
            const int skr = pick(skv, lr, lr & 31);
            // speculation for the lane that ends the take-run: its skip lands
            // on row skr at the same column; while that row is in the tile and
            // is skipped as well, the walk goes on to its skip target in the
            // same step, up to SKIPS times (skips often come in pairs: with one,
            // ~35% fewer steps at the paper-scale workload; trees with wide
            // fan-out have longer runs and use three)
            int tnext = skr;
            bool more = true;
#pragma unroll
            for (int d = 0; d < SKIPS; ++d) {
                const int lr1 = (tnext - r0) & (kTraceTileRows - 1);
                const uint32_t word1 = (uint32_t)pick(wv, lr1, (j0 - col) & 31);
                const int sk1 = pick(skv, lr1, lr1 & 31);
                more = more && tnext >= r0 && !((word1 >> (lr1 & 31)) & 1u);
                tnext = more ? sk1 : tnext;
            }
            if (lane < L) {
                if (BYNODE) chosen[(size_t)item * n + pos] = 1;   // pos: the row's node id here
                else atomicOr(M + pos, hbit);                 // a reduction: the walk does not wait on it
            }
            if (L == 32) {                                    // 32 takes: continue after the last
                j = __shfl_sync(kFull, coln, 31);
                t -= 32;
                continue;
            }
            const int vL = __shfl_sync(kFull, (int)valid, L);
            const int colL = __shfl_sync(kFull, col, L);
            const int skL = __shfl_sync(kFull, tnext, L);
            j = colL;
            if (vL) {
                t = skL;                // row t-L is skipped (and maybe next(t-L)): -1 = past n
            } else {
                t -= L;                                       // (t-L, colL) lies outside the tile
                break;
            }
        }
    }
    if (lane == 0) walk[2] = 1;               // the helpers stop
}


pp_status launch_traceback(pp_instance *inst, int batch, const DpWork &work, const DpGeom &g,
                           const int32_t *item_budget, uint8_t *chosen, const AcceptArgs *acc,
                           cudaStream_t st)
{
    if (batch <= 0 || inst->n == 0) return PP_OK;
    if (g.C < 1 || (g.C & (g.C - 1))) return fail(PP_EINVAL, "columns per thread must be a power of two");
    AcceptArgs a;
    if (acc) a = *acc;
    const int unit = inst->max_weight <= 1;
    const bool bynode = a.mask == nullptr;
    if (inst->trace_skips >= 3) {
        if (bynode) k_traceback<3, true><<<batch, 256, 0, st>>>(inst->n, work, g.C, g.P, g.kpad, unit, item_budget,
                                                                 inst->d_order, chosen, a);
        else k_traceback<3, false><<<batch, 256, 0, st>>>(inst->n, work, g.C, g.P, g.kpad, unit, item_budget,
                                                           inst->d_order, chosen, a);
    } else {
        if (bynode) k_traceback<1, true><<<batch, 256, 0, st>>>(inst->n, work, g.C, g.P, g.kpad, unit, item_budget,
                                                                 inst->d_order, chosen, a);
        else k_traceback<1, false><<<batch, 256, 0, st>>>(inst->n, work, g.C, g.P, g.kpad, unit, item_budget,
                                                           inst->d_order, chosen, a);
    }
    PP_CUDA(cudaGetLastError());
    return PP_OK;
}

}  // namespace pp

using namespace pp;

extern "C" pp_status pp_traceback(pp_instance *inst, int32_t batch, const uint32_t *bits,
                                  const int32_t *budget, int32_t max_budget, uint8_t *chosen,
                                  void *stream)
{
    if (!inst) return fail(PP_EINVAL, "null instance");
    if (batch < 0) return fail(PP_EINVAL, "batch must be >= 0");
    DpGeom g;
    if (!dp_geometry(inst, max_budget, &g, std::max(batch, 1))) return fail(PP_EINVAL, "max_budget out of range");
    if (batch == 0 || inst->n == 0) return PP_OK;
    if (!bits || !budget || !chosen) return fail(PP_EINVAL, "null device pointer");
    return launch_traceback(inst, batch, dp_work_split(const_cast<uint32_t *>(bits), batch, inst->n, g.words), g,
                            budget, chosen, nullptr, (cudaStream_t)stream);
}
