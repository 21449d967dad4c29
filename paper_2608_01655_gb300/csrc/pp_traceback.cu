// Traceback of the tree DP's decision bits (Algorithm 1's backtracking,
// Theorem 1: at most n visited states) and, in the planner, the accept-and-
// update step fused into it (Section IV-C, Prop. 1).  The bits are those
// pp_dp.cu's kernels write, in block pairs: for chain warp g, lane and column
// offset c, the 8-byte word ((item * P + g) * nblk / 2 + r / 64) * C + c) * 32
// + lane holds the take decisions of kept rows r (sweep order, 64 rows, bit
// r % 64) at column (g * 32 + lane) * C + c + 1.
#include "pp_internal.cuh"

namespace pp {

constexpr unsigned kFull = 0xffffffffu;

// ===========================================================================
// Traceback from (0, k) (Algorithm 1, "backtrack"): at a visited row, take ->
// mark b_i, j -= w_i and go to the next kept row; skip -> go to next(i); stop
// at i = n or j = 0.  In kept-row order a take always moves from kept index t
// to t - 1 (the next kept row in preorder, since a pruned interior is all
// "skip"), and a skip moves to skip[t].  The walk is monotone in t and j, so
// one warp reads it tile by tile.  A tile is 64 kept rows x 96 columns in
// shared memory: per column one 64-bit word of take bits (a block pair of the
// DP's), and per row its skip target, preorder position and suffix weight,
// brought in with asynchronous 8- and 4-byte copies.  Inside the tile a step
// is: lane l reads the bit of row t - l at the column reached after taking
// rows t..t-l+1, a warp min-reduction gives the first lane that does not take
// (the take-run's end), and that lane's row is the skip, whose target (and,
// speculatively, the target's own skip in the same column word) comes from
// the same tile.  The rows a step takes form a run of tile rows: they are
// gathered in a 64-bit mask and marked when the walk leaves the tile, so no
// global memory operation sits on the steps' chain of dependent operations.
// The copies are software-pipelined: on entering a tile the walker starts
// those of the tile below it, anchored at its entry column, into the other
// of two buffers; a walk that leaves downwards within 96 columns of that
// anchor (skips are short; ~15 columns per tile on the paper-scale trees)
// finds it on chip, and any other exit copies its tile on demand.
// With unit chunk weights, helper warps of the walking warp's CTA follow its
// position through shared memory and prefetch into L1 the tiles below it in
// its column band, for the demand copies.
// Planner mode (acc.mask != nullptr): the update is accepted in the greedy
// pass, or in refinement iff D[0][k] > sum of p_h over the current T_h
// (equivalent to G(T_-h, T'_h) > G(T) by Prop. 1); an accepted update
// replaces bit h of the holder masks by the traced set.
// ===========================================================================
constexpr int kTraceTileRows = 64;       // kept rows per traceback tile (one 64-bit word per column)
constexpr int kTraceTileCols = 96;       // columns per traceback tile (a multiple of 32)
constexpr int kTraceHelpers = 3;         // prefetching warps beside the walking one
constexpr int kTraceAhead = 4;           // tiles below the walker's that they prefetch
constexpr uint32_t kTracePollLimit = 1u << 22;   // polls of the walker's position (~0.4 s)

// 4- and 8-byte asynchronous global -> shared copies; with `read` false
// nothing is read and the destination is zero-filled
__device__ __forceinline__ void cp_async4(void *dst, const void *src, bool read)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"((uint32_t)__cvta_generic_to_shared(dst)),
                 "l"(__cvta_generic_to_global(src)), "r"(read ? 4 : 0)
                 : "memory");
}
__device__ __forceinline__ void cp_async8(void *dst, const void *src, bool read)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;" ::"r"((uint32_t)__cvta_generic_to_shared(dst)),
                 "l"(__cvta_generic_to_global(src)), "r"(read ? 8 : 0)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }

__device__ __forceinline__ void prefetch_l1(const void *p)
{
    asm volatile("prefetch.global.L1 [%0];" ::"l"(__cvta_generic_to_global(p)));
}

// Helper warps (threads 32 .. 32 * (1 + kTraceHelpers) - 1): while the walker
// works, prefetch the decision-bit lines of the kept-row blocks from its tile
// down to kTraceAhead tiles below, for the 64 columns ending at its column,
// nearest first, and the same rows of the skip targets and positions.  walk[0], walk[1]: the walker's tile (first row, column); walk[2]:
// set when the walk is over.  Every address is inside the item's arrays.
__device__ void trace_prefetch(const uint64_t *Bi, int npair, int C, int P, int nk, const int32_t *sk,
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
        const int b_hi = min(r0 >> 6, min(npair, (nk + 63) >> 6) - 1);      // 64-row block pairs
        const int b_lo = max(0, (r0 >> 6) - kTraceAhead);
        const int nb = b_hi - b_lo + 1;
        const int lines = nb > 0 ? nb * ng * C * 2 : 0;                    // a pair row spans two lines
        for (int x = ht; x < lines; x += NH) {
            const int hh = x & 1, c = (x >> 1) & (C - 1), gb = x >> (lgC + 1);
            // 64 columns span at most three chain warps: no run-time division
            const int bq = ng == 1 ? gb : ng == 2 ? gb >> 1 : gb / 3;
            const int gg = glo + (gb - bq * ng), b = b_hi - bq;
            const int ln = min((gg == glo ? (tlo & 31) : 0) + 16 * hh, 31);
            prefetch_l1(Bi + (((size_t)gg * npair + b) * C + c) * 32 + ln);
        }
        const int rlo = b_lo * 64, rhi = min(nk, (b_hi + 1) * 64);
        for (int r = rlo + 32 * ht; r < rhi; r += 32 * NH) {
            prefetch_l1(sk + r);
            prefetch_l1(rl + r);
        }
    }
}

// One traceback tile in shared memory: kept rows r0..r0+63 at the columns
// a, a-1, .., a-kTraceTileCols+1 (column index c = a - column).
struct TraceTile {
    uint64_t bits[kTraceTileCols];       // bit lr of bits[c]: take at row r0 + lr, column a - c
    int32_t skip[kTraceTileRows];        // skip target (kept index) of row r0 + lr, -1 past n
    int32_t pos[kTraceTileRows];         // preorder position of row r0 + lr (node id in the ABI mode)
    int32_t ws[kTraceTileRows + 1];      // suffix weight at row r0 + lr (lr = 64: at r0 + 64)
};

// BYNODE: the ABI mode (chosen bytes by node id, acc.mask == nullptr);
// otherwise the planner's accept-and-update mode.  UNIT: every chunk weight
// is 1 (and helper warps prefetch for the walker).  Template parameters, so
// that each walk carries no trace of the other modes.
template <int SKIPS, bool BYNODE, bool UNIT>
__global__ void __launch_bounds__(256)
k_traceback(int32_t n, DpWork w, int C, int P, int kpad,
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
    const int npair = (n + 63) / 64;                          // 64-row block pairs per chain warp
    const uint64_t *Bi = reinterpret_cast<const uint64_t *>(w.bits) + (size_t)bi * P * (size_t)npair * C * 32;
    const int32_t *rl = w.rowlist + (size_t)bi * n;
    const int32_t *sk = w.skip + (size_t)bi * n;
    const int32_t *ws = w.wsuf + (size_t)bi * (n + 1);
    const int nk = w.nkept[bi];
    if (threadIdx.x >= 32) {
        if (UNIT && threadIdx.x < 32 * (1 + kTraceHelpers) && kq > 0)
            trace_prefetch(Bi, npair, C, P, nk, sk, rl, walk);
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
    auto word_index = [&](int bp, int col) -> size_t {     // 8-byte word of rows bp*64.. at column col >= 1
        const int q = col - 1;
        const int tt = q >> lgC, c = q & (C - 1);             // C is a power of two
        return (((size_t)(tt >> 5) * npair + bp) * C + c) * 32 + (tt & 31);
    };
    // start the copies of the tile of rows r0.. at columns a, a-1, ..: lane l
    // copies rows r0+l and r0+32+l and columns a-l, a-32-l, .. (one 8-byte
    // word each); what lies left of column 1 or at rows >= nk is zero-filled
    // or stale, and never read as valid
    __shared__ TraceTile s_tile[2];
    auto stage = [&](TraceTile &T, int r0, int a) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int c = lane + 32 * h;
            const int r = r0 + c;
            const bool in = r < nk;
            cp_async4(&T.skip[c], in ? (const void *)(sk + r) : (const void *)Bi, in);
            cp_async4(&T.pos[c], in ? (const void *)(rl + r) : (const void *)Bi, in);
            if (!UNIT) cp_async4(&T.ws[c], in ? (const void *)(ws + r) : (const void *)Bi, in);
        }
        if (!UNIT && lane == 0) cp_async4(&T.ws[kTraceTileRows], ws + min(r0 + kTraceTileRows, nk), true);
#pragma unroll
        for (int c = lane; c < kTraceTileCols; c += 32) {
            const int col = a - c;
            cp_async8(&T.bits[c], col >= 1 ? (const void *)&Bi[word_index(r0 >> 6, col)] : (const void *)Bi, col >= 1);
        }
        cp_async_commit();
    };
    int t = nk - 1;                 // row of position 0 (the first root): swept last
    int pr0 = -1, pa = 0;           // the tile copied ahead: rows pr0.., columns pa, pa-1, ..
    for (int guard = 0; guard <= 2 * n + 2 && t >= 0 && j > 0; ++guard) {
        // ---- the tile holding (t, j), from the copy made ahead when it is that one
        const int r0 = t & ~(kTraceTileRows - 1);
        const int slot = (r0 / kTraceTileRows) & 1;
        TraceTile &T = s_tile[slot];
        cp_async_wait_all();
        __syncwarp();                         // every lane's copies, and the last tile's reads, are done
        int a = pa;
        if (r0 != pr0 || j <= pa - kTraceTileCols) {
            a = j;
            stage(T, r0, a);
            cp_async_wait_all();
            __syncwarp();
        }
        // the preorder positions of this lane's two tile rows, for marking
        // (node ids in the ABI mode, which marks chosen[] by node id)
        int posv[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            posv[h] = T.pos[lane + 32 * h];
            if (BYNODE && r0 + lane + 32 * h < nk) posv[h] = order[posv[h]];
        }
        if (lane == 0) {                      // where the helpers prefetch next
            walk[1] = j;
            walk[0] = r0;
        }
        // ---- copy the tile below ahead, anchored at this column: a walk that
        // leaves downwards (skips are short: ~15 columns per 64-row tile on the
        // paper-scale trees) finds it on chip (tile width: 96 columns took the
        // weighted plan's walks 15.1 -> 14.6 ms and left the unit-weight ones
        // as they were, against 64)
        pr0 = r0 - kTraceTileRows;
        pa = j;
        if (pr0 >= 0) stage(s_tile[slot ^ 1], pr0, pa);
        // ---- walk inside the tile: lane l tests row t-l at the column reached
        // after taking rows t..t-l+1.  The rows a step takes are a run of tile
        // rows, gathered in `taken` and marked when the walk leaves the tile,
        // off the steps' chain of dependent operations.
        uint64_t taken = 0;
        bool inside = t >= r0 && a - j < kTraceTileCols;      // j > 0 here
        while (inside) {
            const int lt = t - r0, lr = lt - lane;
            int col, coln;
            if (UNIT) {
                col = j - lane;
                coln = col - 1;
            } else {
                const int wt = T.ws[lt + 1];
                col = j - (T.ws[max(lr + 1, 0)] - wt);
                coln = j - (T.ws[max(lr, 0)] - wt);
            }
            const int ci = a - col;
            const bool valid = lr >= 0 && col >= 1 && ci < kTraceTileCols;
            const int lrm = lr & (kTraceTileRows - 1);
            const uint64_t word = T.bits[min(max(ci, 0), kTraceTileCols - 1)];
            const int skr = T.skip[lrm];
            const bool take = valid && ((word >> lrm) & 1ull);
            // the first lane that does not take (32: all take): rows t..t-L+1 are taken
            const int L = (int)__reduce_min_sync(kFull, take ? 32u : (unsigned)lane);
            // speculation for the lane that ends the take-run: its skip lands
            // on row skr at the same column (the same word); while that row is
            // in the tile and is skipped as well, the walk goes on to its skip
            // target in the same step, up to SKIPS times (skips often come in
            // pairs; trees with wide fan-out have longer chains and use three)
            int tnext = skr;
            bool more = true;
#pragma unroll
            for (int d = 0; d < SKIPS; ++d) {
                const int l1 = tnext - r0;
                more = more && l1 >= 0 && !((word >> (l1 & (kTraceTileRows - 1))) & 1ull);
                const int s1 = T.skip[l1 & (kTraceTileRows - 1)];
                tnext = more ? s1 : tnext;
            }
            if (L > 0) taken |= ((2ull << (L - 1)) - 1) << (lt - L + 1);
            // next state: after 32 takes, row t-32 at the column after them;
            // else lane L's row is skipped (to tnext) when it lies in the tile,
            // and otherwise the walk leaves the tile at (t-L, its column)
            const int colL = UNIT ? j - L : __shfl_sync(kFull, L == 32 ? coln : col, L == 32 ? 31 : L);
            const int skL = __shfl_sync(kFull, tnext, L & 31);
            const bool all = L == 32;
            const bool inL = !all && lt - L >= 0 && colL >= 1 && a - colL < kTraceTileCols;
            t = all ? t - 32 : inL ? skL : t - L;       // skL = -1: past n
            j = colL;
            inside = (all || inL) && t >= r0 && j > 0 && a - j < kTraceTileCols;
        }
        // ---- mark the taken rows: lane l the tile rows l and l+32
#pragma unroll
        for (int h = 0; h < 2; ++h)
            if ((taken >> (lane + 32 * h)) & 1ull) {
                if (BYNODE) chosen[(size_t)item * n + posv[h]] = 1;
                else atomicOr(M + posv[h], hbit);             // a reduction: the walk does not wait on it
            }
    }
    cp_async_wait_all();                      // no copy outlives the block
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
    const int skips = inst->trace_skips >= 3 ? 3 : 1;
    auto go = [&](auto kern) {
        kern<<<batch, 256, 0, st>>>(inst->n, work, g.C, g.P, g.kpad, item_budget, inst->d_order, chosen, a);
    };
    if (skips == 3) {
        if (bynode) unit ? go(k_traceback<3, true, true>) : go(k_traceback<3, true, false>);
        else unit ? go(k_traceback<3, false, true>) : go(k_traceback<3, false, false>);
    } else {
        if (bynode) unit ? go(k_traceback<1, true, true>) : go(k_traceback<1, true, false>);
        else unit ? go(k_traceback<1, false, true>) : go(k_traceback<1, false, false>);
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
