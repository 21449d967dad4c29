// Exact capacity-k prefix-complete tree knapsack (Eq. 9, Theorem 1); its
// traceback (Algorithm 1's backtracking) is in pp_traceback.cu.
//
//   D[i][0] = 0, D[n][j] = 0,
//   D[i][j] = max{ D[next(i)][j], p_i + D[i+1][j - w_i] }   (take needs j >= w_i)
//
// Rows are preorder positions swept from n-1 down to 0, so row i needs row
// i+1 and row next(i) > i.  Along the capacity axis column j needs only
// column j of row next(i) and column j - w_i of row i+1: the dependency flows
// from low to high columns.  Both kernels split the columns over threads,
// each thread owning C consecutive columns in registers.
//
// k_tree_dp_wave (all chunk weights <= 4): one thread-block cluster of CL
//   CTAs per DP, WPC warps per CTA, and no block-wide barrier in the row loop.
//   Every warp sweeps its own columns row after row; warp g needs, for row i,
//   the last w_i values of row i+1 of warp g-1, which that warp publishes
//   into a ring in warp g's shared memory (DSMEM when g-1 is in the previous
//   CTA of the cluster).  Each slot carries a lap bit, so a slot validates
//   itself and no fence is needed; the consumer acknowledges finished rows so
//   the producer never overwrites an unread slot.  So warps form a wavefront,
//   warp g lagging warp g-1 by a sub-block of rows.  Every wait is bounded in
//   time and reports PP_ETIMEOUT through the status word.
// k_tree_dp_flat (any weight): one CTA per DP, row i+1 staged in shared memory
//   and one __syncthreads per row.
//
// Skip rows: next(i) = i+1 is the row just computed (registers), next(i) = n
// is the zero row, and any other next(i) is the top of the skip-row stack,
// which the wave kernel also keeps in registers (pushes store the new top to
// shared memory, or to instance scratch below L_smem levels; pops reload it).
//
// Decision bits (take = strictly better, so the traceback returns the
// lexicographically smallest optimal preorder indicator): one __ballot_sync
// per (warp, c) gives the word ((item * P + g) * n + i) * C + c whose bit
// `lane` is column (g * 32 + lane) * C + c + 1.
#include <algorithm>
#include <climits>
#include <mutex>

#include "pp_internal.cuh"

namespace pp {

constexpr unsigned kFull = 0xffffffffu;

// ===========================================================================
// inline PTX helpers (cluster, DSMEM, acquire / release, timer)
// ===========================================================================
__device__ __forceinline__ uint32_t cluster_ctarank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ uint32_t cluster_nctarank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ void cluster_sync_all()
{
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ uint32_t smem_addr(const void *p)
{
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ uint32_t map_to_rank(uint32_t addr, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}
__device__ __forceinline__ void ld_volatile_v2_u64(const uint64_t *p, uint64_t &a, uint64_t &b)
{
    asm volatile("ld.volatile.shared.v2.u64 {%0, %1}, [%2];" : "=l"(a), "=l"(b) : "r"(smem_addr(p)) : "memory");
}
// generic address of `p` (this CTA's shared memory) in CTA `rank` of the cluster
__device__ __forceinline__ void *map_generic(const void *p, uint32_t rank)
{
    uint64_t r;
    asm volatile("mapa.u64 %0, %1, %2;" : "=l"(r) : "l"(p), "r"(rank));
    return reinterpret_cast<void *>(r);
}
__device__ __forceinline__ uint64_t global_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Testing hook (pp_test_inject): the chain warp with this index never
// publishes its ring counter, so its right neighbour's bounded wait runs out.
__device__ int32_t g_drop_publish_warp = -1;

namespace wavecfg {
constexpr int kRing = 64;                         // ring slots (rows), power of two
constexpr int kPub = 8;                           // publish / acknowledge every kPub rows
constexpr uint64_t kWaitLimitNs = 500ull * 1000 * 1000;   // one wait gives up after 0.5 s
constexpr int64_t kNeg = LLONG_MIN / 2;           // D at a negative column: never taken
}  // namespace wavecfg

// Bounded spin (warp-uniform): `ready()` is re-evaluated until it holds.
// Gives up after kWaitLimitNs, or as soon as another wait of the launch has
// given up; the first to give up sets PP_ETIMEOUT.
template <typename Ready>
__device__ __forceinline__ bool spin_until(Ready ready, int32_t *status)
{
    uint64_t t0 = 0;
    for (uint32_t it = 0;; ++it) {
        if (__all_sync(kFull, ready())) return true;
        if (it == 0) t0 = global_ns();
        if ((it & 63) == 63) {
            bool give_up = *(volatile int32_t *)status == PP_ETIMEOUT;
            if (!give_up && global_ns() - t0 > wavecfg::kWaitLimitNs) {
                give_up = true;
                if ((threadIdx.x & 31) == 0) atomicExch(status, (int32_t)PP_ETIMEOUT);
            }
            if (__any_sync(kFull, give_up)) return false;
            __nanosleep(32);
        }
    }
}

__host__ __device__ inline size_t wave_fixed_bytes(int WPC, int WMAX)
{
    size_t b = (size_t)WPC * wavecfg::kRing * WMAX * sizeof(uint64_t) + (size_t)WPC * 2 * 32 * 12 +
               (size_t)WPC * sizeof(uint32_t);
    return (b + 15) & ~(size_t)15;
}

// take-branch base values sh[c] = D[i+1][col_c - W] for a static weight W:
// own registers for c >= W, the left neighbour lane for c < W, and for lane 0
// the boundary values bnd[q] = D[i+1][base - WMAX + 1 + q] of the previous warp.
template <int C, int WMAX, int W>
__device__ __forceinline__ void shift_by(const int64_t (&cur)[C], const int64_t (&bnd)[WMAX], bool lane0,
                                         int64_t (&sh)[C])
{
#pragma unroll
    for (int c = 0; c < C; ++c) {
        if (c >= W) {
            sh[c] = cur[c - W];
        } else {
            const int64_t v = __shfl_up_sync(kFull, cur[C - W + c], 1);
            sh[c] = lane0 ? bnd[WMAX - W + c] : v;
        }
    }
}

template <int C, int WMAX>
__device__ __forceinline__ void shift_row(const int64_t (&cur)[C], const int64_t (&bnd)[WMAX], bool lane,
                                          int w, int64_t (&sh)[C])
{
    if constexpr (WMAX == 1) {
        shift_by<C, WMAX, 1>(cur, bnd, lane, sh);
    } else {
        // branch-free: every candidate shift, then a select by w (a per-row
        // branch would end the unrolled straight-line block of rows)
        int64_t up[WMAX];  // up[q]: column C-1-q of the lane to the left (lane 0: the boundary)
#pragma unroll
        for (int q = 0; q < WMAX; ++q) {
            const int64_t v = __shfl_up_sync(kFull, cur[C - 1 - q], 1);
            up[q] = lane ? bnd[WMAX - 1 - q] : v;
        }
#pragma unroll
        for (int c = 0; c < C; ++c) {
            int64_t v = c >= 1 ? cur[c - 1 < 0 ? 0 : c - 1] : up[0];
#pragma unroll
            for (int ww = 2; ww <= WMAX; ++ww) {
                const int64_t cand = c >= ww ? cur[c - ww < 0 ? 0 : c - ww] : up[ww - 1 - c < 0 ? 0 : ww - 1 - c];
                v = w == ww ? cand : v;
            }
            sh[c] = v;
        }
    }
}

// Rows are swept in sub-blocks of kSub rows; the hand-off checks run once
// per sub-block and the rows inside are unrolled.
//
// Hand-off between warp g-1 (producer) and warp g (consumer), fence-free:
// for each row r the producer stores its last WMAX values of that row into
// slot r % kRing of a ring in the consumer's shared memory, each as one
// 64-bit word D | lap << 63 with lap = (r / kRing) % 2 (every D is in
// [0, 2^62], so bit 63 is free).  A slot is self-validating: the consumer
// re-reads the slots of a sub-block until every lap bit is the expected one.
// The consumer reports the rows it has finished with a relaxed store into the
// producer's shared memory, issued only after it used the values it read,
// and the producer never writes a slot whose previous value is unread.
constexpr int kSub = wavecfg::kPub;
constexpr uint64_t kLapBit = 1ull << 63;

template <int C, int WMAX, bool SPILL>
__global__ void __launch_bounds__(512, 1)
k_tree_dp_wave(int32_t n, int32_t nblk, const int64_t *__restrict__ rowp,
               const int32_t *__restrict__ rowm, const int32_t *__restrict__ nkept,
               const int32_t *__restrict__ item_budget, int32_t max_budget,
               const int32_t *__restrict__ item_active, int64_t *__restrict__ best,
               uint32_t *__restrict__ bits, int64_t *__restrict__ gstack, int L_smem, int L_glob,
               int32_t *__restrict__ status, int32_t batch, int32_t slot_base, int32_t ranked)
{
    using namespace wavecfg;
    extern __shared__ __align__(16) unsigned char smem[];
    const int CL = (int)cluster_nctarank();
    const int cr = (int)cluster_ctarank();
    int item = blockIdx.x / CL;
    if (ranked) {
        // split launch (batch <= 32): slot s of the two launches takes the
        // item of rank s by kept rows, most first (ties to the lower index,
        // inactive items last), so the narrower second launch gets the
        // smallest sweeps; every CTA of a cluster computes the same item
        __shared__ int s_item;
        if (threadIdx.x < 32) {
            const int x = threadIdx.x;
            const int key = x < batch && (!item_active || item_active[x]) ? nkept[x] : -1;
            int rank = 0;
            for (int y = 0; y < batch; ++y) {
                const int ky = __shfl_sync(kFull, key, y);
                rank += ky > key || (ky == key && y < x);
            }
            const unsigned m = __ballot_sync(kFull, x < batch && rank == slot_base + item);
            if (x == 0) s_item = m ? __ffs((int)m) - 1 : -1;
        }
        __syncthreads();
        item = s_item;
        if (item < 0) return;           // no such slot: uniform over the cluster
    }
    const int NT = blockDim.x;
    const int WPC = NT >> 5;
    const int wl = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int P = CL * WPC;
    const int g = cr * WPC + wl;
    const int kpad = P * 32 * C;

    // uniform over the whole cluster: return before any DSMEM traffic
    if (item_active && !item_active[item]) return;
    const int32_t kreq = item_budget[item];
    if (kreq < 0 || kreq > max_budget) {
        if (cr == 0 && threadIdx.x == 0) {
            atomicExch(status, (int32_t)PP_EBOUNDS);
            best[item] = 0;
        }
        return;
    }
    const int k = kreq < kpad ? kreq : kpad;   // kpad covers min(max_budget, total weight)

    uint64_t *ring = reinterpret_cast<uint64_t *>(smem);                           // [WPC][kRing][WMAX]
    int64_t *pstage = reinterpret_cast<int64_t *>(ring + (size_t)WPC * kRing * WMAX);  // [WPC][2][32] profits
    int32_t *mstage = reinterpret_cast<int32_t *>(pstage + (size_t)WPC * 64);         // [WPC][2][32] metadata
    uint32_t *ack = reinterpret_cast<uint32_t *>(mstage + (size_t)WPC * 64);          // [WPC]
    int64_t *stk = reinterpret_cast<int64_t *>(smem + wave_fixed_bytes(WPC, WMAX)); // [WPC][L_smem][C][32]
    for (int x = threadIdx.x; x < WPC * kRing * WMAX; x += NT) ring[x] = kLapBit;  // lap of row -1
    if (threadIdx.x < WPC) ack[threadIdx.x] = 0;
    cluster_sync_all();     // every CTA initialised before any remote write

    const bool has_prev = g > 0, has_next = g < P - 1;
    const bool prev_remote = has_prev && wl == 0;
    // the previous warp's acknowledgement word, as a generic cluster address
    volatile uint32_t *pv_ack = nullptr;
    if (has_prev)
        pv_ack = reinterpret_cast<volatile uint32_t *>(
            map_generic(ack + (prev_remote ? WPC - 1 : wl - 1), (uint32_t)(prev_remote ? cr - 1 : cr)));
    const uint64_t *my_ring = ring + (size_t)wl * kRing * WMAX;
    // the next warp's ring through the cluster window (local or remote alike),
    // as a generic address: a plain volatile store lets the compiler schedule
    // the rows around the hand-off (an inline-PTX store cost ~5% per row)
    volatile uint64_t *const nx_gen = has_next ? (volatile uint64_t *)map_generic(ring + (size_t)((wl + 1) % WPC) * kRing * WMAX,
                                                                 (uint32_t)(wl == WPC - 1 ? cr + 1 : cr)) : nullptr;
    int64_t *const my_ps = pstage + (size_t)wl * 64;
    int32_t *const my_ms = mstage + (size_t)wl * 64;
    uint32_t ack_seen = 0;
    bool aborted = false;
    const bool publish = has_next && lane == 31 && g != g_drop_publish_warp;   // this lane stores
    const bool lane0 = lane == 0;

    // decision bits in block pairs: the words of 32-row blocks 2b and 2b+1
    // of one column sit side by side (one 8-byte word per 64 rows)
    uint32_t *Bw = bits + ((size_t)item * P + g) * (size_t)nblk * C * 32 + 2 * lane;
    int64_t *gst = gstack + (((size_t)item * L_glob) * CL + cr) * (size_t)C * NT;
    int64_t *const my_gst = gst + threadIdx.x;
    // this warp's shared-memory stack levels: a column's word of a level sits
    // at a compile-time offset from the lane's base
    int64_t *const my_stk = stk + (size_t)wl * L_smem * C * 32 + lane;
    // the kept rows of the pruned sweep, with their profit and metadata
    // gathered in sweep order
    const int nrows = nkept[item];
    const int64_t *Rp = rowp + (size_t)item * n;
    const int32_t *Rm = rowm + (size_t)item * n;
    const int nblk_item = (nrows + 31) / 32;

    int64_t cur[C], top[C];
#pragma unroll
    for (int c = 0; c < C; ++c) {
        cur[c] = 0;          // row n is the zero boundary, and the top of the empty stack
        top[c] = 0;
    }
    // row metadata, 32 rows per block: lane l copies row blk*32 + l one block
    // ahead into a double buffer in shared memory with cp.async (a register
    // load in flight across the rows held a scoreboard that the rows' own
    // waits then also waited on); the warp turns the flags into warp-uniform
    // masks, bit = row of the block.  Rows past the last one are no-ops
    // (p = -inf, skip = the row just computed), so every warp sweeps
    // nblk_item * 32 rows.
    auto prefetch = [&](int b) {
        const int r = b * 32 + lane, o = (b & 1) * 32 + lane;
        if (r < nrows) {
            asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(smem_addr(my_ps + o)),
                         "l"(__cvta_generic_to_global(Rp + r)) : "memory");
            asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_addr(my_ms + o)),
                         "l"(__cvta_generic_to_global(Rm + r)) : "memory");
        } else {
            my_ps[o] = kNeg;
            my_ms[o] = 0;
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
    prefetch(0);
    // boundary carried between sub-blocks: D[i+1][base - WMAX + 1 + q] of the
    // previous warp for the first row of the next sub-block (row n: zeros)
    int64_t carry[WMAX];
#pragma unroll
    for (int q = 0; q < WMAX; ++q) carry[q] = has_prev ? 0 : (q == WMAX - 1 ? 0 : kNeg);

    for (int blk = 0; blk < nblk_item && !aborted; ++blk) {
        asm volatile("cp.async.wait_all;" ::: "memory");
        __syncwarp();
        const int64_t *const my_p = my_ps + (blk & 1) * 32;      // [32] profits of the block
        const int32_t *const my_m = my_ms + (blk & 1) * 32;      // [32] metadata of the block
        const int32_t mnext = my_m[lane];
        const uint32_t cur_rows = __ballot_sync(kFull, (mnext & (3 << 3)) == (kWaveCur << 3));
        const uint32_t push_rows = __ballot_sync(kFull, (mnext & kWavePush) != 0);
        const uint32_t reload_rows = __ballot_sync(kFull, (mnext & kWaveReload) != 0);
        const uint32_t zero_rows = __ballot_sync(kFull, (mnext & kWaveZeroTop) != 0);
        uint32_t w1_rows = 0, w2_rows = 0;          // bits 0 and 1 of w - 1 (weights <= 4)
        if (WMAX > 1) {
            w1_rows = __ballot_sync(kFull, (mnext & 1) != 0);
            w2_rows = __ballot_sync(kFull, (mnext & 2) != 0);
        }
        if (blk + 1 < nblk_item) prefetch(blk + 1);     // the other buffer: block blk - 1 is done
        uint32_t wbits[C];
#pragma unroll
        for (int c = 0; c < C; ++c) wbits[c] = 0;
        for (int sb = 0; sb < 32 / kSub; ++sb) {
            const int r0 = blk * 32 + sb * kSub;
            // producer: slots r0..r0+kSub-1 last held rows r0-kRing.., which the
            // consumer has finished reading once it reports row r0+kSub+1-kRing
            // consumer: rows r0..r0+kSub-1 of the previous warp, all with the
            // lap bit of this pass over the ring
            const uint64_t lap = (uint64_t)((r0 / kRing) & 1) << 63;
            const uint64_t *sl = my_ring + (size_t)(r0 & (kRing - 1)) * WMAX;
            // the slots' values (read by the wait below); the first warp has no
            // previous warp and reads zeros (column 0 of every row is 0)
            uint64_t sv[WMAX == 1 ? kSub : 1];
#pragma unroll
            for (int u = 0; u < (WMAX == 1 ? kSub : 1); ++u)
                if (!has_prev) sv[u] = 0;
            const bool need_ack = has_next && r0 + kSub + 1 > kRing && ack_seen < (uint32_t)(r0 + kSub + 1 - kRing);
            if (has_prev || need_ack) {
                const uint32_t need = (uint32_t)(r0 + kSub + 1 - kRing);
                auto ready = [&] {
                    bool ok = true;
                    if (need_ack) {
                        ack_seen = *(volatile uint32_t *)(ack + wl);
                        ok = ack_seen >= need;
                    }
                    if (!has_prev) return ok;
                    uint64_t bad = 0;
                    if (WMAX == 1) {
#pragma unroll
                        for (int u = 0; u < kSub; u += 2) {
                            uint64_t x, y;
                            ld_volatile_v2_u64(sl + u, x, y);
                            sv[u] = x;
                            sv[u + 1] = y;
                            bad |= (x ^ lap) | (y ^ lap);
                        }
                    } else {
#pragma unroll
                        for (int u = 0; u < kSub * WMAX; u += 2) {
                            uint64_t x, y;
                            ld_volatile_v2_u64(sl + u, x, y);
                            bad |= (x ^ lap) | (y ^ lap);
                        }
                    }
                    return ok && (bad & kLapBit) == 0;
                };
                if (!spin_until(ready, status)) {
                    aborted = true;
                    break;
                }
            }
            const int s8 = sb * kSub;
            const uint32_t cb = cur_rows >> s8, pb = push_rows >> s8, rb = reload_rows >> s8;
            const uint32_t stk8 = ((push_rows | reload_rows | zero_rows) >> s8) & ((1u << kSub) - 1);
            const uint32_t wb1 = w1_rows >> s8, wb2 = w2_rows >> s8;
            uint32_t wb8[C];
#pragma unroll
            for (int c = 0; c < C; ++c) wb8[c] = 0;
            // the sub-block's profits, read before any skip-row stack store
            // (which the compiler cannot move a later shared load above)
            int64_t pv[kSub];
#pragma unroll
            for (int u = 0; u < kSub; ++u) pv[u] = my_p[s8 + u];
            // one row of Eq. 9 for this warp's columns; STACK: the row may push or pop
            auto row = [&](const int u, const bool STACK, const int SRC) {
                const int64_t p = pv[u];
                // bnd[q] = D[i+1][base - WMAX + 1 + q]: row r-1 of the previous warp
                // (the first warp's sv is all zero: column 0 of every row is 0)
                int64_t bnd[WMAX];
                if (u == 0) {
#pragma unroll
                    for (int q = 0; q < WMAX; ++q) bnd[q] = carry[q];
                } else if (WMAX == 1) {
                    bnd[0] = (int64_t)(sv[WMAX == 1 ? u - 1 : 0] & ~kLapBit);
                } else if (has_prev) {
#pragma unroll
                    for (int q = 0; q < WMAX; ++q) bnd[q] = (int64_t)(sl[(u - 1) * WMAX + q] & ~kLapBit);
                } else {
#pragma unroll
                    for (int q = 0; q < WMAX; ++q) bnd[q] = carry[q];
                }
                const int w = WMAX == 1 ? 1 : 1 + (int)((wb1 >> u) & 1u) + 2 * (int)((wb2 >> u) & 1u);
                int64_t sh[C];
                shift_row<C, WMAX>(cur, bnd, lane0, w, sh);
                // skip row: row i+1 (a leaf) or the stack top
                const bool from_cur = (cb >> u) & 1u;
#pragma unroll
                for (int c = 0; c < C; ++c) {
                    const int64_t sk = SRC == 1 ? cur[c] : SRC == 2 ? top[c] : (from_cur ? cur[c] : top[c]);
                    const int64_t t = p + sh[c];
                    const bool take = t > sk;
                    cur[c] = take ? t : sk;
                    if (take) wb8[c] |= 1u << u;
                }
                // hand this row's last WMAX columns to the next warp (lane 31 only)
#pragma unroll
                for (int q = 0; q < WMAX; ++q)
                    if (publish) nx_gen[(r0 & (kRing - 1)) * WMAX + u * WMAX + q] = (uint64_t)cur[C - WMAX + q] | lap;
                // skip-row stack (warp-uniform masks): push (the new row becomes
                // the top), reload the new top after a pop, or reset it to the zero row
                // the masks are warp-uniform; with unit weights, saying so with a
                // vote lets the compiler drop the reconvergence of every row's
                // branch in the stack path (DP phase of the paper-scale plan
                // 160.1 -> 156.2 ms; the weighted kernels ran slower with it)
                if (STACK && (WMAX == 1 ? __any_sync(kFull, (stk8 >> u) & 1u) : ((stk8 >> u) & 1u) != 0)) {
                    if ((pb >> u) & 1u) {
                        const int lvl = (int)((uint32_t)my_m[s8 + u] >> 16);
#pragma unroll
                        for (int c = 0; c < C; ++c) top[c] = cur[c];
                        if (!SPILL || lvl < L_smem) {
#pragma unroll
                            for (int c = 0; c < C; ++c) my_stk[((size_t)lvl * C + c) * 32] = cur[c];
                        } else {
#pragma unroll
                            for (int c = 0; c < C; ++c) my_gst[(size_t)(lvl - L_smem) * CL * C * NT + (size_t)c * NT] = cur[c];
                        }
                    } else if ((rb >> u) & 1u) {
                        const int lvl = (int)((uint32_t)my_m[s8 + u] >> 16);
                        if (!SPILL || lvl < L_smem) {
#pragma unroll
                            for (int c = 0; c < C; ++c) top[c] = my_stk[((size_t)lvl * C + c) * 32];
                        } else {
#pragma unroll
                            for (int c = 0; c < C; ++c) top[c] = my_gst[(size_t)(lvl - L_smem) * CL * C * NT + (size_t)c * NT];
                        }
                    } else {
#pragma unroll
                        for (int c = 0; c < C; ++c) top[c] = 0;
                    }
                }
            };
            const uint32_t cb8 = cb & ((1u << kSub) - 1);
            if (stk8 == 0) {
                if (cb8 == 0) {
#pragma unroll
                    for (int u = 0; u < kSub; ++u) row(u, false, 2);   // every skip row is the top
                } else {
#pragma unroll
                    for (int u = 0; u < kSub; ++u) row(u, false, 0);   // no push or pop in these rows
                }
            } else if (cb8 == 0) {
#pragma unroll
                for (int u = 0; u < kSub; ++u) row(u, true, 2);        // stack operations, every skip row the top
            } else {
#pragma unroll
                for (int u = 0; u < kSub; ++u) row(u, true, 0);
            }
#pragma unroll
            for (int c = 0; c < C; ++c) wbits[c] |= wb8[c] << s8;
            if (has_prev) {
                // the last row of this sub-block feeds the first row of the next one
                if (WMAX == 1) {
                    carry[0] = (int64_t)(sv[WMAX == 1 ? kSub - 1 : 0] & ~kLapBit);
                } else {
#pragma unroll
                    for (int q = 0; q < WMAX; ++q) carry[q] = (int64_t)(sl[(kSub - 1) * WMAX + q] & ~kLapBit);
                }
                // report the finished rows to the previous warp (values already used)
                if (lane == 0) *pv_ack = (uint32_t)(r0 + kSub);
            }
        }
#pragma unroll
        for (int c = 0; c < C; ++c) Bw[((size_t)(blk >> 1) * C + c) * 64 + (blk & 1)] = wbits[c];
    }

    asm volatile("cp.async.wait_all;" ::: "memory");   // nothing in flight into this CTA's shared memory
    if (!aborted) {
        if (k == 0) {
            if (g == 0 && lane == 0) best[item] = 0;
        } else {
            const int q = k - 1;
            const int tt = q / C;
            const int cc = q - tt * C;
            int64_t v = cur[0];
#pragma unroll
            for (int c = 1; c < C; ++c) v = cc == c ? cur[c] : v;
            if (g == (tt >> 5) && lane == (tt & 31)) best[item] = v;
        }
    }
    cluster_sync_all();     // no CTA leaves while a neighbour may still write its shared memory
}

// ===========================================================================
// General kernel (any chunk weight): one CTA, one barrier per row.
// ===========================================================================
constexpr int kMetaRows = 256;

static size_t flat_smem_fixed(int kpad)
{
    return 2 * (size_t)kpad * sizeof(int64_t) + 2 * kMetaRows * (sizeof(int64_t) + 2 * sizeof(int32_t));
}

template <int C>
__global__ void __launch_bounds__(1024, 1)
k_tree_dp_flat(int32_t n, const int32_t *__restrict__ rowlist, const int32_t *__restrict__ nkept,
               const int64_t *__restrict__ profit, const int32_t *__restrict__ order,
               const int32_t *__restrict__ wpre, const int32_t *__restrict__ meta,
               const int32_t *__restrict__ item_budget, int32_t max_budget,
               const int32_t *__restrict__ item_active, int64_t *__restrict__ best,
               uint32_t *__restrict__ bits, int64_t *__restrict__ gstack, int L_smem, int L_glob,
               int32_t *__restrict__ status)
{
    extern __shared__ __align__(16) unsigned char smem[];
    const int T = blockDim.x;
    const int t = threadIdx.x;
    const int lane = t & 31, warp = t >> 5;
    const int P = T >> 5;
    const int item = blockIdx.x;
    const int kpad = T * C;

    if (item_active && !item_active[item]) return;
    const int32_t kreq = item_budget[item];
    if (kreq < 0 || kreq > max_budget) {
        if (t == 0) {
            atomicExch(status, (int32_t)PP_EBOUNDS);
            best[item] = 0;
        }
        return;
    }
    const int k = kreq < kpad ? kreq : kpad;

    int64_t *srow = reinterpret_cast<int64_t *>(smem);          // [2][C][T]
    int64_t *sstk = srow + 2 * (size_t)kpad;                    // [L_smem][C][T]
    int64_t *sp = sstk + (size_t)L_smem * kpad;                 // [2][kMetaRows]
    int32_t *sw = reinterpret_cast<int32_t *>(sp + 2 * kMetaRows);
    int32_t *sm = sw + 2 * kMetaRows;
    int64_t *gst = gstack + (size_t)item * L_glob * kpad;
    const int64_t *Pp = profit + (size_t)item * n;
    const int nblk = (n + 63) / 64 * 2;                      // 32-row blocks, in pairs
    uint32_t *Bw = bits + ((size_t)item * P + warp) * (size_t)nblk * C * 32 + 2 * lane;
    const int nrows = rowlist ? nkept[item] : n;
    const int32_t *rows = rowlist ? rowlist + (size_t)item * n : nullptr;
    uint32_t wbits[C];
#pragma unroll
    for (int c = 0; c < C; ++c) wbits[c] = 0;

    int64_t cur[C];
#pragma unroll
    for (int c = 0; c < C; ++c) {
        cur[c] = 0;
        srow[c * T + t] = 0;
    }
    for (int x = t; x < kMetaRows && x < nrows; x += T) {
        const int i = rows ? rows[x] : n - 1 - x;
        sp[x] = Pp[order ? order[i] : i];
        sw[x] = wpre[i];
        sm[x] = meta[i];
    }
    __syncthreads();

    int64_t nx_p = 0;
    int32_t nx_w = 0, nx_m = 0;
    for (int r = 0; r < nrows; ++r) {
        const int blk = r / kMetaRows, off = r - blk * kMetaRows, buf = (blk & 1) * kMetaRows;
        if (off == 0) {
            const int x = (blk + 1) * kMetaRows + t;
            if (t < kMetaRows && x < nrows) {
                const int ii = rows ? rows[x] : n - 1 - x;
                nx_p = Pp[order ? order[ii] : ii];
                nx_w = wpre[ii];
                nx_m = meta[ii];
            }
        }
        const int64_t p = sp[buf + off];
        const int w = sw[buf + off];
        const int32_t m = sm[buf + off];
        const int skip = meta_skip(m), push = meta_push(m);
        const int64_t *prev = srow + (r & 1) * kpad;
        int64_t *outr = srow + ((r + 1) & 1) * kpad;
        const uint32_t mrow = 1u << (r & 31);
#pragma unroll
        for (int c = 0; c < C; ++c) {
            int64_t s;
            if (skip == kSkipCur) s = cur[c];
            else if (skip == kSkipZero) s = 0;
            else if (skip < L_smem) s = sstk[((size_t)skip * C + c) * T + t];
            else s = gst[((size_t)(skip - L_smem) * C + c) * T + t];
            const int jj = t * C + c + 1 - w;
            bool take = false;
            int64_t v = s;
            if (jj >= 0) {
                int64_t base = 0;
                if (jj > 0) {
                    const int q = jj - 1;
                    base = prev[(q % C) * T + q / C];
                }
                const int64_t tv = p + base;
                if (tv > s) {
                    v = tv;
                    take = true;
                }
            }
            cur[c] = v;
            outr[c * T + t] = v;
            if (take) wbits[c] |= mrow;
        }
        if ((r & 31) == 31 || r == nrows - 1) {
#pragma unroll
            for (int c = 0; c < C; ++c) {
                Bw[((size_t)(r >> 6) * C + c) * 64 + ((r >> 5) & 1)] = wbits[c];
                wbits[c] = 0;
            }
        }
        if (push >= 0) {
#pragma unroll
            for (int c = 0; c < C; ++c) {
                if (push < L_smem) sstk[((size_t)push * C + c) * T + t] = cur[c];
                else gst[((size_t)(push - L_smem) * C + c) * T + t] = cur[c];
            }
        }
        if (off == kMetaRows - 1) {
            const int x = (blk + 1) * kMetaRows + t;
            const int nb = ((blk + 1) & 1) * kMetaRows;
            if (t < kMetaRows && x < nrows) {
                sp[nb + t] = nx_p;
                sw[nb + t] = nx_w;
                sm[nb + t] = nx_m;
            }
        }
        __syncthreads();
    }
    if (k == 0) {
        if (t == 0) best[item] = 0;
    } else {
        const int q = k - 1;
        if (q / C == t) {
#pragma unroll
            for (int c = 0; c < C; ++c)
                if (c == q % C) best[item] = cur[c];
        }
    }
}

constexpr int kPruneCluster = 8;         // CTAs per item of the pruned-sweep kernel

// ===========================================================================
// Pruned sweep (one cluster of CTAs per item).  A strict descendant set with
// no positive profit is never worth taking: for a parent x whose strict
// descendants all have p <= 0, D[x+1][.] = D[next(x)][.] (selecting nothing
// below x is optimal) and every decision bit below x is "skip".  So the rows
// strictly below x can be removed from the sweep: row x then sees D[next(x)]
// as its row i+1, which is the same values, and no kept row's value or bit
// changes.  With `cnt` the prefix counts of positive profits in preorder, x
// has a positive strict descendant iff cnt[next(x)] - cnt[x + 1] > 0, and row
// i is kept iff it is a root or its parent has one.  A kept row i that is
// itself an identity (p_i <= 0 and no positive strict descendant: D[i] =
// D[next(i)], all bits "skip") is dropped as well (for the one-CTA kernel,
// which follows the host's stack plan, only if it has no stack operation).
// Kept rows are listed in sweep order (decreasing i); every position records
// the first kept row at or after it in preorder, so a skip to a dropped row
// lands where the all-"skip" walk through it would.
// ===========================================================================
__device__ __forceinline__ int block_exclusive_scan(int v, int *total, int *sh)
{
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(kFull, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) sh[wid] = x;
    __syncthreads();
    if (wid == 0) {
        int w = lane < nw ? sh[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(kFull, w, o);
            if (lane >= o) w += y;
        }
        if (lane < nw) sh[lane] = w;           // inclusive warp totals
    }
    __syncthreads();
    const int before = wid > 0 ? sh[wid - 1] : 0;
    *total = sh[nw - 1];
    __syncthreads();                           // sh is reused by the next scan
    return before + x - v;
}

// Exclusive scan over the CTAs of the cluster of one value per CTA (`v`, the
// same in every thread of the CTA).  Returns this CTA's offset and the cluster
// total.  The cluster barriers also order the global writes made before the
// call against the reads of other CTAs after it.
__device__ __forceinline__ int ld_dsmem_s32(uint32_t addr)
{
    int v;
    asm volatile("ld.shared::cluster.s32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
    return v;
}
__device__ int cluster_exclusive_scan(int v, int *total, int *slot, int *bcast)
{
    const int CLn = (int)cluster_nctarank(), cr = (int)cluster_ctarank();
    if (threadIdx.x == 0) *slot = v;
    cluster_sync_all();
    if (threadIdx.x == 0) {
        int ex = 0, tot = 0;
        for (int c = 0; c < CLn; ++c) {
            const int x = ld_dsmem_s32(map_to_rank(smem_addr(slot), (uint32_t)c));
            ex += c < cr ? x : 0;
            tot += x;
        }
        bcast[0] = ex;
        bcast[1] = tot;
    }
    cluster_sync_all();           // every slot read: they may be written again
    *total = bcast[1];
    return bcast[0];
}

// One cluster of CL CTAs per item: every pass splits its index range into CL
// contiguous slices, each CTA walks its slice in tiles of T*V elements (V per
// thread, one block scan per tile), and the slices are joined by a scan over
// the cluster's CTAs.
template <bool BYNODE>
__global__ void __launch_bounds__(1024)
k_prune(int32_t n, const int64_t *__restrict__ profit, const int32_t *__restrict__ order,
        const int32_t *__restrict__ next, const int2 *__restrict__ pspan,
        const int32_t *__restrict__ wpre, const int32_t *__restrict__ wmeta,
        const int32_t *__restrict__ item_active, DpWork w, int prune, int wave, int stack_depth,
        int32_t *__restrict__ status, unsigned long long *__restrict__ rows_kept)
{
    constexpr int V = 4;
    __shared__ int sh[32];
    __shared__ int slot, bcast[2];
    const int CL = (int)cluster_nctarank(), cr = (int)cluster_ctarank();
    const int item = blockIdx.x / CL;
    if (item_active && !item_active[item]) return;       // uniform over the cluster
    const int64_t *Pp = profit + (size_t)item * n;
    int32_t *cnt = w.cnt + (size_t)item * (n + 1);
    int32_t *rl = w.rowlist + (size_t)item * n;
    int32_t *kx = w.kidx + (size_t)item * n;
    const int T = blockDim.x, t = threadIdx.x, tile = T * V;
    auto pval = [&](int i) { return Pp[BYNODE ? order[i] : i]; };
    auto slice = [&](int len, int &lo, int &hi) {
        const int per = (len + CL - 1) / CL;
        lo = min(len, cr * per);
        hi = min(len, lo + per);
    };
    int lo, hi, total;

    // prefix counts of positive profits, preorder
    slice(n, lo, hi);
    int mine = 0;
    for (int i = lo + t; i < hi; i += T) mine += pval(i) > 0;
    block_exclusive_scan(mine, &total, sh);
    int carry = cluster_exclusive_scan(total, &total, &slot, bcast);
    const int npos = total;
    for (int base = lo; base < hi; base += tile) {
        int f[V], c = 0;
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int i = base + t * V + v;
            f[v] = i < hi && pval(i) > 0;
            c += f[v];
        }
        int tt;
        int ex = block_exclusive_scan(c, &tt, sh) + carry;
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int i = base + t * V + v;
            if (i < hi) {
                cnt[i] = ex;
                ex += f[v];
            }
        }
        carry += tt;
    }
    if (cr == 0 && t == 0) cnt[n] = npos;
    cluster_sync_all();                                   // cnt complete for every CTA

    // kept rows in sweep order r = n - 1 - i, their kept index, their total weight
    auto keep = [&](int r) -> bool {
        if (!prune) return true;
        const int i = n - 1 - r;
        const int2 sp = pspan[i];
        if (!(sp.x < 0 || cnt[sp.y] - cnt[sp.x] > 0)) return false;
        // an identity row (p <= 0 and no positive strict descendant, so D[i] =
        // D[next(i)] and every bit is "skip") is dropped too: a skip to it
        // lands on the first kept row after it, which holds the same values.
        // The one-CTA kernel reads the host's stack plan and keeps the ones
        // with a stack operation; the wavefront kernel's plan is rebuilt below
        const bool ident = cnt[next[i]] - cnt[i + 1] == 0 && pval(i) <= 0;
        return !(ident && (wave || (wmeta[i] & kWaveStackOps) == 0));
    };
    slice(n, lo, hi);
    int kmine = 0;
    for (int r = lo + t; r < hi; r += T) kmine += keep(r);
    block_exclusive_scan(kmine, &total, sh);
    int kcarry = cluster_exclusive_scan(total, &total, &slot, bcast);
    const int nk = total;
    for (int base = lo; base < hi; base += tile) {
        bool kp[V];
        int kc = 0;
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int r = base + t * V + v;
            kp[v] = r < hi && keep(r);
            kc += kp[v];
        }
        int tt;
        int ex = block_exclusive_scan(kc, &tt, sh) + kcarry;
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int r = base + t * V + v;
            if (r < hi) {
                const int i = n - 1 - r;
                if (kp[v]) {
                    rl[ex] = i;
                    kx[i] = ex++;
                } else {
                    kx[i] = ex - 1;         // the first kept row at or after position i (-1: none)
                }
            }
        }
        kcarry += tt;
    }
    if (cr == 0 && t == 0) {
        w.nkept[item] = nk;
        if (rows_kept) atomicAdd(rows_kept, (unsigned long long)nk);
    }
    cluster_sync_all();                                   // rl and kx complete

    // per kept row: skip target, the DP's row stream (profit, metadata) and
    // the suffix weights of the traceback
    int32_t *sk = w.skip + (size_t)item * n;
    int32_t *ws = w.wsuf + (size_t)item * (n + 1);
    int64_t *rp = w.rowp + (size_t)item * n;
    int32_t *rm = w.rowm + (size_t)item * n;
    slice(nk, lo, hi);
    int wmine = 0;
    for (int q = lo + t; q < hi; q += T) wmine += wpre[rl[q]];
    block_exclusive_scan(wmine, &total, sh);
    int wtot;                                             // weight of all kept rows
    int wcarry = cluster_exclusive_scan(total, &wtot, &slot, bcast);
    for (int base = lo; base < hi; base += tile) {
        int wq[V], wl = 0;
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int q = base + t * V + v;
            wq[v] = 0;
            if (q < hi) {
                const int i = rl[q];
                const int nx = next[i];
                sk[q] = nx < n ? kx[nx] : -1;
                wq[v] = wpre[i];
                rp[q] = pval(i);
                rm[q] = wmeta[i];               // the wavefront kernel's is rebuilt below
                if (wave) cnt[q] = -1;          // cnt (done with) becomes last_top_reader
            }
            wl += wq[v];
        }
        int tt;
        int ex = block_exclusive_scan(wl, &tt, sh) + wcarry;   // weight of kept rows before q
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int q = base + t * V + v;
            if (q < hi) {
                ws[q] = wtot - ex;                                 // weight of kept rows q..nk-1
                ex += wq[v];
            }
        }
        wcarry += tt;
    }
    if (cr == 0 && t == 0) ws[nk] = 0;
    if (!wave) return;

    // Skip-row stack plan of the wavefront kernel over the kept rows (the
    // host's plan is for the whole tree; after pruning many of its pushes
    // have no reader left).  Kept row q reads row sk[q]: the row just
    // computed when sk[q] = q - 1, else the stack top (the zero row when the
    // stack is empty, which is the case whenever sk[q] = -1).  A row read
    // through the stack is pushed when computed and popped after its last
    // such reader; the rows pushed in between are popped before it, so
    // every read is of the top.
    int32_t *lr_ = cnt;                                   // last_top_reader[target]
    cluster_sync_all();                                   // sk and the -1s complete
    for (int q = lo + t; q < hi; q += T) {
        const int s = sk[q];
        if (s >= 0 && s != q - 1) atomicMax(lr_ + s, q);
    }
    cluster_sync_all();                                   // last readers complete
    auto delta = [&](int q, bool &pop, bool &push) {
        const int s = sk[q];
        pop = s >= 0 && s != q - 1 && lr_[s] == q;
        push = lr_[q] >= 0;
        return (int)push - (int)pop;
    };
    int dmine = 0;
    for (int q = lo + t; q < hi; q += T) {
        bool a, b;
        dmine += delta(q, a, b);
    }
    block_exclusive_scan(dmine, &total, sh);
    int dcarry = cluster_exclusive_scan(total, &total, &slot, bcast);
    for (int base = lo; base < hi; base += tile) {
        int dq[V], dl = 0;
        bool pq[V], uq[V];
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int q = base + t * V + v;
            dq[v] = 0;
            pq[v] = uq[v] = false;
            if (q < hi) dq[v] = delta(q, pq[v], uq[v]);
            dl += dq[v];
        }
        int tt;
        int ex = block_exclusive_scan(dl, &tt, sh) + dcarry;   // stack depth before row q
#pragma unroll
        for (int v = 0; v < V; ++v) {
            const int q = base + t * V + v;
            if (q < hi) {
                const int s = sk[q];
                const int d = ex - (int)pq[v];            // after the pop
                int flags = 0, lvl = 0;
                if (uq[v]) {
                    flags = kWavePush;
                    lvl = d;
                } else if (pq[v] && d > 0) {
                    flags = kWaveReload;                  // the level below becomes the top
                    lvl = d - 1;
                } else if (pq[v]) {
                    flags = kWaveZeroTop;                 // the stack emptied: top = zero row
                }
                if ((flags & (kWavePush | kWaveReload)) && lvl >= stack_depth) {
                    // cannot happen (the plan of an ancestor-closed sub-forest is
                    // never deeper than the whole tree's): report, stay in bounds
                    atomicExch(status, (int32_t)PP_EBOUNDS);
                    flags = 0;
                    lvl = 0;
                }
                const int wq = wpre[rl[q]];
                // a row whose skip row is the row just computed reads it from the
                // stack top when that row was pushed (the push made it the top):
                // the same values, and sub-blocks without "cur" rows need no
                // per-row choice of skip source
                const bool cur = s >= 0 && s == q - 1 && lr_[q - 1] < 0;
                rm[q] = wave_pack(wq > 8 ? 8 : wq, cur ? kWaveCur : kWaveTop, flags, lvl);
                ex += dq[v];
            }
        }
        dcarry += tt;
    }
}

static size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

size_t dp_work_bytes(int batch, int n, int words)
{
    const size_t nb = (size_t)(n + 63) / 64 * 64, B = (size_t)std::max(batch, 1), N = (size_t)std::max(n, 1);
    return align256(B * nb * words * 4) + 4 * align256(B * N * 4) + 2 * align256(B * (N + 1) * 4) +
           align256(B * 4) + align256(B * N * 8);
}

DpWork dp_work_split(void *base, int batch, int n, int words)
{
    const size_t nb = (size_t)(n + 63) / 64 * 64, B = (size_t)std::max(batch, 1), N = (size_t)std::max(n, 1);
    char *p = reinterpret_cast<char *>(base);
    DpWork w;
    w.bits = reinterpret_cast<uint32_t *>(p);
    p += align256(B * nb * words * 4);
    w.rowlist = reinterpret_cast<int32_t *>(p);
    p += align256(B * N * 4);
    w.kidx = reinterpret_cast<int32_t *>(p);
    p += align256(B * N * 4);
    w.cnt = reinterpret_cast<int32_t *>(p);
    p += align256(B * (N + 1) * 4);
    w.nkept = reinterpret_cast<int32_t *>(p);
    p += align256(B * 4);
    w.skip = reinterpret_cast<int32_t *>(p);
    p += align256(B * N * 4);
    w.wsuf = reinterpret_cast<int32_t *>(p);
    p += align256(B * (N + 1) * 4);
    w.rowp = reinterpret_cast<int64_t *>(p);
    p += align256(B * N * 8);
    w.rowm = reinterpret_cast<int32_t *>(p);
    return w;
}

DpWork dp_work_item(const DpWork &w, int item, int n, int words)
{
    const size_t nb = (size_t)(n + 63) / 64 * 64, N = (size_t)std::max(n, 1), it = (size_t)item;
    DpWork o;
    o.bits = w.bits + it * nb * words;
    o.rowlist = w.rowlist + it * N;
    o.kidx = w.kidx + it * N;
    o.cnt = w.cnt + it * (N + 1);
    o.nkept = w.nkept + it;
    o.skip = w.skip + it * N;
    o.wsuf = w.wsuf + it * (N + 1);
    o.rowp = w.rowp + it * N;
    o.rowm = w.rowm + it * N;
    return o;
}

// ===========================================================================
// geometry and launch
// ===========================================================================
template <int C, int WMAX>
static const void *wave_kernel(bool spill)
{
    return spill ? (const void *)k_tree_dp_wave<C, WMAX, true> : (const void *)k_tree_dp_wave<C, WMAX, false>;
}

// spill: some skip-row stack levels live in global memory (the kernel without
// that branch is ~5% faster per row)
static const void *wave_kernel_for(int C, int WMAX, bool spill)
{
#define PP_WAVE_CASE(CC, WW) if (C == CC && WMAX == WW) return wave_kernel<CC, WW>(spill);
    PP_WAVE_CASE(1, 1) PP_WAVE_CASE(2, 1) PP_WAVE_CASE(4, 1) PP_WAVE_CASE(8, 1)
    PP_WAVE_CASE(2, 2) PP_WAVE_CASE(4, 2) PP_WAVE_CASE(8, 2)
    PP_WAVE_CASE(4, 4) PP_WAVE_CASE(8, 4)
#undef PP_WAVE_CASE
    return nullptr;
}

static int max_smem_optin(const pp_instance *inst)
{
    int v = 0;
    cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, inst->device);
    return v;
}

// Split launch: measured on GB300 (152 SMs), the placement of clusters of 8
// CTAs at one CTA per SM finds room for 15 of them; a 16th cluster then shares
// SMs with other items and slows them and itself by ~25% per row.  When the
// batch exceeds that count by at most 2, the extra items (the smallest
// sweeps, by rank in the kernel) run as clusters of CL / 2 CTAs on the SMs
// that are left, in a second launch on its own stream.
static void split_geometry(const pp_instance *inst, int batch, const void *fn, const cudaLaunchConfig_t &cfg0,
                           int smem_max, DpGeom *g)
{
    if (inst->tune_cl > 0 || inst->tune_c > 0 || batch < 2 || batch > 32 || g->CL < 2 || (g->CL & 1) || 2 * g->WPC > 16)
        return;
    int per_sm = 0;
    cudaDeviceGetAttribute(&per_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, inst->device);
    const size_t excl = std::max(g->smem, (size_t)per_sm / 2);   // two CTAs never fit in one SM
    if (excl > (size_t)smem_max) return;
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)excl) != cudaSuccess) {
        cudaGetLastError();
        return;
    }
    cudaLaunchConfig_t cfg = cfg0;
    cfg.dynamicSmemBytes = excl;
    int m1 = 0;
    if (cudaOccupancyMaxActiveClusters(&m1, fn, &cfg) != cudaSuccess) {
        cudaGetLastError();
        return;
    }
    if (m1 < 1 || batch <= m1 || batch - m1 > 2) return;
    const int CL2 = g->CL / 2, WPC2 = 2 * g->WPC;
    const size_t fixed2 = wave_fixed_bytes(WPC2, g->WMAX);
    const size_t level2 = (size_t)g->C * WPC2 * 32 * sizeof(int64_t);
    if (fixed2 > (size_t)smem_max) return;
    const int L2 = (int)std::min<size_t>((size_t)inst->stack_depth, ((size_t)smem_max - fixed2) / level2);
    const size_t smem2 = std::max(fixed2 + (size_t)L2 * level2, excl);
    const void *fn2 = wave_kernel_for(g->C, g->WMAX, L2 < inst->stack_depth);
    if (!fn2 || cudaFuncSetAttribute(fn2, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem2) != cudaSuccess) {
        cudaGetLastError();
        return;
    }
    cudaLaunchConfig_t cfg2 = cfg0;
    cfg2.gridDim = dim3(CL2 * (batch - m1));
    cfg2.blockDim = dim3(WPC2 * 32);
    cfg2.dynamicSmemBytes = smem2;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CL2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg2.attrs = attr;
    cfg2.numAttrs = 1;
    int m2 = 0;
    if (cudaOccupancyMaxActiveClusters(&m2, fn2, &cfg2) != cudaSuccess) {
        cudaGetLastError();
        return;
    }
    if (m2 < batch - m1) return;
    g->split = m1;
    g->smem_x = excl;
    g->CL2 = CL2;
    g->WPC2 = WPC2;
    g->L_smem2 = L2;
    g->smem2 = smem2;
}

static bool wave_geometry(const pp_instance *inst, int64_t k, int batch, DpGeom *g)
{
    const int WMAX = inst->max_weight <= 1 ? 1 : (inst->max_weight <= 2 ? 2 : 4);
    const int smem_max = max_smem_optin(inst);
    int per_item = inst->sm_count / std::max(batch, 1);
    per_item = std::max(1, std::min(8, per_item));
    int cl_hi = per_item;
    if (inst->tune_cl > 0) cl_hi = std::min(inst->tune_cl, 8);
    // Shape chosen by timing whole plans of the paper-scale workload at budgets
    // 128 to 4,096: 2 columns per thread (1 and 4 were slower) unless that
    // needs more than 32 warps per DP, then 4; a budget of at most 128 columns
    // on a single warp (no hand-off at all); the warps spread over the widest
    // cluster the SMs per item allow, so that a CTA holds at most 4 warps
    // while the DP has at most 32 (with 1 or 2 warps per CTA most hand-offs
    // cross CTAs, which cost more).  A batch just above the number of such
    // clusters that fit at one CTA per SM is split (split_geometry).
    int C = WMAX;
    bool one_warp = false;
    if (inst->tune_c > 0) {
        C = std::max(std::min(inst->tune_c, 8), WMAX);
    } else if (k <= 128) {
        while (32 * C < k) C *= 2;
        one_warp = inst->tune_cl <= 0;
    } else {
        C = std::max(WMAX, 2);
        if ((k + 32 * C - 1) / (32 * C) > 32 && C < 4) C = 4;
        if ((k + 32 * C - 1) / (32 * C) > 128) C = 8;
    }
    const int64_t P = (k + 32 * C - 1) / (32 * C);     // warps per DP
    if (inst->tune_cl <= 0) cl_hi = (int)std::min<int64_t>(one_warp ? 1 : cl_hi, P);
    for (int CL = cl_hi; CL >= 1; --CL) {
        const int WPC = (int)((P + CL - 1) / CL);
        if (WPC > 16) continue;
        const size_t fixed = wave_fixed_bytes(WPC, WMAX);
        const size_t level = (size_t)C * WPC * 32 * sizeof(int64_t);
        if (fixed > (size_t)smem_max) continue;
        const int L_smem = (int)std::min<size_t>((size_t)inst->stack_depth, ((size_t)smem_max - fixed) / level);
        const void *fn = wave_kernel_for(C, WMAX, L_smem < inst->stack_depth);
        if (!fn) continue;
        const size_t smem = fixed + (size_t)L_smem * level;
        if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess) {
            cudaGetLastError();
            continue;
        }
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(CL * std::max(batch, 1));
        cfg.blockDim = dim3(WPC * 32);
        cfg.dynamicSmemBytes = smem;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = CL;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int clusters = 0;
        if (cudaOccupancyMaxActiveClusters(&clusters, fn, &cfg) != cudaSuccess) {
            cudaGetLastError();
            clusters = 0;
        }
        if (clusters < 1) continue;
        if (clusters < batch && CL > 1) continue;       // prefer fewer SMs per DP to a second wave
        g->wave = 1;
        g->CL = CL;
        g->WPC = WPC;
        g->C = C;
        g->WMAX = WMAX;
        g->P = CL * WPC;
        g->T = g->P * 32;
        g->kpad = g->T * C;
        g->words = g->kpad / 32;
        g->L_smem = L_smem;
        g->smem = smem;
        g->split = 0;
        split_geometry(inst, batch, fn, cfg, smem_max, g);
        return true;
    }
    return false;
}

bool dp_geometry(const pp_instance *inst, int32_t max_budget, DpGeom *g, int batch)
{
    if (max_budget < 0) return false;
    int64_t k = max_budget;
    if (k > inst->total_weight) k = inst->total_weight;   // larger budgets change nothing
    if (k < 1) k = 1;
    if (inst->max_weight <= 4 && inst->n > 0 && !inst->tune_flat && wave_geometry(inst, k, batch, g)) return true;
    int C = 1;
    while ((int64_t)C * 1024 < k) C *= 2;
    if (C > 32) return false;
    int T = (int)((k + C - 1) / C);
    T = (T + 31) / 32 * 32;
    if (T < 32) T = 32;
    g->wave = 0;
    g->CL = 1;
    g->C = C;
    g->T = T;
    g->P = T / 32;
    g->WPC = g->P;
    g->kpad = T * C;
    g->words = g->kpad / 32;
    const size_t fixed = flat_smem_fixed(g->kpad);
    const size_t row_bytes = (size_t)g->kpad * sizeof(int64_t);
    const int smem_max = inst->n > 0 ? max_smem_optin(inst) : 0;
    if (inst->n > 0 && fixed > (size_t)smem_max) return false;
    g->L_smem = inst->n > 0 ? (int)std::min<size_t>((size_t)inst->stack_depth, ((size_t)smem_max - fixed) / row_bytes) : 0;
    g->smem = fixed + (size_t)g->L_smem * row_bytes;
    return true;
}

static pp_status ensure_split_streams(pp_instance *inst)
{
    if (inst->split_hi) return PP_OK;
    int least = 0, greatest = 0;
    PP_CUDA(cudaDeviceGetStreamPriorityRange(&least, &greatest));
    PP_CUDA(cudaStreamCreateWithPriority(&inst->split_hi, cudaStreamNonBlocking, greatest));
    PP_CUDA(cudaStreamCreateWithPriority(&inst->split_lo, cudaStreamNonBlocking, least));
    PP_CUDA(cudaEventCreateWithFlags(&inst->split_fork, cudaEventDisableTiming));
    PP_CUDA(cudaEventCreateWithFlags(&inst->split_join_hi, cudaEventDisableTiming));
    PP_CUDA(cudaEventCreateWithFlags(&inst->split_join_lo, cudaEventDisableTiming));
    return PP_OK;
}

template <int C>
static pp_status launch_flat_c(pp_instance *inst, int batch, const int64_t *profit, bool by_node,
                               const int32_t *item_budget, int32_t max_budget,
                               const int32_t *item_active, const DpGeom &g, int64_t *best,
                               const DpWork &work, int64_t *gstack, int L_glob, cudaStream_t st)
{
    uint32_t *bits = work.bits;
    PP_CUDA(cudaFuncSetAttribute(k_tree_dp_flat<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)g.smem));
    k_tree_dp_flat<C><<<batch, g.T, g.smem, st>>>(inst->n, work.rowlist, work.nkept, profit,
                                                   by_node ? inst->d_order : nullptr,
                                                   inst->d_wpre, inst->d_meta, item_budget, max_budget,
                                                   item_active, best, bits, gstack, g.L_smem, L_glob,
                                                   inst->d_status);
    PP_CUDA(cudaGetLastError());
    return PP_OK;
}

// Launch the DP kernel selected by the geometry with the skip-row stack levels
// below L_smem kept in `gstack` (batch * L_glob * kpad int64, may be null when
// L_glob == 0).
static pp_status launch_dp_kernels(pp_instance *inst, int batch, const int64_t *profit, bool by_node,
                                   const int32_t *item_budget, const int32_t *item_active,
                                   const DpGeom &g, int64_t *best, const DpWork &work, cudaStream_t st,
                                   int32_t max_budget, int64_t *gstack, int L_glob,
                                   unsigned long long *rows_kept)
{
    // the pruned sweep of every item, then the DP over its kept rows
    {
        cudaLaunchConfig_t pc = {};
        pc.gridDim = dim3(kPruneCluster * batch);
        pc.blockDim = dim3(1024);
        pc.stream = st;
        cudaLaunchAttribute pa[1];
        pa[0].id = cudaLaunchAttributeClusterDimension;
        pa[0].val.clusterDim.x = kPruneCluster;
        pa[0].val.clusterDim.y = 1;
        pa[0].val.clusterDim.z = 1;
        pc.attrs = pa;
        pc.numAttrs = 1;
        const int32_t *ord = inst->d_order, *nxt = inst->d_next, *wp = inst->d_wpre, *wm = inst->d_wave;
        const int2 *psp = inst->d_pspan;
        const int pr = !inst->tune_noprune, wv = g.wave, sd = inst->stack_depth;
        int32_t *stt = inst->d_status;
        if (by_node)
            PP_CUDA(cudaLaunchKernelEx(&pc, k_prune<true>, inst->n, profit, ord, nxt, psp, wp, wm, item_active,
                                       work, pr, wv, sd, stt, rows_kept));
        else
            PP_CUDA(cudaLaunchKernelEx(&pc, k_prune<false>, inst->n, profit, ord, nxt, psp, wp, wm, item_active,
                                       work, pr, wv, sd, stt, rows_kept));
    }
    PP_CUDA(cudaGetLastError());
    uint32_t *bits = work.bits;
    const int32_t *nkept = work.nkept;
    if (g.wave) {
        int32_t n = inst->n;
        int32_t nblk = (n + 63) / 64 * 2;                    // 32-row blocks, in pairs
        const int64_t *rowp = work.rowp;
        const int32_t *rowm = work.rowm;
        int32_t *status = inst->d_status;
        int32_t nb = batch;
        auto launch = [&](int CL, int WPC, size_t smem, int32_t L_smem, int items, int32_t slot_base,
                          cudaStream_t s) -> pp_status {
            const void *fn = wave_kernel_for(g.C, g.WMAX, L_smem < inst->stack_depth);
            if (!fn) return fail(PP_EINVAL, "unsupported DP geometry");
            PP_CUDA(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3(CL * items);
            cfg.blockDim = dim3(WPC * 32);
            cfg.dynamicSmemBytes = smem;
            cfg.stream = s;
            cudaLaunchAttribute attr[1];
            attr[0].id = cudaLaunchAttributeClusterDimension;
            attr[0].val.clusterDim.x = CL;
            attr[0].val.clusterDim.y = 1;
            attr[0].val.clusterDim.z = 1;
            cfg.attrs = attr;
            cfg.numAttrs = 1;
            int32_t Lg = L_glob, ranked = g.split > 0;
            void *args[] = {&n, &nblk, (void *)&rowp, (void *)&rowm, (void *)&nkept, (void *)&item_budget,
                            &max_budget, (void *)&item_active, &best, &bits, &gstack, &L_smem, &Lg, &status,
                            &nb, &slot_base, &ranked};
            PP_CUDA(cudaLaunchKernelExC(&cfg, fn, args));
            return PP_OK;
        };
        if (!g.split) return launch(g.CL, g.WPC, g.smem, g.L_smem, batch, 0, st);
        pp_status s;
        if ((s = ensure_split_streams(inst))) return s;
        // fork: the wide launch first, on the higher-priority stream, so its
        // clusters are placed before the narrow ones take the SMs left over
        PP_CUDA(cudaEventRecord(inst->split_fork, st));
        PP_CUDA(cudaStreamWaitEvent(inst->split_hi, inst->split_fork, 0));
        PP_CUDA(cudaStreamWaitEvent(inst->split_lo, inst->split_fork, 0));
        if ((s = launch(g.CL, g.WPC, g.smem_x, g.L_smem, g.split, 0, inst->split_hi))) return s;
        if ((s = launch(g.CL2, g.WPC2, g.smem2, g.L_smem2, batch - g.split, g.split, inst->split_lo))) return s;
        PP_CUDA(cudaEventRecord(inst->split_join_hi, inst->split_hi));
        PP_CUDA(cudaEventRecord(inst->split_join_lo, inst->split_lo));
        PP_CUDA(cudaStreamWaitEvent(st, inst->split_join_hi, 0));
        PP_CUDA(cudaStreamWaitEvent(st, inst->split_join_lo, 0));
        return PP_OK;
    }
    switch (g.C) {
    case 1: return launch_flat_c<1>(inst, batch, profit, by_node, item_budget, max_budget, item_active, g, best, work, gstack, L_glob, st);
    case 2: return launch_flat_c<2>(inst, batch, profit, by_node, item_budget, max_budget, item_active, g, best, work, gstack, L_glob, st);
    case 4: return launch_flat_c<4>(inst, batch, profit, by_node, item_budget, max_budget, item_active, g, best, work, gstack, L_glob, st);
    case 8: return launch_flat_c<8>(inst, batch, profit, by_node, item_budget, max_budget, item_active, g, best, work, gstack, L_glob, st);
    case 16: return launch_flat_c<16>(inst, batch, profit, by_node, item_budget, max_budget, item_active, g, best, work, gstack, L_glob, st);
    case 32: return launch_flat_c<32>(inst, batch, profit, by_node, item_budget, max_budget, item_active, g, best, work, gstack, L_glob, st);
    default: return fail(PP_EINVAL, "unsupported DP geometry");
    }
}

// Skip-row stack levels below shared memory, per item (the larger need of the
// two launches of a split).
static int dp_global_levels(const pp_instance *inst, const DpGeom &g)
{
    return std::max(0, inst->stack_depth - (g.split ? std::min(g.L_smem, g.L_smem2) : g.L_smem));
}

pp_status ensure_dp_stack(pp_instance *inst, const DpGeom &g, int items)
{
    const int L_glob = dp_global_levels(inst, g);
    if (L_glob <= 0) return PP_OK;
    return ensure_scratch(inst->stack, (size_t)items * L_glob * (size_t)g.kpad * sizeof(int64_t));
}

pp_status launch_tree_dp(pp_instance *inst, int batch, const int64_t *profit, bool by_node,
                         const int32_t *item_budget, const int32_t *item_active, const DpGeom &g,
                         int64_t *best, const DpWork &work, cudaStream_t st, int32_t max_budget,
                         unsigned long long *rows_kept, int stack_item)
{
    if (batch <= 0) return PP_OK;
    if (inst->n == 0) {
        PP_CUDA(cudaMemsetAsync(best, 0, sizeof(int64_t) * batch, st));
        return PP_OK;
    }
    const int L_glob = dp_global_levels(inst, g);
    pp_status s = ensure_dp_stack(inst, g, stack_item + batch);
    if (s != PP_OK) return s;
    int64_t *gstack = reinterpret_cast<int64_t *>(inst->stack.ptr);
    if (gstack && L_glob > 0) gstack += (size_t)stack_item * L_glob * (size_t)g.kpad;
    return launch_dp_kernels(inst, batch, profit, by_node, item_budget, item_active, g, best, work, st,
                             max_budget, gstack, L_glob, rows_kept);
}

}  // namespace pp

using namespace pp;

extern "C" size_t pp_dp_bits_size(const pp_instance *inst, int32_t batch, int32_t max_budget)
{
    DpGeom g;
    if (!inst || batch <= 0 || !dp_geometry(inst, max_budget, &g, batch)) return 0;
    return dp_work_bytes(batch, inst->n, g.words);
}

extern "C" pp_status pp_tree_dp(pp_instance *inst, int32_t batch, const int64_t *profit,
                                const int32_t *budget, int32_t max_budget, int64_t *best,
                                uint32_t *bits, void *stream)
{
    if (!inst) return fail(PP_EINVAL, "null instance");
    if (batch < 0) return fail(PP_EINVAL, "batch must be >= 0");
    DpGeom g;
    if (!dp_geometry(inst, max_budget, &g, std::max(batch, 1))) return fail(PP_EINVAL, "max_budget out of range");
    if (batch == 0) return PP_OK;
    if (!budget || !best || (inst->n > 0 && (!profit || !bits)))
        return fail(PP_EINVAL, "null device pointer");
    return launch_tree_dp(inst, batch, profit, true, budget, nullptr, g, best,
                          dp_work_split(bits, batch, inst->n, g.words), (cudaStream_t)stream, max_budget);
}

extern "C" pp_status pp_test_inject(int32_t kind, int32_t value)
{
    if (kind != 1) return fail(PP_EINVAL, "unknown injection kind");
    PP_CUDA(cudaMemcpyToSymbol(g_drop_publish_warp, &value, sizeof(value)));
    return PP_OK;
}

extern "C" pp_status pp_tune_dp(pp_instance *inst, int32_t cluster_ctas, int32_t columns_per_thread,
                                int32_t force_flat, int32_t no_prune)
{
    if (!inst) return fail(PP_EINVAL, "null instance");
    if (cluster_ctas < 0 || cluster_ctas > 8 || columns_per_thread < 0 || columns_per_thread > 16 ||
        (columns_per_thread & (columns_per_thread - 1)) != 0)
        return fail(PP_EINVAL, "cluster_ctas must be 0..8 and columns_per_thread 0 or a power of two <= 16");
    inst->tune_cl = cluster_ctas;
    inst->tune_c = columns_per_thread;
    inst->tune_flat = force_flat != 0;
    inst->tune_noprune = no_prune != 0;
    return PP_OK;
}

extern "C" pp_status pp_dp_geometry(const pp_instance *inst, int32_t batch, int32_t max_budget,
                                    int32_t *out)
{
    if (!inst || !out) return fail(PP_EINVAL, "null pointer");
    DpGeom g;
    if (!dp_geometry(inst, max_budget, &g, std::max(batch, 1))) return fail(PP_EINVAL, "max_budget out of range");
    out[0] = g.wave;
    out[1] = g.CL;
    out[2] = g.WPC;
    out[3] = g.C;
    out[4] = g.P;
    out[5] = g.L_smem;
    out[6] = (int32_t)g.smem;
    out[7] = g.kpad;
    return PP_OK;
}

extern "C" pp_status pp_dp_split(const pp_instance *inst, int32_t batch, int32_t max_budget, int32_t *out)
{
    if (!inst || !out) return fail(PP_EINVAL, "null pointer");
    DpGeom g;
    if (!dp_geometry(inst, max_budget, &g, std::max(batch, 1))) return fail(PP_EINVAL, "max_budget out of range");
    out[0] = g.split;
    out[1] = g.split ? g.CL2 : 0;
    out[2] = g.split ? g.WPC2 : 0;
    out[3] = g.split ? g.L_smem2 : 0;
    out[4] = g.split ? (int32_t)g.smem_x : 0;
    return PP_OK;
}

// ===========================================================================
// pp_tree_dp_noalloc: the same DP launch with the skip-row stack levels that do
// not fit in shared memory kept in a fixed array of this library's device
// memory instead of instance scratch, so the call never allocates.
// ===========================================================================
namespace pp {

constexpr size_t kStaticStackBytes = (size_t)16 << 20;   // per device, held until the process exits
static __device__ __align__(256) int64_t g_static_stack[kStaticStackBytes / sizeof(int64_t)];

constexpr int kMaxDevices = 64;
static std::mutex g_static_stack_mu;
static int64_t *g_static_stack_addr[kMaxDevices] = {};

// Device address of g_static_stack on `device`, resolved on first use with
// that device current (host code cannot use the symbol itself as a pointer).
static pp_status static_stack_address(int device, int64_t **out)
{
    if (device < 0 || device >= kMaxDevices) return fail(PP_EINVAL, "device ordinal out of range");
    std::lock_guard<std::mutex> lock(g_static_stack_mu);
    if (!g_static_stack_addr[device]) {
        void *ptr = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&ptr, g_static_stack);
        if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(fixed DP stack scratch)");
        g_static_stack_addr[device] = reinterpret_cast<int64_t *>(ptr);
    }
    *out = g_static_stack_addr[device];
    return PP_OK;
}

}  // namespace pp

extern "C" pp_status pp_tree_dp_noalloc(pp_instance *inst, int32_t batch, const int64_t *profit,
                                        const int32_t *budget, int32_t max_budget, int64_t *best,
                                        uint32_t *bits, void *stream)
{
    if (!inst) return fail(PP_EINVAL, "null instance");
    if (batch < 0) return fail(PP_EINVAL, "batch must be >= 0");
    int cur_dev = -1;
    PP_CUDA(cudaGetDevice(&cur_dev));
    if (cur_dev != inst->device) return fail(PP_EINVAL, "the instance's device must be the current device");
    int64_t *scratch = nullptr;
    pp_status s = static_stack_address(cur_dev, &scratch);     // one-time set-up per device
    if (s != PP_OK) return s;
    DpGeom g;
    if (!dp_geometry(inst, max_budget, &g, std::max(batch, 1))) return fail(PP_EINVAL, "max_budget out of range");
    if (batch == 0) return PP_OK;
    if (!budget || !best || (inst->n > 0 && (!profit || !bits)))
        return fail(PP_EINVAL, "null device pointer");
    cudaStream_t st = (cudaStream_t)stream;
    if (inst->n == 0) {
        PP_CUDA(cudaMemsetAsync(best, 0, sizeof(int64_t) * batch, st));
        return PP_OK;
    }
    g.split = 0;                        // one launch: no internal streams or events
    const int L_glob = dp_global_levels(inst, g);
    const size_t need = (size_t)batch * (size_t)L_glob * (size_t)g.kpad * sizeof(int64_t);
    if (need > kStaticStackBytes)
        return fail(PP_EINVAL, "pp_tree_dp_noalloc: this launch needs " + std::to_string(need) +
                                   " bytes of skip-row stack scratch, more than its fixed " +
                                   std::to_string(kStaticStackBytes) +
                                   " bytes; use a smaller batch or pp_tree_dp");
    return launch_dp_kernels(inst, batch, profit, true, budget, nullptr, g, best,
                             dp_work_split(bits, batch, inst->n, g.words), st, max_budget, scratch, L_glob,
                             nullptr);
}

extern "C" pp_status pp_dp_stack_bytes(const pp_instance *inst, size_t *out)
{
    if (!inst || !out) return fail(PP_EINVAL, "null pointer");
    *out = inst->stack.ptr ? inst->stack.bytes : 0;
    return PP_OK;
}

extern "C" pp_status pp_dp_rows_swept(const pp_instance *inst, int32_t batch, int32_t max_budget,
                                      const uint32_t *workspace, int32_t *rows, void *stream)
{
    if (!inst || !rows) return fail(PP_EINVAL, "null pointer");
    if (batch <= 0) return PP_OK;
    DpGeom g;
    if (!dp_geometry(inst, max_budget, &g, batch)) return fail(PP_EINVAL, "max_budget out of range");
    if (inst->n == 0) {
        for (int32_t b = 0; b < batch; ++b) rows[b] = 0;
        return PP_OK;
    }
    if (!workspace) return fail(PP_EINVAL, "null workspace");
    const DpWork w = dp_work_split(const_cast<uint32_t *>(workspace), batch, inst->n, g.words);
    PP_CUDA(cudaMemcpyAsync(rows, w.nkept, sizeof(int32_t) * batch, cudaMemcpyDeviceToHost, (cudaStream_t)stream));
    PP_CUDA(cudaStreamSynchronize((cudaStream_t)stream));
    return PP_OK;
}
