// Exact capacity-k prefix-complete tree knapsack (Eq. 9, Theorem 1) and its
// traceback (Algorithm 1, RootedDP).
//
// One CTA sweeps one DP instance.  Rows are preorder positions i = n-1..0;
// the capacity axis is split across the CTA: thread t owns columns
// t*C + c + 1 and keeps its part of row i+1 in registers.  Per row:
//   skip  s_j = D[next(i)][j]: the registers (leaf, next(i) = i+1), zero
//         (next(i) = n) or a saved row of the skip-row stack (shared memory
//         for the top levels, instance scratch in global memory below them);
//   take  t_j = p_i + D[i+1][j - w_i] for j >= w_i: row i+1 is also staged in
//         shared memory (column-major per thread, conflict-free) so that the
//         w_i-column shift can cross thread boundaries;
//   D[i][j] = take ? t_j : s_j with take = (t_j > s_j), so the traceback
//         yields the lexicographically smallest optimal preorder indicator;
//   decision bits: one __ballot_sync per (warp, c) gives a 32-bit word,
//         stored row-major at bits[i][warp*C + c].
// Row metadata (p_i, w_i, skip/push codes) is staged through shared memory in
// blocks of kMetaRows rows, prefetched one block ahead.
#include <algorithm>

#include "pp_internal.cuh"

namespace pp {

constexpr int kMetaRows = 256;

static size_t dp_smem_fixed(const DpGeom &g)
{
    return 2 * (size_t)g.kpad * sizeof(int64_t) + 2 * kMetaRows * (sizeof(int64_t) + 2 * sizeof(int32_t));
}

template <int C>
__global__ void __launch_bounds__(1024, 1)
k_tree_dp(int32_t n, const int64_t *__restrict__ profit, const int32_t *__restrict__ order,
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
    const int item = blockIdx.x;
    const int kpad = T * C;
    const int words = kpad >> 5;

    if (item_active && !item_active[item]) return;
    const int32_t kreq = item_budget[item];
    if (kreq < 0 || kreq > max_budget) {
        if (t == 0) {
            atomicExch(status, (int32_t)PP_EBOUNDS);
            best[item] = 0;
        }
        return;
    }
    const int k = kreq < kpad ? kreq : kpad;   // kpad covers min(max_budget, total weight)

    int64_t *srow = reinterpret_cast<int64_t *>(smem);          // [2][C][T]
    int64_t *sstk = srow + 2 * (size_t)kpad;                    // [L_smem][C][T]
    int64_t *sp = sstk + (size_t)L_smem * kpad;                 // [2][kMetaRows]
    int32_t *sw = reinterpret_cast<int32_t *>(sp + 2 * kMetaRows);
    int32_t *sm = sw + 2 * kMetaRows;
    int64_t *gst = gstack + (size_t)item * L_glob * kpad;
    const int64_t *P = profit + (size_t)item * n;
    uint32_t *B = bits + (size_t)item * n * words;

    int64_t cur[C];                      // D[i+1][t*C + c + 1]
#pragma unroll
    for (int c = 0; c < C; ++c) {
        cur[c] = 0;                      // row n is the zero boundary
        srow[c * T + t] = 0;
    }
    for (int x = t; x < kMetaRows && x < n; x += T) {
        const int i = n - 1 - x;
        sp[x] = P[order ? order[i] : i];
        sw[x] = wpre[i];
        sm[x] = meta[i];
    }
    __syncthreads();

    int64_t nx_p = 0;
    int32_t nx_w = 0, nx_m = 0;
    for (int r = 0; r < n; ++r) {
        const int i = n - 1 - r;
        const int blk = r / kMetaRows, off = r - blk * kMetaRows, buf = (blk & 1) * kMetaRows;
        if (off == 0) {                  // prefetch the next metadata block into registers
            const int x = (blk + 1) * kMetaRows + t;
            if (t < kMetaRows && x < n) {
                const int ii = n - 1 - x;
                nx_p = P[order ? order[ii] : ii];
                nx_w = wpre[ii];
                nx_m = meta[ii];
            }
        }
        const int64_t p = sp[buf + off];
        const int w = sw[buf + off];
        const int32_t m = sm[buf + off];
        const int skip = meta_skip(m), push = meta_push(m);
        const int64_t *prev = srow + (r & 1) * kpad;            // D[i+1], column-major
        int64_t *outr = srow + ((r + 1) & 1) * kpad;            // D[i]
        uint32_t myword = 0;
#pragma unroll
        for (int c = 0; c < C; ++c) {
            int64_t s;
            if (skip == kSkipCur) s = cur[c];
            else if (skip == kSkipZero) s = 0;
            else if (skip < L_smem) s = sstk[((size_t)skip * C + c) * T + t];
            else s = gst[((size_t)(skip - L_smem) * C + c) * T + t];
            const int col = t * C + c + 1;
            const int jj = col - w;
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
            const uint32_t bw = __ballot_sync(0xffffffffu, take);
            if (lane == c) myword = bw;
        }
        if (lane < C) B[(size_t)i * words + warp * C + lane] = myword;
        if (push >= 0) {
#pragma unroll
            for (int c = 0; c < C; ++c) {
                if (push < L_smem) sstk[((size_t)push * C + c) * T + t] = cur[c];
                else gst[((size_t)(push - L_smem) * C + c) * T + t] = cur[c];
            }
        }
        if (off == kMetaRows - 1) {      // publish the prefetched block
            const int x = (blk + 1) * kMetaRows + t;
            const int nb = ((blk + 1) & 1) * kMetaRows;
            if (t < kMetaRows && x < n) {
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

// ---------------------------------------------------------------------------
// Traceback from (0, k): read the decision bit of (i, j); take -> mark b_i,
// j -= w_i, i += 1; skip -> i = next(i).  Stops at i = n or j = 0 (no column
// 0 bit is ever set).  One thread walks; the block first clears the output.
// Planner mode (acc != nullptr): the update of worker h is accepted in the
// greedy pass, or in refinement iff D[0][k] > sum of p_h over the current
// T_h (equivalent to G(T_-h, T'_h) > G(T) by Prop. 1); an accepted update
// replaces bit h of the holder masks by the traced set.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
k_traceback(int32_t n, const uint32_t *__restrict__ bits, int C, int kpad,
            const int32_t *__restrict__ item_budget, const int32_t *__restrict__ order,
            const int32_t *__restrict__ wpre, const int32_t *__restrict__ next,
            uint8_t *__restrict__ chosen, AcceptArgs acc)
{
    const int item = blockIdx.x;
    const int words = kpad >> 5;
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
        for (int32_t x = threadIdx.x; x < n; x += blockDim.x) M[x] &= ~hbit;
    } else {
        uint8_t *ch = chosen + (size_t)item * n;
        for (int32_t x = threadIdx.x; x < n; x += blockDim.x) ch[x] = 0;
    }
    __syncthreads();
    if (threadIdx.x != 0) return;
    if (acc.mask && !acc.greedy) {
        acc.improved[item] = 1;
        acc.accepted[item] += 1;
    }
    int32_t kq = item_budget[item];
    if (kq <= 0) return;
    int32_t j = kq < kpad ? kq : kpad;
    const uint32_t *Bi = bits + (size_t)item * n * words;
    int32_t i = 0;
    while (i < n && j > 0) {
        const int q = j - 1;
        const int tt = q / C, c = q - tt * C;
        const uint32_t word = Bi[(size_t)i * words + (tt >> 5) * C + c];
        if ((word >> (tt & 31)) & 1u) {
            if (M) M[i] |= hbit;
            else chosen[(size_t)item * n + order[i]] = 1;
            j -= wpre[i];
            i += 1;
        } else {
            i = next[i];
        }
    }
}

template <int C>
static pp_status launch_dp_c(pp_instance *inst, int batch, const int64_t *profit, bool by_node,
                             const int32_t *item_budget, int32_t max_budget,
                             const int32_t *item_active, const DpGeom &g, int64_t *best,
                             uint32_t *bits, cudaStream_t st)
{
    int dev_smem = 0;
    PP_CUDA(cudaDeviceGetAttribute(&dev_smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, inst->device));
    const size_t fixed = dp_smem_fixed(g);
    const size_t row_bytes = (size_t)g.kpad * sizeof(int64_t);
    if (fixed > (size_t)dev_smem) return fail(PP_EINVAL, "budget too large for the DP kernel");
    int L_smem = (int)std::min<size_t>((size_t)inst->stack_depth, ((size_t)dev_smem - fixed) / row_bytes);
    int L_glob = inst->stack_depth - L_smem;
    if (L_glob > 0) {
        pp_status s = ensure_scratch(inst->stack, (size_t)batch * L_glob * row_bytes);
        if (s != PP_OK) return s;
    }
    const size_t smem = fixed + (size_t)L_smem * row_bytes;
    PP_CUDA(cudaFuncSetAttribute(k_tree_dp<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    k_tree_dp<C><<<batch, g.T, smem, st>>>(inst->n, profit, by_node ? inst->d_order : nullptr,
                                            inst->d_wpre, inst->d_meta, item_budget, max_budget,
                                            item_active, best, bits,
                                            reinterpret_cast<int64_t *>(inst->stack.ptr), L_smem,
                                            L_glob, inst->d_status);
    PP_CUDA(cudaGetLastError());
    return PP_OK;
}

pp_status launch_tree_dp(pp_instance *inst, int batch, const int64_t *profit, bool by_node,
                         const int32_t *item_budget, const int32_t *item_active, const DpGeom &g,
                         int64_t *best, uint32_t *bits, cudaStream_t st, int32_t max_budget)
{
    if (batch <= 0) return PP_OK;
    if (inst->n == 0) {
        PP_CUDA(cudaMemsetAsync(best, 0, sizeof(int64_t) * batch, st));
        return PP_OK;
    }
    switch (g.C) {
    case 1: return launch_dp_c<1>(inst, batch, profit, by_node, item_budget, max_budget, item_active, g, best, bits, st);
    case 2: return launch_dp_c<2>(inst, batch, profit, by_node, item_budget, max_budget, item_active, g, best, bits, st);
    case 4: return launch_dp_c<4>(inst, batch, profit, by_node, item_budget, max_budget, item_active, g, best, bits, st);
    case 8: return launch_dp_c<8>(inst, batch, profit, by_node, item_budget, max_budget, item_active, g, best, bits, st);
    case 16: return launch_dp_c<16>(inst, batch, profit, by_node, item_budget, max_budget, item_active, g, best, bits, st);
    case 32: return launch_dp_c<32>(inst, batch, profit, by_node, item_budget, max_budget, item_active, g, best, bits, st);
    default: return fail(PP_EINVAL, "unsupported DP geometry");
    }
}

pp_status launch_traceback(pp_instance *inst, int batch, const uint32_t *bits, const DpGeom &g,
                           const int32_t *item_budget, uint8_t *chosen, const AcceptArgs *acc,
                           cudaStream_t st)
{
    if (batch <= 0 || inst->n == 0) return PP_OK;
    AcceptArgs a;
    if (acc) a = *acc;
    k_traceback<<<batch, 256, 0, st>>>(inst->n, bits, g.C, g.kpad, item_budget, inst->d_order,
                                       inst->d_wpre, inst->d_next, chosen, a);
    PP_CUDA(cudaGetLastError());
    return PP_OK;
}

}  // namespace pp

using namespace pp;

extern "C" size_t pp_dp_bits_size(const pp_instance *inst, int32_t batch, int32_t max_budget)
{
    DpGeom g;
    if (!inst || batch <= 0 || !dp_geometry(inst, max_budget, &g)) return 0;
    return (size_t)batch * (size_t)inst->n * (size_t)g.words * sizeof(uint32_t);
}

extern "C" pp_status pp_tree_dp(pp_instance *inst, int32_t batch, const int64_t *profit,
                                const int32_t *budget, int32_t max_budget, int64_t *best,
                                uint32_t *bits, void *stream)
{
    if (!inst) return fail(PP_EINVAL, "null instance");
    if (batch < 0) return fail(PP_EINVAL, "batch must be >= 0");
    DpGeom g;
    if (!dp_geometry(inst, max_budget, &g)) return fail(PP_EINVAL, "max_budget out of range");
    if (batch == 0) return PP_OK;
    if (!budget || !best || (inst->n > 0 && (!profit || !bits)))
        return fail(PP_EINVAL, "null device pointer");
    return launch_tree_dp(inst, batch, profit, true, budget, nullptr, g, best, bits,
                          (cudaStream_t)stream, max_budget);
}

extern "C" pp_status pp_traceback(pp_instance *inst, int32_t batch, const uint32_t *bits,
                                  const int32_t *budget, int32_t max_budget, uint8_t *chosen,
                                  void *stream)
{
    if (!inst) return fail(PP_EINVAL, "null instance");
    if (batch < 0) return fail(PP_EINVAL, "batch must be >= 0");
    DpGeom g;
    if (!dp_geometry(inst, max_budget, &g)) return fail(PP_EINVAL, "max_budget out of range");
    if (batch == 0 || inst->n == 0) return PP_OK;
    if (!bits || !budget || !chosen) return fail(PP_EINVAL, "null device pointer");
    return launch_traceback(inst, batch, bits, g, budget, chosen, nullptr, (cudaStream_t)stream);
}
