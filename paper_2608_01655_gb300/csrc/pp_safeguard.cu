// Safeguard candidates of Algorithm 1 for the requester-side objective
// (Section IV-C; the comparators of Section V-A).  Every worker's target is
// the exact rooted-tree DP (Eq. 9) on one of three profits:
//   Independent  Lambda_m(b) w_m(b) = a_m(b) + Lambda_m(b) [w_m(b) - f_m(b)]_+
//                (the worker alone: cross-worker reuse ignored)
//   Popularity   Lambda_m(b) (local demand alone)
//   LocalDedup   workers in index order; a chunk an earlier worker already
//                holds is worth only a_m(b) (Eq. 2), any other chunk
//                Lambda_m(b) w_m(b) -- the worker's own first-copy saving,
//                not the requester-wide Delta(b) of Eq. 3.
// Independent and Popularity are 2W independent DPs in one batched launch;
// LocalDedup is W dependent single-item launches.
#include <algorithm>
#include <cstring>
#include <vector>

#include "pp_internal.cuh"

namespace pp {

// item b (blockIdx.y): worker[b], kind[b] = 0 Independent, 1 Popularity,
// 2 LocalDedup against the holder mask `held` (preorder, bits of earlier workers)
__global__ void k_sg_profit(int32_t n, const int32_t *__restrict__ kind, const int32_t *__restrict__ worker,
                            const uint32_t *__restrict__ held, const int64_t *__restrict__ a,
                            const int64_t *__restrict__ own, const int64_t *__restrict__ pop,
                            int64_t *__restrict__ profit)
{
    const int b = blockIdx.y;
    const int m = worker[b], kd = kind[b];
    int64_t *out = profit + (size_t)b * n;
    for (int32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        const size_t o = (size_t)m * n + i;
        int64_t p;
        if (kd == 1) p = pop[o];
        else if (kd == 2 && held[i] != 0) p = a[o];
        else p = a[o] + own[o];
        out[i] = p;
    }
}

// cand[c][i] = OR of the C groups of W rows (each row holds one worker's bit)
__global__ void k_or_rows(int32_t n, int32_t W, int32_t C, const uint32_t *__restrict__ rows,
                          uint32_t *__restrict__ cand)
{
    const int c = blockIdx.y;
    for (int32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        uint32_t v = 0;
        for (int m = 0; m < W; ++m) v |= rows[((size_t)c * W + m) * n + i];
        cand[(size_t)c * n + i] = v;
    }
}

static size_t a256(size_t x) { return (x + 255) & ~(size_t)255; }

pp_status safeguards_impl(pp_instance *inst, cudaStream_t st, const uint32_t **masks, int64_t *obj,
                          int *launches, int64_t *cells, int *dp_launches)
{
    if (inst->mode != PP_TRANSFER_REQUESTER)
        return fail(PP_EINVAL, "safeguard candidates are defined for the requester-side objective only");
    const int32_t n = inst->n, W = inst->W;
    const int B = 2 * W;
    int32_t maxk = 0;
    int64_t sumk = 0;
    for (int32_t m = 0; m < W; ++m) {
        maxk = std::max(maxk, inst->h_budget[m]);
        sumk += inst->h_budget[m];
    }
    DpGeom gB, g1;
    if (!dp_geometry(inst, maxk, &gB, B) || !dp_geometry(inst, maxk, &g1, 1))
        return fail(PP_EINVAL, "budget too large for the DP kernel");
    const size_t N = (size_t)std::max(n, 1);
    // rows [B][n] | cand [3][n] | profit [B][n] | best [B] | objd [3] | ints [5][B] | DP work
    const size_t o_rows = 0, o_cand = o_rows + a256(4 * N * B), o_prof = o_cand + a256(4 * N * 3);
    const size_t o_best = o_prof + a256(8 * N * B), o_obj = o_best + a256(8 * (size_t)B);
    const size_t o_int = o_obj + a256(8 * 3), o_work = o_int + a256(4 * 5 * (size_t)B);
    const size_t wbytes = std::max(dp_work_bytes(B, n, gB.words), dp_work_bytes(1, n, g1.words));
    pp_status s = ensure_scratch(inst->sg, o_work + wbytes);
    if (s != PP_OK) return s;
    char *base = reinterpret_cast<char *>(inst->sg.ptr);
    uint32_t *rows = reinterpret_cast<uint32_t *>(base + o_rows);
    uint32_t *cand = reinterpret_cast<uint32_t *>(base + o_cand);
    int64_t *profit = reinterpret_cast<int64_t *>(base + o_prof);
    int64_t *best = reinterpret_cast<int64_t *>(base + o_best);
    int64_t *objd = reinterpret_cast<int64_t *>(base + o_obj);
    int32_t *ints = reinterpret_cast<int32_t *>(base + o_int);
    int32_t *kind = ints, *worker = ints + B, *kb = ints + 2 * B, *active = ints + 3 * B, *dd_kind = ints + 4 * B;
    std::vector<int32_t> h(5 * (size_t)B);
    for (int m = 0; m < W; ++m) {
        h[m] = 0;                                   // Independent
        h[W + m] = 1;                               // Popularity
        h[B + m] = h[B + W + m] = m;                // workers
        h[2 * B + m] = h[2 * B + W + m] = inst->h_budget[m];
        h[3 * B + m] = h[3 * B + W + m] = 1;        // active
        h[4 * B + m] = h[4 * B + W + m] = 2;        // LocalDedup
    }
    PP_CUDA(cudaMemcpyAsync(ints, h.data(), 4 * h.size(), cudaMemcpyHostToDevice, st));
    PP_CUDA(cudaMemsetAsync(rows, 0, 4 * N * B, st));
    PP_CUDA(cudaMemsetAsync(cand, 0, 4 * N * 3, st));
    int nl = 0;
    if (n > 0 && W > 0) {
        int bx = (n + 255) / 256;
        if (bx > 2 * inst->sm_count) bx = 2 * inst->sm_count;
        const DpWork wB = dp_work_split(base + o_work, B, n, gB.words);
        const DpWork w1 = dp_work_split(base + o_work, 1, n, g1.words);
        // Independent and Popularity: 2W independent DPs, one batch
        k_sg_profit<<<dim3(bx, B), 256, 0, st>>>(n, kind, worker, nullptr, inst->d_a, inst->d_own, inst->d_pop,
                                                 profit);
        PP_CUDA(cudaGetLastError());
        if ((s = launch_tree_dp(inst, B, profit, false, kb, nullptr, gB, best, wB, st, maxk))) return s;
        AcceptArgs acc;
        acc.worker = worker;
        acc.best = best;
        acc.active = active;
        acc.mask = rows;
        acc.greedy = 1;
        if ((s = launch_traceback(inst, B, wB, gB, kb, nullptr, &acc, st))) return s;
        k_or_rows<<<dim3(bx, 2), 256, 0, st>>>(n, W, 2, rows, cand);
        PP_CUDA(cudaGetLastError());
        nl += 5 + (gB.split ? 1 : 0);             // a split DP is two launches
        // LocalDedup: worker m sees the chunks of workers 0..m-1 in cand[2]
        uint32_t *dd = cand + 2 * N;
        for (int m = 0; m < W; ++m) {
            k_sg_profit<<<dim3(bx, 1), 256, 0, st>>>(n, dd_kind + m, worker + m, dd, inst->d_a, inst->d_own,
                                                     inst->d_pop, profit);
            PP_CUDA(cudaGetLastError());
            if ((s = launch_tree_dp(inst, 1, profit, false, kb + m, nullptr, g1, best, w1, st, maxk))) return s;
            AcceptArgs a1;
            a1.worker = worker + m;
            a1.best = best;
            a1.active = active;
            a1.mask = dd;
            a1.greedy = 1;
            if ((s = launch_traceback(inst, 1, w1, g1, kb + m, nullptr, &a1, st))) return s;
            nl += 4;
        }
    }
    if ((s = launch_objective(inst, 3, cand, nullptr, objd, st))) return s;
    nl += 1;
    PP_CUDA(cudaMemcpyAsync(obj, objd, 8 * 3, cudaMemcpyDeviceToHost, st));
    PP_CUDA(cudaStreamSynchronize(st));
    *masks = cand;
    if (launches) *launches += nl;
    if (cells) *cells += 3 * (int64_t)n * sumk;
    if (dp_launches) *dp_launches += (n > 0 && W > 0) ? 1 + W : 0;
    return PP_OK;
}

}  // namespace pp

using namespace pp;

extern "C" pp_status pp_safeguards(pp_instance *inst, uint8_t *placement, int64_t *objective, void *stream)
{
    if (!inst || !placement || !objective) return fail(PP_EINVAL, "null argument");
    int cur = 0;
    PP_CUDA(cudaGetDevice(&cur));
    if (cur != inst->device) return fail(PP_EINVAL, "the instance's device must be the current device");
    cudaStream_t st = (cudaStream_t)stream;
    const uint32_t *masks = nullptr;
    pp_status s = safeguards_impl(inst, st, &masks, objective, nullptr, nullptr, nullptr);
    if (s != PP_OK) return s;
    const int32_t n = inst->n, W = inst->W;
    std::memset(placement, 0, (size_t)3 * W * n);
    if (n == 0) return PP_OK;
    std::vector<uint32_t> mk((size_t)3 * n);
    PP_CUDA(cudaMemcpyAsync(mk.data(), masks, 4 * mk.size(), cudaMemcpyDeviceToHost, st));
    PP_CUDA(cudaStreamSynchronize(st));
    for (int c = 0; c < 3; ++c)
        for (int32_t i = 0; i < n; ++i) {
            uint32_t m = mk[(size_t)c * n + i];
            while (m) {
                const int h = __builtin_ctz(m);
                m &= m - 1;
                placement[((size_t)c * W + h) * n + inst->h_order[i]] = 1;
            }
        }
    return PP_OK;
}
