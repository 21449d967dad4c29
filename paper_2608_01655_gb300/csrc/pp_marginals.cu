// Per-worker exact node marginals (Prop. 1) and the planner objective.
//   requester-side (Eq. 10):   p_h(b) = a_h(b) + 1{no holder l != h} Delta(b)
//   source-dependent (Eq. 7):  p_h(b) = sum_m [g_h,m(b) - max_{l in H_b \ h} g_l,m(b)]_+
// where g_h,m(b) = Lambda_m(b) q_{m<-h}(b) (Eq. 5) is precomputed per instance
// and the max over an empty holder set is 0.  Objectives: F (Eq. 4) and
// F_pair (Eq. 6).  All arithmetic is exact int64.
#include "pp_internal.cuh"

namespace pp {

__device__ __forceinline__ int64_t warp_sum64(int64_t v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(0xffffffffu, v, o);
    return v;
}

// block-wide sum added atomically into *dst (integer addition is exact, so the
// result does not depend on the order of the atomics)
__device__ __forceinline__ void block_add64(int64_t v, int64_t *dst)
{
    __shared__ int64_t part[32];
    v = warp_sum64(v);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0) part[wid] = v;
    __syncthreads();
    if (wid == 0) {
        int nw = (blockDim.x + 31) >> 5;
        int64_t x = lane < nw ? part[lane] : 0;
        x = warp_sum64(x);
        if (lane == 0 && x != 0) atomicAdd((unsigned long long *)dst, (unsigned long long)x);
    }
}

// Marginal of one chunk at preorder position i for worker h; `others` is the
// holder mask without bit h.
template <int MODE>
__device__ __forceinline__ int64_t marginal_at(int32_t n, int32_t W, int32_t h, int32_t i,
                                               uint32_t others, const int64_t *__restrict__ a,
                                               const int64_t *__restrict__ delta,
                                               const int64_t *__restrict__ g)
{
    if (MODE == 0) {
        int64_t p = a[(size_t)h * n + i];
        if (others == 0) p += delta[i];
        return p;
    } else {
        int64_t p = 0;
        for (int32_t m = 0; m < W; ++m) {
            int64_t mine = g[((size_t)h * W + m) * n + i];
            int64_t v = 0;
            uint32_t o = others;
            while (o) {
                int l = __ffs(o) - 1;
                o &= o - 1;
                int64_t x = g[((size_t)l * W + m) * n + i];
                v = x > v ? x : v;
            }
            p += mine > v ? mine - v : 0;
        }
        return p;
    }
}

// grid: (blocks over positions, batch).  BYNODE: masks / profits indexed by
// node id (ABI); otherwise by preorder position (planner).  oldsum (optional)
// receives sum of p_h over the chunks worker h currently holds, which equals
// G(T) - G(T_-h, {}) by Prop. 1 and is the refinement's acceptance threshold.
template <bool BYNODE, int MODE>
__global__ void __launch_bounds__(256) k_marginals(int32_t n, int32_t W,
                                                    const int32_t *__restrict__ worker,
                                                    const uint32_t *__restrict__ mask,
                                                    const int32_t *__restrict__ order,
                                                    const int64_t *__restrict__ a,
                                                    const int64_t *__restrict__ delta,
                                                    const int64_t *__restrict__ g,
                                                    const int32_t *__restrict__ item_active,
                                                    int64_t *__restrict__ profit,
                                                    int64_t *__restrict__ oldsum,
                                                    int32_t *__restrict__ status)
{
    const int item = blockIdx.y;
    if (item_active && !item_active[item]) return;
    const int32_t h = worker[item];
    const uint32_t *M = mask + (size_t)item * n;
    int64_t *P = profit + (size_t)item * n;
    if (h < 0 || h >= W) {
        if (threadIdx.x == 0 && blockIdx.x == 0) atomicExch(status, (int32_t)PP_EBOUNDS);
        for (int32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x)
            P[i] = 0;
        return;
    }
    const uint32_t hb = 1u << h;
    int64_t held = 0;
    for (int32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        const int32_t idx = BYNODE ? order[i] : i;
        const uint32_t mk = M[idx];
        const int64_t p = marginal_at<MODE>(n, W, h, i, mk & ~hb, a, delta, g);
        P[idx] = p;
        if (mk & hb) held += p;
    }
    if (oldsum) block_add64(held, oldsum + item);
}

template <bool BYNODE>
static void marg_dispatch(pp_instance *inst, dim3 grid, int batch, const int32_t *worker,
                          const uint32_t *mask, const int32_t *item_active, int64_t *profit,
                          int64_t *oldsum, cudaStream_t st)
{
    if (inst->mode == 0)
        k_marginals<BYNODE, 0><<<grid, 256, 0, st>>>(inst->n, inst->W, worker, mask, inst->d_order,
                                                     inst->d_a, inst->d_delta, inst->d_g,
                                                     item_active, profit, oldsum, inst->d_status);
    else
        k_marginals<BYNODE, 1><<<grid, 256, 0, st>>>(inst->n, inst->W, worker, mask, inst->d_order,
                                                     inst->d_a, inst->d_delta, inst->d_g,
                                                     item_active, profit, oldsum, inst->d_status);
}

pp_status launch_marginals(pp_instance *inst, int batch, const int32_t *worker,
                           const uint32_t *mask, bool by_node, const int32_t *item_active,
                           int64_t *profit, int64_t *oldsum, cudaStream_t st)
{
    if (batch <= 0 || inst->n == 0) return PP_OK;
    if (oldsum) PP_CUDA(cudaMemsetAsync(oldsum, 0, sizeof(int64_t) * batch, st));
    int bx = (inst->n + 255) / 256;
    int cap = (2 * inst->sm_count * 8 + batch - 1) / batch;   // ~16 blocks per SM overall
    if (bx > cap) bx = cap;
    if (bx < 1) bx = 1;
    dim3 grid(bx, batch);
    if (by_node) marg_dispatch<true>(inst, grid, batch, worker, mask, item_active, profit, oldsum, st);
    else marg_dispatch<false>(inst, grid, batch, worker, mask, item_active, profit, oldsum, st);
    PP_CUDA(cudaGetLastError());
    return PP_OK;
}

// ---------------------------------------------------------------------------
// Source-dependent marginals from top-2 holder tables (Section IV-C: keeping
// the largest and second-largest current holder value of every requester-
// chunk pair gives every leave-one-worker-out marginal in O(M^2 n) per sweep).
// Per start s, requester m and position i: v1 = max over the holders l of
// g_{l,m}(i), l1 = the first holder reaching it, v2 = the largest value among
// the other holders (0 with fewer than two).  Then
//   max_{l in H_b \ h} g_{l,m}(b) = (l1 == h) ? v2 : v1,
// which is exact also under ties (then v2 = v1).  The marginal kernel records
// each chunk's bit h before the update, and the next step's marginal pass
// first applies the change of exactly the chunks whose bit h changed.
// ---------------------------------------------------------------------------
// Apply worker h's change at chunk i to the top-2 tables (tb = the start's
// table base): h joined -> insert its values; h left -> rebuild the entries
// where it was the top holder or tied the second.
__device__ __forceinline__ void top2_apply(int32_t n, int32_t W, int32_t h, int32_t i, uint32_t mk, bool now,
                                           size_t tb, const int64_t *__restrict__ g, int64_t *__restrict__ v1,
                                           int64_t *__restrict__ v2, int8_t *__restrict__ l1)
{
    for (int32_t m = 0; m < W; ++m) {
        const size_t q = tb + (size_t)m * n + i;
        const int64_t x = g[((size_t)h * W + m) * n + i];
        if (now) {
            if (l1[q] < 0 || x > v1[q]) {
                v2[q] = l1[q] < 0 ? 0 : v1[q];
                v1[q] = x;
                l1[q] = (int8_t)h;
            } else if (x > v2[q]) {
                v2[q] = x;
            }
            continue;
        }
        if (l1[q] != h && x < v2[q]) continue;
        int64_t b1 = 0, b2 = 0;
        int id1 = -1;
        uint32_t o = mk;
        while (o) {
            const int l = __ffs(o) - 1;
            o &= o - 1;
            const int64_t y = g[((size_t)l * W + m) * n + i];
            if (id1 < 0 || y > b1) {
                b2 = id1 < 0 ? 0 : b1;
                b1 = y;
                id1 = l;
            } else if (y > b2) {
                b2 = y;
            }
        }
        v1[q] = b1;
        v2[q] = b2;
        l1[q] = (int8_t)id1;
    }
}

// prev_worker (optional): the worker of the start's previous step, whose
// change is applied to the tables first (the bit recorded then vs the mask now)
__global__ void __launch_bounds__(256) k_marginals_top2(int32_t n, int32_t W,
                                                         const int32_t *__restrict__ prev_worker,
                                                         const int32_t *__restrict__ worker,
                                                         const uint32_t *__restrict__ mask,
                                                         const int64_t *__restrict__ g,
                                                         int64_t *__restrict__ v1,
                                                         int64_t *__restrict__ v2,
                                                         int8_t *__restrict__ l1,
                                                         const int32_t *__restrict__ item_active,
                                                         int64_t *__restrict__ profit,
                                                         int64_t *__restrict__ oldsum,
                                                         uint8_t *__restrict__ oldbit,
                                                         int32_t *__restrict__ status)
{
    const int item = blockIdx.y;
    if (item_active && !item_active[item]) return;
    const int32_t h = worker[item];
    const uint32_t *M = mask + (size_t)item * n;
    int64_t *P = profit + (size_t)item * n;
    if (h < 0 || h >= W) {
        if (threadIdx.x == 0 && blockIdx.x == 0) atomicExch(status, (int32_t)PP_EBOUNDS);
        for (int32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) P[i] = 0;
        return;
    }
    const size_t tb = (size_t)item * W * n;
    const int32_t hp = prev_worker ? prev_worker[item] : -1;
    int64_t held = 0;
    for (int32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        const uint32_t mk = M[i];
        if (hp >= 0 && hp < W) {
            const bool now = (mk >> hp) & 1u;
            if (now != (bool)oldbit[(size_t)item * n + i]) top2_apply(n, W, hp, i, mk, now, tb, g, v1, v2, l1);
        }
        int64_t p = 0;
        for (int32_t m = 0; m < W; ++m) {
            const size_t o = tb + (size_t)m * n + i;
            const int64_t other = l1[o] == h ? v2[o] : v1[o];
            const int64_t mine = g[((size_t)h * W + m) * n + i];
            p += mine > other ? mine - other : 0;
        }
        P[i] = p;
        const bool hh = (mk >> h) & 1u;
        oldbit[(size_t)item * n + i] = hh;
        if (hh) held += p;
    }
    if (oldsum) block_add64(held, oldsum + item);
}

pp_status launch_marginals_top2(pp_instance *inst, int batch, const int32_t *prev_worker, const int32_t *worker,
                                const uint32_t *mask, const int32_t *item_active, const Top2 &t2,
                                int64_t *profit, int64_t *oldsum, cudaStream_t st)
{
    if (batch <= 0 || inst->n == 0) return PP_OK;
    if (oldsum) PP_CUDA(cudaMemsetAsync(oldsum, 0, sizeof(int64_t) * batch, st));
    int bx = (inst->n + 255) / 256;
    int cap = (2 * inst->sm_count * 8 + batch - 1) / batch;
    if (bx > cap) bx = cap;
    if (bx < 1) bx = 1;
    k_marginals_top2<<<dim3(bx, batch), 256, 0, st>>>(inst->n, inst->W, prev_worker, worker, mask, inst->d_g,
                                                      t2.v1, t2.v2,
                                                      t2.l1, item_active, profit, oldsum, t2.oldbit,
                                                      inst->d_status);
    PP_CUDA(cudaGetLastError());
    return PP_OK;
}

// ---------------------------------------------------------------------------
// Objective of holder masks (planner, preorder) or of [W][n] byte placements
// by node id (ABI).  Eq. 4: sum over held (m, b) of a_m(b) plus Delta(b) once
// per covered chunk.  Eq. 6: sum_b sum_m max_{h in H_b} g_h,m(b).
// ---------------------------------------------------------------------------
template <bool FROM_BYTES, int MODE>
__global__ void __launch_bounds__(256) k_objective(int32_t n, int32_t W,
                                                    const uint32_t *__restrict__ mask,
                                                    const uint8_t *__restrict__ chosen,
                                                    const int32_t *__restrict__ order,
                                                    const int64_t *__restrict__ a,
                                                    const int64_t *__restrict__ delta,
                                                    const int64_t *__restrict__ g,
                                                    int64_t *__restrict__ obj)
{
    const int item = blockIdx.y;
    int64_t acc = 0;
    for (int32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        uint32_t mk = 0;
        if (FROM_BYTES) {
            const int32_t b = order[i];
            for (int32_t m = 0; m < W; ++m)
                if (chosen[((size_t)item * W + m) * n + b]) mk |= 1u << m;
        } else {
            mk = mask[(size_t)item * n + i];
        }
        if (mk == 0) continue;
        if (MODE == 0) {
            uint32_t o = mk;
            while (o) {
                int m = __ffs(o) - 1;
                o &= o - 1;
                acc += a[(size_t)m * n + i];
            }
            acc += delta[i];
        } else {
            for (int32_t m = 0; m < W; ++m) {
                int64_t best = 0;
                uint32_t o = mk;
                while (o) {
                    int h = __ffs(o) - 1;
                    o &= o - 1;
                    int64_t x = g[((size_t)h * W + m) * n + i];
                    best = x > best ? x : best;
                }
                acc += best;
            }
        }
    }
    block_add64(acc, obj + item);
}

pp_status launch_objective(pp_instance *inst, int batch, const uint32_t *mask,
                           const uint8_t *chosen, int64_t *obj, cudaStream_t st)
{
    if (batch <= 0) return PP_OK;
    PP_CUDA(cudaMemsetAsync(obj, 0, sizeof(int64_t) * batch, st));
    if (inst->n == 0) return PP_OK;
    int bx = (inst->n + 255) / 256;
    int cap = (2 * inst->sm_count * 8 + batch - 1) / batch;
    if (bx > cap) bx = cap;
    if (bx < 1) bx = 1;
    dim3 grid(bx, batch);
    const int32_t n = inst->n, W = inst->W;
    if (chosen) {
        if (inst->mode == 0)
            k_objective<true, 0><<<grid, 256, 0, st>>>(n, W, nullptr, chosen, inst->d_order, inst->d_a,
                                                       inst->d_delta, inst->d_g, obj);
        else
            k_objective<true, 1><<<grid, 256, 0, st>>>(n, W, nullptr, chosen, inst->d_order, inst->d_a,
                                                       inst->d_delta, inst->d_g, obj);
    } else {
        if (inst->mode == 0)
            k_objective<false, 0><<<grid, 256, 0, st>>>(n, W, mask, nullptr, inst->d_order, inst->d_a,
                                                        inst->d_delta, inst->d_g, obj);
        else
            k_objective<false, 1><<<grid, 256, 0, st>>>(n, W, mask, nullptr, inst->d_order, inst->d_a,
                                                        inst->d_delta, inst->d_g, obj);
    }
    PP_CUDA(cudaGetLastError());
    return PP_OK;
}

}  // namespace pp

using namespace pp;

extern "C" pp_status pp_marginals(pp_instance *inst, int32_t batch, const int32_t *worker,
                                  const uint32_t *holder_mask, int64_t *profit, void *stream)
{
    if (!inst) return fail(PP_EINVAL, "null instance");
    if (batch < 0) return fail(PP_EINVAL, "batch must be >= 0");
    if (batch == 0 || inst->n == 0) return PP_OK;
    if (!worker || !holder_mask || !profit) return fail(PP_EINVAL, "null device pointer");
    return launch_marginals(inst, batch, worker, holder_mask, true, nullptr, profit, nullptr,
                            (cudaStream_t)stream);
}

extern "C" pp_status pp_objective(pp_instance *inst, int32_t batch, const uint8_t *chosen,
                                  int64_t *obj, void *stream)
{
    if (!inst) return fail(PP_EINVAL, "null instance");
    if (batch < 0) return fail(PP_EINVAL, "batch must be >= 0");
    if (batch == 0) return PP_OK;
    if (!obj || (inst->n > 0 && !chosen)) return fail(PP_EINVAL, "null device pointer");
    return launch_objective(inst, batch, nullptr, chosen, obj, (cudaStream_t)stream);
}
