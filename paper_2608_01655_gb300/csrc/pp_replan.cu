// Epoch update (Section IV-D; the amortisation rule and break-even requests of
// RQ5, Section V).  The instance carries the refreshed demand.  The incumbent
// placement is scored with the objective kernel, a reoptimised target comes
// from pp_plan_run, and the one-time cost of the target is the Section III-A
// materialisation cost, under the incumbent, of every chunk a worker newly
// holds: the cheaper of recomputing it and fetching it from a worker holding
// it in the incumbent (recomputing when none does).  The target is adopted iff
//   (G(T_new) - G(T_old)) * horizon_requests > cost * epoch_requests,
// G being a saving per epoch of epoch_requests requests.
#include <cstdint>
#include <cstring>
#include <vector>

#include "pp_internal.cuh"

namespace pp {

// sum over (m, b) with nw[m][b] && !old[m][b] of min(w_m(b), fetch from an old holder)
template <int MODE>
__global__ void k_mat_cost(int32_t n, int32_t W, const uint8_t *__restrict__ old, const uint8_t *__restrict__ nw,
                           const int64_t *__restrict__ rec, const int64_t *__restrict__ tr,
                           unsigned long long *__restrict__ total)
{
    const int m = blockIdx.y;
    int64_t acc = 0;
    for (int32_t b = blockIdx.x * blockDim.x + threadIdx.x; b < n; b += gridDim.x * blockDim.x) {
        const size_t o = (size_t)m * n + b;
        if (!nw[o] || old[o]) continue;
        int64_t c = rec[o];
        for (int h = 0; h < W; ++h) {
            if (h == m || !old[(size_t)h * n + b]) continue;
            const int64_t f = MODE == 0 ? tr[o] : tr[((size_t)h * W + m) * n + b];
            c = f < c ? f : c;
        }
        acc += c;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) acc += __shfl_down_sync(0xffffffffu, acc, off);
    if ((threadIdx.x & 31) == 0 && acc) atomicAdd(total, (unsigned long long)acc);
}

}  // namespace pp

using namespace pp;

extern "C" pp_status pp_replan(pp_instance *inst, const uint8_t *incumbent, int32_t n_starts,
                               const int32_t *orders, int32_t max_rounds, int64_t epoch_requests,
                               int64_t horizon_requests, uint8_t *placement, pp_replan_result *result,
                               pp_plan_stats *stats, void *stream)
{
    if (!inst || !incumbent || !placement || !result) return fail(PP_EINVAL, "null argument");
    if (epoch_requests <= 0 || horizon_requests < 0)
        return fail(PP_EINVAL, "epoch_requests must be > 0 and horizon_requests >= 0");
    cudaStream_t st = (cudaStream_t)stream;
    const int32_t n = inst->n, W = inst->W;
    const size_t Wn = (size_t)W * n;
    std::vector<uint8_t> target(Wn ? Wn : 1);
    int64_t g_new = 0;
    pp_status s = plan_impl(inst, n_starts, orders, max_rounds, target.data(), &g_new, stats, st);
    if (s != PP_OK) return s;
    // incumbent and target on the device: objective of the incumbent, cost of the target
    const size_t a = (Wn + 255) & ~(size_t)255;
    if ((s = ensure_scratch(inst->rp, 2 * a + 256))) return s;
    uint8_t *d_old = reinterpret_cast<uint8_t *>(inst->rp.ptr), *d_new = d_old + a;
    int64_t *d_out = reinterpret_cast<int64_t *>(d_new + a);            // [0] objective, [1] cost
    int64_t h_out[2] = {0, 0};
    PP_CUDA(cudaMemsetAsync(d_out, 0, 16, st));
    if (Wn > 0) {
        PP_CUDA(cudaMemcpyAsync(d_old, incumbent, Wn, cudaMemcpyHostToDevice, st));
        PP_CUDA(cudaMemcpyAsync(d_new, target.data(), Wn, cudaMemcpyHostToDevice, st));
        if ((s = launch_objective(inst, 1, nullptr, d_old, d_out, st))) return s;
        int bx = (n + 255) / 256;
        if (bx > 2 * inst->sm_count) bx = 2 * inst->sm_count;
        const dim3 grid(bx, W);
        auto *tot = reinterpret_cast<unsigned long long *>(d_out + 1);
        if (inst->mode == PP_TRANSFER_REQUESTER)
            k_mat_cost<0><<<grid, 256, 0, st>>>(n, W, d_old, d_new, inst->d_rec, inst->d_tr, tot);
        else
            k_mat_cost<1><<<grid, 256, 0, st>>>(n, W, d_old, d_new, inst->d_rec, inst->d_tr, tot);
        PP_CUDA(cudaGetLastError());
        PP_CUDA(cudaMemcpyAsync(h_out, d_out, 16, cudaMemcpyDeviceToHost, st));
    }
    PP_CUDA(cudaStreamSynchronize(st));
    const int64_t g_old = h_out[0], cost = h_out[1], gain = g_new - g_old;
    result->incumbent_objective = g_old;
    result->new_objective = g_new;
    result->materialization_cost = cost;
    result->break_even_requests = -1;
    if (gain > 0) {                     // the ceiling, saturated at INT64_MAX
        const __int128 num = (__int128)cost * epoch_requests;
        const __int128 q = (num + gain - 1) / gain;
        result->break_even_requests = q > (__int128)INT64_MAX ? INT64_MAX : (int64_t)q;
    }
    result->adopted = gain > 0 && (__int128)gain * horizon_requests > (__int128)cost * epoch_requests;
    std::memcpy(placement, result->adopted ? target.data() : incumbent, Wn);
    return PP_OK;
}
