// Instance set-up: validation, preorder (Section IV-A), the DP's skip-row
// stack plan, and the gain tables of Eq. 2-3 (requester-side) or Eq. 5
// (source-dependent) computed on the device.
#include <algorithm>
#include <cstdio>
#include <cstring>
#include <new>
#include <thread>
#include <vector>

#include "pp_internal.cuh"

namespace pp {

static thread_local std::string g_last_error;

pp_status fail(pp_status s, const std::string &msg)
{
    g_last_error = msg;
    return s;
}

pp_status cuda_fail(cudaError_t e, const char *what)
{
    g_last_error = std::string(what) + ": " + cudaGetErrorString(e);
    return e == cudaErrorMemoryAllocation ? PP_ENOMEM : PP_ECUDA;
}

pp_status ensure_scratch(Scratch &s, size_t bytes)
{
    if (s.bytes >= bytes && s.ptr) return PP_OK;
    free_scratch(s);
    if (bytes == 0) return PP_OK;
    cudaError_t e = cudaMalloc(&s.ptr, bytes);
    if (e != cudaSuccess) {
        s.ptr = nullptr;
        return cuda_fail(e, "cudaMalloc(scratch)");
    }
    s.bytes = bytes;
    return PP_OK;
}

void free_scratch(Scratch &s)
{
    if (s.ptr) cudaFree(s.ptr);
    s.ptr = nullptr;
    s.bytes = 0;
}

// ---------------------------------------------------------------------------
// Preorder with roots first and children in ascending node id; next(i) is the
// first position after the subtree at position i.  Returns false if parent[]
// is not a forest.
// ---------------------------------------------------------------------------
static bool build_preorder(int32_t n, const int32_t *parent, std::vector<int32_t> &order,
                           std::vector<int32_t> &next)
{
    std::vector<int32_t> head(n + 1, -1), sib(n, -1), stack;
    // children lists in ascending id: insert in descending id at the head
    for (int32_t v = n - 1; v >= 0; --v) {
        int32_t p = parent[v] < 0 ? n : parent[v];
        sib[v] = head[p];
        head[p] = v;
    }
    order.assign(n, 0);
    next.assign(n, 0);
    std::vector<int32_t> pos(n, -1);
    int32_t cnt = 0;
    // iterative DFS: a stack of "next child to visit" cursors
    std::vector<int32_t> cursor;
    cursor.push_back(head[n]);
    std::vector<int32_t> path;     // nodes whose subtree is open
    while (!cursor.empty()) {
        int32_t c = cursor.back();
        if (c < 0) {
            cursor.pop_back();
            if (!path.empty()) {
                int32_t u = path.back();
                path.pop_back();
                next[pos[u]] = cnt;
            }
            continue;
        }
        cursor.back() = sib[c];
        pos[c] = cnt;
        order[cnt++] = c;
        path.push_back(c);
        cursor.push_back(head[c]);
        if ((int32_t)path.size() > n) return false;
    }
    return cnt == n;
}

// Skip-row stack plan: see the DP row metadata comment in pp_internal.cuh.
static bool build_row_meta(int32_t n, const std::vector<int32_t> &next, std::vector<int32_t> &meta,
                           int32_t *depth_out, const std::vector<int32_t> *wpre = nullptr,
                           std::vector<int32_t> *wave = nullptr)
{
    meta.assign(n, 0);
    if (wave) wave->assign(n, 0);
    // last_reader[r] = smallest q with next(q) == r and q < r - 1 (stack reads only)
    std::vector<int32_t> last_reader(n + 1, -1);
    for (int32_t q = n - 1; q >= 0; --q) {
        int32_t r = next[q];
        if (r != q + 1 && r != n) last_reader[r] = q;
    }
    std::vector<int32_t> level(n + 1, -1);
    int32_t depth = 0, maxd = 0;
    for (int32_t i = n - 1; i >= 0; --i) {
        int32_t r = next[i];
        int skip;
        bool pop = false;
        if (r == i + 1) skip = kSkipCur;
        else if (r == n) skip = kSkipZero;
        else {
            skip = level[r];
            // every stack read is of the top: the rows pushed after row r belong
            // to the subtree of position i and were popped before i is reached
            if (skip < 0 || skip != depth - 1) return false;
            if (last_reader[r] == i) {          // last reader: pop
                --depth;
                pop = true;
            }
        }
        const int32_t depth_read = depth;        // after any pop, before any push
        int push = -1;
        if (i >= 1 && last_reader[i] >= 0) {
            push = depth;
            level[i] = depth++;
            if (depth > maxd) maxd = depth;
            if (depth > kMaxStackLevels) return false;
        }
        meta[i] = meta_pack(skip, push);
        if (wave) {
            const int w = (*wpre)[i];
            // next(i) = n only happens with an empty stack, whose top is the zero row
            if (skip == kSkipZero && depth_read != 0) return false;
            const int kind = skip == kSkipCur ? kWaveCur : kWaveTop;
            int flags = 0, lvl = 0;
            if (push >= 0) {
                flags = kWavePush;
                lvl = push;
            } else if (pop && depth_read > 0) {
                flags = kWaveReload;                 // the level below becomes the top
                lvl = depth_read - 1;
            } else if (pop) {
                flags = kWaveZeroTop;                // the stack emptied: top = zero row
            }
            (*wave)[i] = wave_pack(w > 8 ? 8 : w, kind, flags, lvl);
        }
    }
    *depth_out = maxd;
    return true;
}

// ---------------------------------------------------------------------------
// Gain tables (one-time precompute, preorder-indexed):
//   mode 0: a[m][i] = Lambda_m(b) min{w_m(b), f_m(b)}            (Eq. 2)
//           Delta[i] = sum_m Lambda_m(b) [w_m(b) - f_m(b)]_+       (Eq. 3)
//   mode 1: g[h][m][i] = Lambda_m(b) q_{m<-h}(b)                   (Eq. 5)
// with b = order[i].  Lambda >= 0 commutes with min, max and [.]_+, so Eq. 7
// can be evaluated on these products exactly.
// ---------------------------------------------------------------------------
__global__ void k_gain_requester(int32_t n, int32_t W, const int32_t *__restrict__ order,
                                 const int64_t *__restrict__ demand,
                                 const int64_t *__restrict__ recompute,
                                 const int64_t *__restrict__ transfer, int64_t *__restrict__ a,
                                 int64_t *__restrict__ delta, int64_t *__restrict__ own,
                                 int64_t *__restrict__ pop)
{
    for (int32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        int32_t b = order[i];
        int64_t d = 0;
        for (int32_t m = 0; m < W; ++m) {
            size_t o = (size_t)m * n + b;
            int64_t lam = demand[o], w = recompute[o], f = transfer[o];
            a[(size_t)m * n + i] = lam * (w < f ? w : f);
            own[(size_t)m * n + i] = lam * (w > f ? w - f : 0);
            pop[(size_t)m * n + i] = lam;
            d += lam * (w > f ? w - f : 0);
        }
        delta[i] = d;
    }
}

__global__ void k_gain_source(int32_t n, int32_t W, const int32_t *__restrict__ order,
                              const int64_t *__restrict__ demand,
                              const int64_t *__restrict__ recompute,
                              const int64_t *__restrict__ transfer, int64_t *__restrict__ g)
{
    const int32_t hm = blockIdx.y;               // h * W + m
    const int32_t h = hm / W, m = hm % W;
    for (int32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        int32_t b = order[i];
        int64_t lam = demand[(size_t)m * n + b], w = recompute[(size_t)m * n + b];
        int64_t q;
        if (h == m) q = w;
        else {
            int64_t f = transfer[(size_t)hm * n + b];
            q = w > f ? w - f : 0;
        }
        g[(size_t)hm * n + i] = lam * q;
    }
}

}  // namespace pp

using namespace pp;

extern "C" const char *pp_last_error(void) { return g_last_error.c_str(); }

extern "C" pp_status pp_instance_destroy(pp_instance *inst)
{
    if (!inst) return PP_OK;
    int cur = 0;
    cudaGetDevice(&cur);
    cudaSetDevice(inst->device);
    cudaFree(inst->d_order);
    cudaFree(inst->d_next);
    cudaFree(inst->d_wpre);
    cudaFree(inst->d_meta);
    cudaFree(inst->d_wave);
    cudaFree(inst->d_pspan);
    cudaFree(inst->d_budget);
    cudaFree(inst->d_a);
    cudaFree(inst->d_delta);
    cudaFree(inst->d_own);
    cudaFree(inst->d_pop);
    cudaFree(inst->d_rec);
    cudaFree(inst->d_tr);
    cudaFree(inst->d_g);
    cudaFree(inst->d_status);
    free_scratch(inst->stack);
    free_scratch(inst->plan);
    free_scratch(inst->plan_bits);
    free_scratch(inst->sg);
    free_scratch(inst->rp);
    free_scratch(inst->top2);
    if (inst->split_hi) cudaStreamDestroy(inst->split_hi);
    if (inst->split_lo) cudaStreamDestroy(inst->split_lo);
    if (inst->split_fork) cudaEventDestroy(inst->split_fork);
    if (inst->split_join_hi) cudaEventDestroy(inst->split_join_hi);
    if (inst->split_join_lo) cudaEventDestroy(inst->split_join_lo);
    for (cudaStream_t x : inst->plan_streams) cudaStreamDestroy(x);
    for (cudaEvent_t x : inst->plan_join) cudaEventDestroy(x);
    if (inst->plan_fork) cudaEventDestroy(inst->plan_fork);
    for (cudaEvent_t x : inst->phase_events) cudaEventDestroy(x);
    cudaSetDevice(cur);
    delete inst;
    return PP_OK;
}

template <typename T>
static pp_status upload(T **dst, const T *src, size_t count, cudaStream_t st)
{
    PP_CUDA(cudaMalloc((void **)dst, sizeof(T) * (count ? count : 1)));
    if (count) PP_CUDA(cudaMemcpyAsync(*dst, src, sizeof(T) * count, cudaMemcpyHostToDevice, st));
    return PP_OK;
}

// The tree's host tables of an instance: preorder, next, weights by
// position, the traceback's skip depth, the skip-row stack plan, budgets.
static pp_status build_host_tables(int32_t n, int32_t W, const int32_t *parent, const int32_t *weight,
                                   int32_t mode, const int32_t *budget, pp_instance *inst)
{
    inst->n = n;
    inst->W = W;
    inst->mode = mode;
    if (!build_preorder(n, parent, inst->h_order, inst->h_next))
        return fail(PP_ENOTTREE, "parent array contains a cycle");
    inst->h_wpre.resize(n);
    inst->total_weight = 0;
    inst->max_weight = 1;
    for (int32_t i = 0; i < n; ++i) {
        inst->h_wpre[i] = weight[inst->h_order[i]];
        inst->total_weight += weight[i];
        inst->max_weight = std::max(inst->max_weight, weight[i]);
    }
    {
        // the traceback's skip speculation: deeper where a chunk has many
        // siblings (long runs of skipped siblings), i.e. where the size-biased
        // mean fan-out sum c^2 / sum c over the chunks' child counts c is large
        std::vector<int64_t> nch(n, 0);
        for (int32_t v = 0; v < n; ++v)
            if (parent[v] >= 0) nch[parent[v]] += 1;
        int64_t s1 = 0, s2 = 0;
        for (int32_t v = 0; v < n; ++v) {
            s1 += nch[v];
            s2 += nch[v] * nch[v];
        }
        inst->trace_skips = s1 > 0 && s2 > 5 * s1 ? 3 : 1;
    }
    if (!build_row_meta(n, inst->h_next, inst->h_meta, &inst->stack_depth, &inst->h_wpre, &inst->h_wave))
        return fail(PP_EINVAL, "skip-row stack deeper than supported");
    inst->h_budget.assign(budget, budget + W);
    return PP_OK;
}

static pp_status create_impl(int32_t n, int32_t W, const int32_t *parent, const int32_t *weight,
                             const int64_t *demand, const int64_t *recompute,
                             const int64_t *transfer, int32_t mode, const int32_t *budget,
                             cudaStream_t st, pp_instance *inst)
{
    if (n < 0) return fail(PP_EINVAL, "n must be >= 0");
    if (W < 1 || W > 32) return fail(PP_EINVAL, "W must be in 1..32");
    if (mode != PP_TRANSFER_REQUESTER && mode != PP_TRANSFER_SOURCE)
        return fail(PP_EINVAL, "transfer_mode must be 0 (requester) or 1 (source)");
    if (!budget || (n > 0 && (!parent || !weight || !demand || !recompute || !transfer)))
        return fail(PP_EINVAL, "null input pointer");
    for (int32_t m = 0; m < W; ++m)
        if (budget[m] < 0) return fail(PP_EINVAL, "budget must be >= 0");
    for (int32_t v = 0; v < n; ++v) {
        if (parent[v] < -1 || parent[v] >= n || parent[v] == v)
            return fail(PP_ENOTTREE, "parent id out of range or self-parent at node " + std::to_string(v));
        if (weight[v] < 1) return fail(PP_EINVAL, "chunk weight must be >= 1");
    }
    const size_t Wn = (size_t)W * n;
    const size_t tn = mode == PP_TRANSFER_SOURCE ? (size_t)W * Wn : Wn;
    // Three exact sums bound every int64 value the library forms:
    //  sum Lambda * w: objectives (Eq. 4, Eq. 6), marginals and DP values;
    //  sum Lambda:     the Popularity safeguard's DP values (profit Lambda);
    //  sum w:          the epoch update's one-time cost (at most one w per (m, b)).
    // The cost arrays are checked before anything is allocated, on up to 16
    // host threads when they are large (the source-dependent transfer costs
    // are W^2 n values: 102 MB at the paper-scale workload), while this thread
    // builds the tree's host tables; cost errors are reported first.
    // Unsigned 128-bit sums (a negative value sets bit 63 of the OR and fails
    // before its sum is used); the products and the running sum of products
    // are capped at 2^63, above the 2^62 limit, so nothing wraps.
    using u128 = unsigned __int128;
    const u128 cap = (u128)1 << 63;
    struct Part {
        u128 total = 0, demand = 0, recompute = 0;
        uint64_t dr_bits = 0, t_bits = 0;          // OR of the values: bit 63 = a negative one
    };
    const size_t work = Wn + tn;
    const unsigned hw = std::max(1u, std::thread::hardware_concurrency());
    const int nth = work < ((size_t)1 << 20) ? 1 : (int)std::min<unsigned>(hw, 16);
    std::vector<Part> parts(nth);
    auto check = [&](int q) {
        Part &P = parts[q];
        const size_t a = Wn * q / nth, b = Wn * (q + 1) / nth;
        for (size_t x = a; x < b; ++x) {
            const uint64_t dv = (uint64_t)demand[x], rv = (uint64_t)recompute[x];
            P.dr_bits |= dv | rv;
            const u128 pr = (u128)dv * rv;
            P.total = std::min<u128>(P.total + std::min(pr, cap), cap);
            P.demand += dv;
            P.recompute += rv;
        }
        const size_t c = tn * q / nth, d = tn * (q + 1) / nth;
        uint64_t tb = 0;
        for (size_t x = c; x < d; ++x) tb |= (uint64_t)transfer[x];
        P.t_bits = tb;
    };
    std::vector<std::thread> pool;
    if (nth == 1) {
        check(0);
    } else {
        pool.reserve(nth);
        for (int q = 0; q < nth; ++q) pool.emplace_back(check, q);
    }
    const pp_status tables = build_host_tables(n, W, parent, weight, mode, budget, inst);
    for (auto &th : pool) th.join();
    u128 total = 0, sum_demand = 0, sum_recompute = 0;
    uint64_t dr_bits = 0, t_bits = 0;
    for (const Part &P : parts) {
        total = std::min<u128>(total + P.total, cap);
        sum_demand += P.demand;
        sum_recompute += P.recompute;
        dr_bits |= P.dr_bits;
        t_bits |= P.t_bits;
    }
    if (dr_bits >> 63) return fail(PP_EINVAL, "negative demand or recompute cost");
    if (t_bits >> 63) return fail(PP_EINVAL, "negative transfer cost");
    const u128 lim = (u128)1 << 62;
    if (total > lim) return fail(PP_EOVERFLOW, "sum of demand * recompute exceeds 2^62");
    if (sum_demand > lim) return fail(PP_EOVERFLOW, "sum of demand exceeds 2^62");
    if (sum_recompute > lim) return fail(PP_EOVERFLOW, "sum of recompute costs exceeds 2^62");
    if (tables != PP_OK) return tables;

    PP_CUDA(cudaGetDevice(&inst->device));
    PP_CUDA(cudaDeviceGetAttribute(&inst->sm_count, cudaDevAttrMultiProcessorCount, inst->device));
    pp_status s;
    if ((s = upload(&inst->d_order, inst->h_order.data(), n, st))) return s;
    if ((s = upload(&inst->d_next, inst->h_next.data(), n, st))) return s;
    if ((s = upload(&inst->d_wpre, inst->h_wpre.data(), n, st))) return s;
    if ((s = upload(&inst->d_meta, inst->h_meta.data(), n, st))) return s;
    if ((s = upload(&inst->d_wave, inst->h_wave.data(), n, st))) return s;
    {
        // for the parent x of each position: the preorder range [x + 1, next(x))
        // of x's strict descendants (the pruned sweep's test)
        std::vector<int32_t> pos(n);
        std::vector<int2> span(n);
        for (int32_t i = 0; i < n; ++i) pos[inst->h_order[i]] = i;
        for (int32_t i = 0; i < n; ++i) {
            const int32_t par = parent[inst->h_order[i]];
            span[i] = par < 0 ? make_int2(-1, -1) : make_int2(pos[par] + 1, inst->h_next[pos[par]]);
        }
        if ((s = upload(&inst->d_pspan, span.data(), n, st))) return s;
        PP_CUDA(cudaStreamSynchronize(st));          // the host vectors die here
    }
    if ((s = upload(&inst->d_budget, budget, W, st))) return s;
    PP_CUDA(cudaMalloc(&inst->d_status, sizeof(int32_t)));
    PP_CUDA(cudaMemsetAsync(inst->d_status, 0, sizeof(int32_t), st));

    // recompute and transfer costs stay resident (by node id) for the epoch
    // update's materialisation cost; demand is needed only here
    int64_t *d_dem = nullptr;
    if ((s = upload(&d_dem, demand, Wn, st))) return s;
    if ((s = upload(&inst->d_rec, recompute, Wn, st))) { cudaFree(d_dem); return s; }
    if ((s = upload(&inst->d_tr, transfer, tn, st))) { cudaFree(d_dem); return s; }
    int64_t *const d_rec = inst->d_rec, *const d_tr = inst->d_tr;
    cudaError_t e = cudaSuccess;
    int blocks = (int)((n + 255) / 256);
    if (blocks > 4 * inst->sm_count) blocks = 4 * inst->sm_count;
    if (blocks < 1) blocks = 1;
    if (mode == PP_TRANSFER_REQUESTER) {
        e = cudaMalloc(&inst->d_a, sizeof(int64_t) * (Wn ? Wn : 1));
        if (e == cudaSuccess) e = cudaMalloc(&inst->d_delta, sizeof(int64_t) * (n ? n : 1));
        if (e == cudaSuccess) e = cudaMalloc(&inst->d_own, sizeof(int64_t) * (Wn ? Wn : 1));
        if (e == cudaSuccess) e = cudaMalloc(&inst->d_pop, sizeof(int64_t) * (Wn ? Wn : 1));
        if (e == cudaSuccess && n > 0)
            k_gain_requester<<<blocks, 256, 0, st>>>(n, W, inst->d_order, d_dem, d_rec, d_tr,
                                                     inst->d_a, inst->d_delta, inst->d_own, inst->d_pop);
    } else {
        e = cudaMalloc(&inst->d_g, sizeof(int64_t) * (tn ? tn : 1));
        if (e == cudaSuccess && n > 0) {
            dim3 grid((unsigned)((blocks + W * W - 1) / (W * W) + 1), (unsigned)(W * W));
            k_gain_source<<<grid, 256, 0, st>>>(n, W, inst->d_order, d_dem, d_rec, d_tr, inst->d_g);
        }
    }
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    cudaFree(d_dem);
    if (e != cudaSuccess) return cuda_fail(e, "gain precompute");
    return PP_OK;
}

extern "C" pp_status pp_instance_create(int32_t n, int32_t W, const int32_t *parent,
                                        const int32_t *weight, const int64_t *demand,
                                        const int64_t *recompute, const int64_t *transfer,
                                        int32_t transfer_mode, const int32_t *budget, void *stream,
                                        pp_instance **out)
{
    if (!out) return fail(PP_EINVAL, "out is null");
    *out = nullptr;
    pp_instance *inst = new (std::nothrow) pp_instance();
    if (!inst) return fail(PP_ENOMEM, "host allocation failed");
    pp_status s = create_impl(n, W, parent, weight, demand, recompute, transfer, transfer_mode,
                              budget, (cudaStream_t)stream, inst);
    if (s != PP_OK) {
        pp_instance_destroy(inst);
        return s;
    }
    *out = inst;
    return PP_OK;
}

extern "C" pp_status pp_instance_preorder(const pp_instance *inst, int32_t *order, int32_t *next,
                                          int32_t *stack_depth)
{
    if (!inst) return fail(PP_EINVAL, "null instance");
    if (inst->n > 0 && (!order || !next)) return fail(PP_EINVAL, "null output");
    if (inst->n > 0) {
        std::memcpy(order, inst->h_order.data(), sizeof(int32_t) * inst->n);
        std::memcpy(next, inst->h_next.data(), sizeof(int32_t) * inst->n);
    }
    if (stack_depth) *stack_depth = inst->stack_depth;
    return PP_OK;
}

extern "C" pp_status pp_row_plan(int32_t n, const int32_t *parent, int32_t *order, int32_t *next,
                                 int32_t *skip_code, int32_t *push_level, int32_t *stack_depth)
{
    if (n < 0) return fail(PP_EINVAL, "n must be >= 0");
    if (n > 0 && (!parent || !order || !next || !skip_code || !push_level))
        return fail(PP_EINVAL, "null pointer");
    for (int32_t v = 0; v < n; ++v)
        if (parent[v] < -1 || parent[v] >= n || parent[v] == v)
            return fail(PP_ENOTTREE, "parent id out of range or self-parent at node " + std::to_string(v));
    std::vector<int32_t> o, nx, meta;
    if (!build_preorder(n, parent, o, nx)) return fail(PP_ENOTTREE, "parent array contains a cycle");
    int32_t depth = 0;
    if (!build_row_meta(n, nx, meta, &depth)) return fail(PP_EINVAL, "skip-row stack deeper than supported");
    for (int32_t i = 0; i < n; ++i) {
        order[i] = o[i];
        next[i] = nx[i];
        skip_code[i] = meta_skip(meta[i]);
        push_level[i] = meta_push(meta[i]);
    }
    if (stack_depth) *stack_depth = depth;
    return PP_OK;
}

extern "C" pp_status pp_row_plan_registers(int32_t n, const int32_t *parent, const int32_t *weight,
                                           int32_t *code)
{
    if (n < 0) return fail(PP_EINVAL, "n must be >= 0");
    if (n > 0 && (!parent || !weight || !code)) return fail(PP_EINVAL, "null pointer");
    for (int32_t v = 0; v < n; ++v) {
        if (parent[v] < -1 || parent[v] >= n || parent[v] == v)
            return fail(PP_ENOTTREE, "parent id out of range or self-parent at node " + std::to_string(v));
        if (weight[v] < 1) return fail(PP_EINVAL, "chunk weight must be >= 1");
    }
    std::vector<int32_t> o, nx, meta, wave, wpre(n);
    if (!build_preorder(n, parent, o, nx)) return fail(PP_ENOTTREE, "parent array contains a cycle");
    for (int32_t i = 0; i < n; ++i) wpre[i] = weight[o[i]];
    int32_t depth = 0;
    if (!build_row_meta(n, nx, meta, &depth, &wpre, &wave))
        return fail(PP_EINVAL, "skip-row stack deeper than supported");
    for (int32_t i = 0; i < n; ++i) code[i] = wave[i];
    return PP_OK;
}

extern "C" pp_status pp_instance_sync(pp_instance *inst, void *stream)
{
    if (!inst) return fail(PP_EINVAL, "null instance");
    PP_CUDA(cudaStreamSynchronize((cudaStream_t)stream));
    int32_t v = 0;
    PP_CUDA(cudaMemcpy(&v, inst->d_status, sizeof(v), cudaMemcpyDeviceToHost));
    PP_CUDA(cudaMemset(inst->d_status, 0, sizeof(int32_t)));
    if (v == PP_ETIMEOUT) return fail(PP_ETIMEOUT, "a bounded device wait ran out");
    if (v == PP_EBOUNDS) return fail(PP_EBOUNDS, "device bounds check failed (budget or worker id)");
    if (v != 0) return fail(PP_ECUDA, "unknown device status " + std::to_string(v));
    return PP_OK;
}
