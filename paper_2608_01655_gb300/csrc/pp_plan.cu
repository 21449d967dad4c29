// pp_plan_run: Algorithm 1 (procedure PrefixPlace) with the S start orders as
// the batch axis.  Each step t processes worker pi_s[t] of every start s at
// once:  marginals (Eq. 10 / Eq. 7) -> tree DP (Eq. 9) -> traceback with the
// accept-and-update test fused in.  The greedy pass always accepts
// (WorkerGreedy, Theorem 3); a refinement sweep accepts only strict
// improvements (Section IV-C), and a start whose sweep accepted nothing stops
// (its later kernels return at once).  Holder sets live on the device as one
// 32-bit mask per chunk and start, in preorder.
#include <algorithm>
#include <cstdlib>
#include <cstring>
#include <numeric>

#include "pp_internal.cuh"

namespace pp {

// automatic choice of the top-2 marginals: whenever the tables (17 bytes per
// start, requester and chunk) fit in this much device memory
constexpr size_t kTop2MaxBytes = (size_t)16 << 30;

// per-sweep bookkeeping: a start that accepted nothing is done
__global__ void k_sweep_end(int S, int32_t *active, int32_t *improved, int32_t *sweeps)
{
    int s = blockIdx.x * blockDim.x + threadIdx.x;
    if (s < S && active[s]) {
        sweeps[s] += 1;
        active[s] = improved[s];
        improved[s] = 0;                // for the next sweep
    }
}

// streams of the per-start schedule (starts beyond share them round-robin)
constexpr int kPlanStreams = 32;

static pp_status ensure_plan_streams(pp_instance *inst, int ns)
{
    while ((int)inst->plan_streams.size() < ns) {
        cudaStream_t x;
        cudaEvent_t e;
        PP_CUDA(cudaStreamCreateWithFlags(&x, cudaStreamNonBlocking));
        inst->plan_streams.push_back(x);
        PP_CUDA(cudaEventCreateWithFlags(&e, cudaEventDisableTiming));
        inst->plan_join.push_back(e);
    }
    if (!inst->plan_fork) PP_CUDA(cudaEventCreateWithFlags(&inst->plan_fork, cudaEventDisableTiming));
    return PP_OK;
}

// CUDA_DEVICE_MAX_CONNECTIONS as the process sees it now (8 when unset); the
// driver reads it when the context is created
static int hardware_queues()
{
    const char *e = std::getenv("CUDA_DEVICE_MAX_CONNECTIONS");
    const int c = e ? std::atoi(e) : 8;
    return c > 0 ? c : 8;
}

// SplitMix64 (Steele, Lea and Flood, OOPSLA 2014)
static uint64_t splitmix64(uint64_t &x)
{
    uint64_t z = (x += 0x9E3779B97F4A7C15ULL);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

struct PlanBuffers {
    uint32_t *mask;      // [B][n]
    int64_t *profit;     // [B][n]
    int64_t *best;       // [B]
    int64_t *oldsum;     // [B]
    int64_t *obj;        // [B]
    int32_t *active;     // [B]
    int32_t *improved;   // [B]
    int32_t *accepted;   // [B]
    int32_t *sweeps;     // [B]
    int32_t *work;       // [W + 1][B]: step workers, then standalone ids
    int32_t *kbud;       // [W + 1][B]: step budgets, then standalone budgets
    unsigned long long *rows;   // [1] DP rows swept (pruned sweep) over the plan
};

static size_t align_up(size_t x) { return (x + 255) & ~(size_t)255; }

static pp_status plan_buffers(pp_instance *inst, int B, PlanBuffers *pb)
{
    const size_t n = (size_t)std::max(inst->n, 1);
    const int W = inst->W;
    size_t off[12], tot = 0;
    const size_t sz[12] = {4 * n * B, 8 * n * B, 8 * (size_t)B, 8 * (size_t)B, 8 * (size_t)B,
                           4 * (size_t)B, 4 * (size_t)B, 4 * (size_t)B, 4 * (size_t)B,
                           4 * (size_t)(W + 1) * B, 4 * (size_t)(W + 1) * B, 8};
    for (int x = 0; x < 12; ++x) {
        off[x] = tot;
        tot += align_up(sz[x]);
    }
    pp_status s = ensure_scratch(inst->plan, tot);
    if (s != PP_OK) return s;
    char *base = reinterpret_cast<char *>(inst->plan.ptr);
    pb->mask = reinterpret_cast<uint32_t *>(base + off[0]);
    pb->profit = reinterpret_cast<int64_t *>(base + off[1]);
    pb->best = reinterpret_cast<int64_t *>(base + off[2]);
    pb->oldsum = reinterpret_cast<int64_t *>(base + off[3]);
    pb->obj = reinterpret_cast<int64_t *>(base + off[4]);
    pb->active = reinterpret_cast<int32_t *>(base + off[5]);
    pb->improved = reinterpret_cast<int32_t *>(base + off[6]);
    pb->accepted = reinterpret_cast<int32_t *>(base + off[7]);
    pb->sweeps = reinterpret_cast<int32_t *>(base + off[8]);
    pb->work = reinterpret_cast<int32_t *>(base + off[9]);
    pb->kbud = reinterpret_cast<int32_t *>(base + off[10]);
    pb->rows = reinterpret_cast<unsigned long long *>(base + off[11]);
    return PP_OK;
}

pp_status plan_impl(pp_instance *inst, int32_t S, const int32_t *orders, int32_t R,
                    uint8_t *placement, int64_t *objective, pp_plan_stats *stats,
                    cudaStream_t st, bool orders_only)
{
    const int32_t n = inst->n, W = inst->W;
    if (stats && (stats->schedule < 0 || stats->schedule > 2)) return fail(PP_EINVAL, "schedule must be 0, 1 or 2");
    int launches = 0;
    int64_t standalone_cells = 0;
    int32_t maxk = 0;
    int64_t sumk = 0;
    for (int32_t m = 0; m < W; ++m) {
        maxk = std::max(maxk, inst->h_budget[m]);
        sumk += inst->h_budget[m];
    }
    // launch geometry of the start batch and of the standalone-score batch
    DpGeom g, gw;
    if (!dp_geometry(inst, maxk, &g, S) || !dp_geometry(inst, maxk, &gw, W))
        return fail(PP_EINVAL, "budget too large for the DP kernel");
    const int B = std::max(S, W);
    PlanBuffers pb;
    pp_status s = plan_buffers(inst, B, &pb);
    if (s != PP_OK) return s;
    s = ensure_scratch(inst->plan_bits, std::max(dp_work_bytes(S, n, g.words), dp_work_bytes(W, n, gw.words)));
    if (s != PP_OK) return s;
    const DpWork work = dp_work_split(inst->plan_bits.ptr, S, n, g.words);
    const DpWork work_w = dp_work_split(inst->plan_bits.ptr, W, n, gw.words);
    unsigned long long *rows_kept = pb.rows;
    PP_CUDA(cudaMemsetAsync(rows_kept, 0, sizeof(unsigned long long), st));

    // optional per-phase timing: events around every launch, read once at the end
    const bool timing = stats && stats->time_phases;
    int32_t dp_launches = 0;
    std::vector<cudaEvent_t> ev;        // lock step: every mark; per-start streams: the standalone step
    size_t pool_used = 0;
    auto take = [&](cudaEvent_t *e) -> pp_status {
        if (pool_used == inst->phase_events.size()) {
            cudaEvent_t x;
            PP_CUDA(cudaEventCreate(&x));
            inst->phase_events.push_back(x);
        }
        *e = inst->phase_events[pool_used++];
        return PP_OK;
    };
    auto mark = [&]() -> pp_status {
        if (!timing) return PP_OK;
        cudaEvent_t e;
        pp_status r = take(&e);
        if (r) return r;
        ev.push_back(e);
        PP_CUDA(cudaEventRecord(e, st));
        return PP_OK;
    };

    // ---- start orders -----------------------------------------------------
    std::vector<int32_t> ord((size_t)S * W);
    if (orders) {
        for (int32_t x = 0; x < S; ++x) {
            std::vector<int> seen(W, 0);
            for (int32_t t = 0; t < W; ++t) {
                int32_t h = orders[(size_t)x * W + t];
                if (h < 0 || h >= W || seen[h]++) return fail(PP_EINVAL, "orders must be permutations of 0..W-1");
            }
        }
        std::memcpy(ord.data(), orders, sizeof(int32_t) * ord.size());
    } else {
        for (int32_t x = 0; x < S; ++x)
            std::iota(ord.begin() + (size_t)x * W, ord.begin() + (size_t)(x + 1) * W, 0);
        if (S > 1) {
            // standalone score of every worker: its DP optimum with no other holder
            std::vector<int32_t> ids(W), kb(W);
            std::iota(ids.begin(), ids.end(), 0);
            for (int32_t m = 0; m < W; ++m) kb[m] = inst->h_budget[m];
            int32_t *d_ids = pb.work + (size_t)W * B, *d_kb = pb.kbud + (size_t)W * B;
            PP_CUDA(cudaMemcpyAsync(d_ids, ids.data(), 4 * W, cudaMemcpyHostToDevice, st));
            PP_CUDA(cudaMemcpyAsync(d_kb, kb.data(), 4 * W, cudaMemcpyHostToDevice, st));
            PP_CUDA(cudaMemsetAsync(pb.mask, 0, (size_t)4 * std::max(n, 1) * W, st));
            if ((s = mark())) return s;
            if ((s = launch_marginals(inst, W, d_ids, pb.mask, false, nullptr, pb.profit, nullptr, st))) return s;
            if ((s = mark())) return s;
            if ((s = launch_tree_dp(inst, W, pb.profit, false, d_kb, nullptr, gw, pb.best, work_w, st, maxk,
                                    rows_kept)))
                return s;
            if ((s = mark())) return s;
            if ((s = mark())) return s;   // no traceback for the standalone scores
            launches += 3 + (gw.split ? 1 : 0);     // a split DP is two launches
            dp_launches += 1;
            std::vector<int64_t> score(W);
            standalone_cells = (int64_t)n * sumk;
            PP_CUDA(cudaMemcpyAsync(score.data(), pb.best, 8 * W, cudaMemcpyDeviceToHost, st));
            PP_CUDA(cudaStreamSynchronize(st));
            std::vector<int32_t> o(W);
            std::iota(o.begin(), o.end(), 0);
            std::stable_sort(o.begin(), o.end(), [&](int32_t x, int32_t y) { return score[x] > score[y]; });
            std::copy(o.begin(), o.end(), ord.begin());
            std::copy(o.rbegin(), o.rend(), ord.begin() + W);
            for (int32_t x = 2; x < S; ++x) {
                int32_t *q = ord.data() + (size_t)x * W;
                uint64_t sm = (uint64_t)x;
                for (int32_t i = W - 1; i >= 1; --i) {
                    int32_t j = (int32_t)(splitmix64(sm) % (uint64_t)(i + 1));
                    std::swap(q[i], q[j]);
                }
            }
        }
    }
    if (stats && stats->orders_used) std::memcpy(stats->orders_used, ord.data(), sizeof(int32_t) * ord.size());
    if (orders_only) return PP_OK;

    // ---- per-step worker / budget tables: work[t][s] = pi_s[t] -------------
    std::vector<int32_t> hw((size_t)W * B, 0), hk((size_t)W * B, 0);
    for (int32_t t = 0; t < W; ++t)
        for (int32_t x = 0; x < S; ++x) {
            int32_t h = ord[(size_t)x * W + t];
            hw[(size_t)t * B + x] = h;
            hk[(size_t)t * B + x] = inst->h_budget[h];
        }
    PP_CUDA(cudaMemcpyAsync(pb.work, hw.data(), 4 * hw.size(), cudaMemcpyHostToDevice, st));
    PP_CUDA(cudaMemcpyAsync(pb.kbud, hk.data(), 4 * hk.size(), cudaMemcpyHostToDevice, st));
    std::vector<int32_t> ones(S, 1);
    PP_CUDA(cudaMemcpyAsync(pb.active, ones.data(), 4 * S, cudaMemcpyHostToDevice, st));
    PP_CUDA(cudaMemsetAsync(pb.mask, 0, (size_t)4 * std::max(n, 1) * S, st));
    PP_CUDA(cudaMemsetAsync(pb.accepted, 0, 4 * S, st));
    PP_CUDA(cudaMemsetAsync(pb.sweeps, 0, 4 * S, st));

    int dp_count = standalone_cells ? W : 0;
    int64_t cells = standalone_cells;
    // source-dependent marginals: scan each chunk's holders, or keep top-2
    // holder tables (Section IV-C); automatic = top-2 when the tables fit
    const int mreq = stats ? stats->marginals : 0;
    if (mreq < 0 || mreq > 2) return fail(PP_EINVAL, "stats->marginals must be 0, 1 or 2");
    const bool use_top2 = inst->mode == PP_TRANSFER_SOURCE && n > 0 &&
                          (mreq == 2 || (mreq == 0 && (size_t)S * W * n * 17 <= kTop2MaxBytes));
    Top2 t2;
    if (use_top2) {
        const size_t tw = (size_t)S * W * n, a = 255;
        const size_t b1 = (8 * tw + a) & ~a, b2 = b1 + ((8 * tw + a) & ~a), b3 = b2 + ((tw + a) & ~a);
        if ((s = ensure_scratch(inst->top2, b3 + (size_t)S * n))) return s;
        char *base = reinterpret_cast<char *>(inst->top2.ptr);
        t2.v1 = reinterpret_cast<int64_t *>(base);
        t2.v2 = reinterpret_cast<int64_t *>(base + b1);
        t2.l1 = reinterpret_cast<int8_t *>(base + b2);
        t2.oldbit = reinterpret_cast<uint8_t *>(base + b3);
        PP_CUDA(cudaMemsetAsync(base, 0, b2, st));                 // v1 = v2 = 0: no holders yet
        PP_CUDA(cudaMemsetAsync(t2.l1, 0xFF, tw, st));             // l1 = -1
        PP_CUDA(cudaMemsetAsync(t2.oldbit, 0, (size_t)S * n, st)); // nobody holds anything yet
    }
    PP_CUDA(cudaMemsetAsync(pb.improved, 0, 4 * S, st));
    // The first greedy update of every start runs against an empty placement,
    // so its marginals and its DP are exactly the standalone-score DP of its
    // worker, computed above for the default orders: the start walks those
    // decision bits (one batched traceback, item s reading DP item pi_s[0] of
    // the standalone workspace) instead of running that DP again.
    const bool reuse = standalone_cells > 0;
    int64_t reused_cells = 0;
    if (reuse)
        for (int32_t x = 0; x < S; ++x) reused_cells += (int64_t)n * inst->h_budget[ord[(size_t)x * W]];
    auto first_from_standalone = [&]() -> pp_status {
        pp_status r;
        if ((r = mark())) return r;
        if ((r = mark())) return r;       // no marginal pass
        if ((r = mark())) return r;       // no DP
        AcceptArgs a;
        a.worker = pb.work;               // step 0: pi_s[0]
        a.best = pb.best;
        a.oldsum = pb.oldsum;
        a.active = pb.active;
        a.improved = pb.improved;
        a.accepted = pb.accepted;
        a.mask = pb.mask;
        a.greedy = 1;
        a.bits_item = pb.work;
        if ((r = launch_traceback(inst, S, work_w, gw, pb.kbud, nullptr, &a, st))) return r;
        if ((r = mark())) return r;
        launches += 1;
        return PP_OK;
    };
    // lock step unless asked for per-start streams, or (automatic) unless every
    // start's stream gets a hardware queue of its own: streams that share a
    // queue wait on one another's launches, which costs more than lock step
    const int32_t sched = stats ? stats->schedule : 0;
    const bool lockstep = S == 1 || sched == 1 ||
                          (sched == 0 && hardware_queues() < std::min<int>(S, kPlanStreams));
    int32_t start_steps = 0;            // per-start streams: updates launched per start
    std::vector<std::vector<cudaEvent_t>> sev;   // per-start streams: each start's phase events
    if (lockstep) {
        const int32_t *prev_wk = nullptr;     // top-2: worker of the previous step, per start
        auto step = [&](int t, int greedy) -> pp_status {
            const int32_t *wk = pb.work + (size_t)t * B;
            const int32_t *kb = pb.kbud + (size_t)t * B;
            pp_status r;
            if ((r = mark())) return r;
            if (use_top2) {
                // the previous step's change is folded into this step's marginal pass
                r = launch_marginals_top2(inst, S, prev_wk, wk, pb.mask, pb.active, t2, pb.profit, pb.oldsum, st);
                prev_wk = wk;
            } else {
                r = launch_marginals(inst, S, wk, pb.mask, false, pb.active, pb.profit, pb.oldsum, st);
            }
            if (r) return r;
            if ((r = mark())) return r;
            if ((r = launch_tree_dp(inst, S, pb.profit, false, kb, pb.active, g, pb.best, work, st, maxk, rows_kept)))
                return r;
            if ((r = mark())) return r;
            AcceptArgs a;
            a.worker = wk;
            a.best = pb.best;
            a.oldsum = pb.oldsum;
            a.active = pb.active;
            a.improved = pb.improved;
            a.accepted = pb.accepted;
            a.mask = pb.mask;
            a.greedy = greedy;
            if ((r = launch_traceback(inst, S, work, g, kb, nullptr, &a, st))) return r;
            if ((r = mark())) return r;
            launches += 4 + (g.split ? 1 : 0);
            dp_launches += 1;
            return PP_OK;
        };

        // WorkerGreedy pass
        for (int32_t t = 0; t < W; ++t) {
            if (t == 0 && reuse) {
                if ((s = first_from_standalone())) return s;
                prev_wk = pb.work;        // top-2: step 0's change is folded in at step 1
                continue;
            }
            if ((s = step(t, 1))) return s;
        }
        dp_count += S * W - (reuse ? S : 0);
        cells += (int64_t)S * n * sumk - reused_cells;

        // coordinate refinement
        std::vector<int32_t> act(S, 1);
        for (int32_t r = 0; r < R; ++r) {
            int nact = 0;
            for (int32_t x = 0; x < S; ++x) nact += act[x] != 0;
            if (nact == 0) break;
            PP_CUDA(cudaMemsetAsync(pb.improved, 0, 4 * S, st));
            for (int32_t t = 0; t < W; ++t)
                if ((s = step(t, 0))) return s;
            dp_count += nact * W;
            cells += (int64_t)nact * n * sumk;
            k_sweep_end<<<(S + 127) / 128, 128, 0, st>>>(S, pb.active, pb.improved, pb.sweeps);
            PP_CUDA(cudaGetLastError());
            launches += 1;
            PP_CUDA(cudaMemcpyAsync(act.data(), pb.active, 4 * S, cudaMemcpyDeviceToHost, st));
            PP_CUDA(cudaStreamSynchronize(st));
        }
    } else {
        // Every start on its own stream: start s runs its W (1 + R) updates
        // back to back and never waits for a slower start (in lock step each
        // step waits for the start with the most kept rows).  Each update is
        // the same kernels at batch one on the start's slice of every buffer,
        // in the batch's launch shape (no split: a launch holds one item).
        // All R sweeps are enqueued; a start whose sweep accepted nothing is
        // inactive from then on and its later kernels return at once.
        const int NS = std::min(S, kPlanStreams);
        if ((s = ensure_plan_streams(inst, NS))) return s;
        if ((s = ensure_dp_stack(inst, g, S))) return s;   // one stack slot per start, allocated up front
        DpGeom g1 = g;
        g1.split = 0;
        {
            // more than half an SM's shared memory per CTA: two DP CTAs on one SM
            // slow each other down (~25% per row); with one per SM a start whose
            // cluster finds no room waits instead (plan 208.6 -> 205.6 ms)
            int per_sm = 0, optin = 0;
            PP_CUDA(cudaDeviceGetAttribute(&per_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, inst->device));
            PP_CUDA(cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, inst->device));
            g1.smem = std::max(g1.smem, (size_t)std::min(per_sm / 2, optin));
        }
        if (reuse && (s = first_from_standalone())) return s;     // on the caller's stream, before the fork
        PP_CUDA(cudaEventRecord(inst->plan_fork, st));
        for (int x = 0; x < NS; ++x) PP_CUDA(cudaStreamWaitEvent(inst->plan_streams[x], inst->plan_fork, 0));
        std::vector<const int32_t *> prev(S, nullptr);
        sev.resize(timing ? S : 0);
        auto smark = [&](int x, cudaStream_t sx) -> pp_status {
            if (!timing) return PP_OK;
            cudaEvent_t e;
            pp_status r = take(&e);
            if (r) return r;
            sev[x].push_back(e);
            PP_CUDA(cudaEventRecord(e, sx));
            return PP_OK;
        };
        const size_t N = (size_t)std::max(n, 1);
        for (int q = 0; q < W * (1 + R); ++q) {
            const int pass = q / W, t = q % W;
            if (q == 0 && reuse) {
                for (int x = 0; x < S; ++x) prev[x] = pb.work + x;    // top-2: folded in at step 1
                continue;
            }
            for (int x = 0; x < S; ++x) {
                cudaStream_t sx = inst->plan_streams[x % NS];
                const int32_t *wk = pb.work + (size_t)t * B + x;
                const int32_t *kb = pb.kbud + (size_t)t * B + x;
                uint32_t *mk = pb.mask + (size_t)x * N;
                int64_t *pf = pb.profit + (size_t)x * N;
                if ((s = smark(x, sx))) return s;
                if (use_top2) {
                    Top2 tx = t2;
                    tx.v1 += (size_t)x * W * N;
                    tx.v2 += (size_t)x * W * N;
                    tx.l1 += (size_t)x * W * N;
                    tx.oldbit += (size_t)x * N;
                    s = launch_marginals_top2(inst, 1, prev[x], wk, mk, pb.active + x, tx, pf, pb.oldsum + x, sx);
                    prev[x] = wk;
                } else {
                    s = launch_marginals(inst, 1, wk, mk, false, pb.active + x, pf, pb.oldsum + x, sx);
                }
                if (s) return s;
                if ((s = smark(x, sx))) return s;
                const DpWork wx = dp_work_item(work, x, n, g.words);
                if ((s = launch_tree_dp(inst, 1, pf, false, kb, pb.active + x, g1, pb.best + x, wx, sx, maxk,
                                        rows_kept, x)))
                    return s;
                if ((s = smark(x, sx))) return s;
                AcceptArgs a;
                a.worker = wk;
                a.best = pb.best + x;
                a.oldsum = pb.oldsum + x;
                a.active = pb.active + x;
                a.improved = pb.improved + x;
                a.accepted = pb.accepted + x;
                a.mask = mk;
                a.greedy = pass == 0;
                if ((s = launch_traceback(inst, 1, wx, g1, kb, nullptr, &a, sx))) return s;
                if ((s = smark(x, sx))) return s;
                launches += 4;
                if (pass > 0 && t == W - 1) {
                    k_sweep_end<<<1, 32, 0, sx>>>(1, pb.active + x, pb.improved + x, pb.sweeps + x);
                    PP_CUDA(cudaGetLastError());
                    launches += 1;
                }
            }
        }
        start_steps = W * (1 + R);
        for (int x = 0; x < NS; ++x) {
            PP_CUDA(cudaEventRecord(inst->plan_join[x], inst->plan_streams[x]));
            PP_CUDA(cudaStreamWaitEvent(st, inst->plan_join[x], 0));
        }
    }

    // objective of every candidate, argmax (ties to the lowest start)
    if ((s = launch_objective(inst, S, pb.mask, nullptr, pb.obj, st))) return s;
    launches += 1;
    std::vector<int64_t> obj(S);
    std::vector<int32_t> sw(S), acc(S);
    unsigned long long rows_swept = 0;
    PP_CUDA(cudaMemcpyAsync(&rows_swept, rows_kept, sizeof(rows_swept), cudaMemcpyDeviceToHost, st));
    PP_CUDA(cudaMemcpyAsync(obj.data(), pb.obj, 8 * S, cudaMemcpyDeviceToHost, st));
    PP_CUDA(cudaMemcpyAsync(sw.data(), pb.sweeps, 4 * S, cudaMemcpyDeviceToHost, st));
    PP_CUDA(cudaMemcpyAsync(acc.data(), pb.accepted, 4 * S, cudaMemcpyDeviceToHost, st));
    PP_CUDA(cudaStreamSynchronize(st));
    if (!lockstep) {
        // executed updates, from the sweeps each start ran (the greedy pass always runs)
        int64_t swsum = 0;
        for (int32_t x = 0; x < S; ++x) swsum += sw[x];
        dp_count += (int)(S * W + swsum * W) - (reuse ? S : 0);
        cells += ((int64_t)S + swsum) * n * sumk - reused_cells;
        dp_launches += (int32_t)((W * (S + swsum) - (reuse ? S : 0) + S / 2) / S);
    }
    int32_t bs = 0;
    for (int32_t x = 1; x < S; ++x)
        if (obj[x] > obj[bs]) bs = x;
    int64_t best_obj = obj[bs];
    const uint32_t *best_mask = pb.mask + (size_t)bs * n;
    // requester-side safeguard candidates S, S+1, S+2 (ties stay with the lower index)
    int64_t so[3] = {0, 0, 0};
    if (inst->mode == PP_TRANSFER_REQUESTER && !(stats && stats->no_safeguards)) {
        const uint32_t *sgm = nullptr;
        if ((s = safeguards_impl(inst, st, &sgm, so, &launches, &cells, &dp_launches))) return s;
        dp_count += 3 * W;
        for (int c = 0; c < 3; ++c)
            if (so[c] > best_obj) {
                best_obj = so[c];
                bs = S + c;
                best_mask = sgm + (size_t)c * n;
            }
    }
    std::vector<uint32_t> mk(std::max(n, 1));
    if (n > 0) {
        PP_CUDA(cudaMemcpyAsync(mk.data(), best_mask, 4 * (size_t)n, cudaMemcpyDeviceToHost, st));
        PP_CUDA(cudaStreamSynchronize(st));
    }
    std::memset(placement, 0, (size_t)W * n);
    for (int32_t i = 0; i < n; ++i) {
        const int32_t b = inst->h_order[i];
        uint32_t m = mk[i];
        while (m) {
            int h = __builtin_ctz(m);
            m &= m - 1;
            placement[(size_t)h * n + b] = 1;
        }
    }
    *objective = best_obj;
    if (stats) {
        if (stats->per_start_objective) std::copy(obj.begin(), obj.end(), stats->per_start_objective);
        if (stats->per_start_sweeps) std::copy(sw.begin(), sw.end(), stats->per_start_sweeps);
        if (stats->per_start_accepted) std::copy(acc.begin(), acc.end(), stats->per_start_accepted);
        stats->best_start = bs;
        stats->dp_count = dp_count;
        stats->dp_cells = cells;
        stats->kernel_launches = launches;
        stats->dp_rows_swept = (int64_t)rows_swept;
        stats->dp_launches = dp_launches;
        for (int c = 0; c < 3; ++c) stats->safeguard_objective[c] = so[c];
        stats->used_top2 = use_top2;
        stats->schedule = lockstep ? 1 : 2;
        stats->hw_queues = hardware_queues();
        stats->phase_ms[0] = stats->phase_ms[1] = stats->phase_ms[2] = 0.f;
        // groups of four marks: before the marginals, the DP and the traceback, and after
        auto add = [&](const std::vector<cudaEvent_t> &v, size_t from, size_t to, float scale) {
            to = std::min(to, v.size());       // no events without time_phases
            for (size_t x = from; x + 3 < to; x += 4) {
                float a = 0.f, b = 0.f, c = 0.f;
                cudaEventElapsedTime(&a, v[x], v[x + 1]);
                cudaEventElapsedTime(&b, v[x + 1], v[x + 2]);
                cudaEventElapsedTime(&c, v[x + 2], v[x + 3]);
                stats->phase_ms[0] += a * scale;
                stats->phase_ms[1] += b * scale;
                stats->phase_ms[2] += c * scale;
            }
        };
        if (lockstep) {
            add(ev, 0, ev.size(), 1.f);
        } else {
            // the standalone-score step (on the caller's stream), then the mean over starts
            add(ev, 0, standalone_cells ? 8 : 0, 1.f);      // with the batched first traceback
            for (const auto &v : sev) add(v, 0, v.size(), 1.f / (float)S);
        }
    }
    return PP_OK;
}

}  // namespace pp

using namespace pp;

extern "C" pp_status pp_plan_run(pp_instance *inst, int32_t n_starts, const int32_t *orders,
                                 int32_t max_rounds, uint8_t *placement, int64_t *objective,
                                 pp_plan_stats *stats, void *stream)
{
    if (!inst) return fail(PP_EINVAL, "null instance");
    if (n_starts < 1) return fail(PP_EINVAL, "n_starts must be >= 1");
    if (max_rounds < 0) return fail(PP_EINVAL, "max_rounds must be >= 0");
    if (!objective || (inst->n > 0 && !placement)) return fail(PP_EINVAL, "null output pointer");
    cudaStream_t st = (cudaStream_t)stream;
    pp_status s = plan_impl(inst, n_starts, orders, max_rounds, placement, objective, stats, st);
    if (s != PP_OK) return s;
    return pp_instance_sync(inst, stream);
}

extern "C" pp_status pp_default_orders(pp_instance *inst, int32_t n_starts, int32_t *orders, void *stream)
{
    if (!inst) return fail(PP_EINVAL, "null instance");
    if (n_starts < 1) return fail(PP_EINVAL, "n_starts must be >= 1");
    if (!orders) return fail(PP_EINVAL, "null output pointer");
    pp_plan_stats st = {};
    st.orders_used = orders;
    int64_t unused = 0;
    pp_status s = plan_impl(inst, n_starts, nullptr, 0, nullptr, &unused, &st, (cudaStream_t)stream, true);
    if (s != PP_OK) return s;
    return pp_instance_sync(inst, stream);
}
