// runtime.cpp -- host side of the C ABI in include/adpsgd.h: argument checks, the context,
// the ADPSGD period rule (Algorithm 2), the step-size schedule, the run loop and the bounded
// waits.  All device work goes through the library's kernels (kernels.cu, sync_step.cu,
// interval.cu, transfer.cu) on the caller's stream.
#include <cuda_runtime_api.h>

#include <algorithm>
#include <chrono>
#include <cstdint>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <thread>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "../../include/adpsgd.h"
#include "launch.h"

namespace {

thread_local std::string g_last_error;

// NVTX range for profiler timelines (header-only NVTX 3; a no-op without a tool attached).
struct NvtxRange {
    explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
};

int cuda_fail(cudaError_t e, const char* where)
{
    g_last_error = std::string(where) + ": " + cudaGetErrorName(e) + ": " + cudaGetErrorString(e);
    return ADPSGD_E_CUDA;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

constexpr int64_t kMaxK = int64_t(1) << 32;  // the step index is one 32-bit Philox counter word

int check_shard(const adpsgd_shard* sh)
{
    if (sh == nullptr || sh->shards < 1 || sh->index < 0 || sh->index >= sh->shards) return ADPSGD_E_INVAL;
    if (sh->col0 < 0 || sh->col0 % 4 != 0 || sh->P_total < sh->col0) return ADPSGD_E_INVAL;
    if (sh->shards > 1 && sh->gather == nullptr) return ADPSGD_E_INVAL;
    return ADPSGD_OK;
}

// Every shard's `count` doubles through shard->gather, added in shard order from 0.
int shard_combine(const adpsgd_shard* sh, const double* local, int64_t count, double* out)
{
    if (sh->gather == nullptr) {  // a single shard
        for (int64_t t = 0; t < count; ++t) out[t] = 0.0 + local[t];
        return ADPSGD_OK;
    }
    std::vector<double> all((size_t)count * (size_t)sh->shards, 0.0);
    const int rc = sh->gather(local, count, all.data(), sh->user);
    if (rc != 0) {
        g_last_error = "shard exchange failed with code " + std::to_string(rc);
        return ADPSGD_E_PEER;
    }
    for (int64_t t = 0; t < count; ++t) {
        double total = 0.0;
        for (int32_t r = 0; r < sh->shards; ++r) total += all[(size_t)r * (size_t)count + (size_t)t];
        out[t] = total;
    }
    return ADPSGD_OK;
}

}  // namespace

struct TimedLaunch {
    cudaEvent_t start, stop;
    int kind;  // 0 local step, 1 averaging, 2 fused interval, 3 fused sync step
};

struct adpsgd_ctx {
    adpsgd_config cfg{};
    float* x = nullptr;
    float* v = nullptr;
    const float* h = nullptr;
    const float* c = nullptr;
    const uint16_t* noise = nullptr;
    cudaStream_t stream = nullptr;
    int device = 0;
    int sms = 0;
    adpsgd::PhiloxKeys keys{};
    double* d_partials = nullptr;
    double* d_out = nullptr;  // D, loss, then the averaging kernel's completion counter (4 slots)
    double* h_out = nullptr;  // pinned copy of D and loss
    cudaEvent_t done = nullptr;
    double* d_var = nullptr;  // per-iteration variance slots (2 doubles each), grown on demand
    int64_t d_var_cap = 0;
    int grid_avg = 0, grid_avg_loss = 0, grid_var = 0, grid_interval = 0;
    int grid_sync = 0;  // > 0: the fused sync step is available (cfg.fuse_sync_step and supported)
    // kernel timing
    std::vector<cudaEvent_t> free_events;
    std::vector<TimedLaunch> pending;
    // per kernel kind: 0 local step, 1 averaging, 2 fused interval, 3 fused sync step
    double ms[4] = {0.0, 0.0, 0.0, 0.0};
    int64_t launches[4] = {0, 0, 0, 0};
    int64_t timed_launches[4] = {0, 0, 0, 0};
    bool force_incomplete = false;
    // column sharding (adpsgd_set_shard): the Philox block of column 0 and the exchange of the
    // partial sums (also used by a replica split)
    uint32_t q0 = 0;
    bool sharded = false;
    adpsgd_shard shard{};
    // replica split (adpsgd_set_replica_split): this process's first global replica, the
    // replicas of the whole problem, the averaging's column chunk and its grids
    bool replica = false;
    adpsgd_replica_split split{};
    uint32_t r0 = 0;
    int32_t n_total = 0;  // replicas of the whole problem (cfg.n unless split)
    int grid_chunk = 0, grid_chunk_loss = 0, grid_chunk_var = 0;
};

namespace {

int64_t timeout_ms(const adpsgd_ctx* ctx)
{
    return ctx->cfg.wait_timeout_ms > 0 ? ctx->cfg.wait_timeout_ms : 60000;
}

// Poll an event until it completes or the context's time limit passes.
int wait_event(adpsgd_ctx* ctx, cudaEvent_t ev)
{
    const auto t0 = std::chrono::steady_clock::now();
    const auto limit = std::chrono::milliseconds(timeout_ms(ctx));
    int spins = 0;
    for (;;) {
        cudaError_t e = ctx->force_incomplete ? cudaErrorNotReady : cudaEventQuery(ev);
        if (e == cudaSuccess) return ADPSGD_OK;
        if (e != cudaErrorNotReady) return cuda_fail(e, "cudaEventQuery");
        if (std::chrono::steady_clock::now() - t0 > limit) {
            g_last_error = "bounded wait ran out";
            return ADPSGD_E_TIMEOUT;
        }
        if (++spins > 2000) std::this_thread::sleep_for(std::chrono::microseconds(20));
    }
}

int take_event(adpsgd_ctx* ctx, cudaEvent_t* ev)
{
    if (!ctx->free_events.empty()) {
        *ev = ctx->free_events.back();
        ctx->free_events.pop_back();
        return ADPSGD_OK;
    }
    cudaError_t e = cudaEventCreate(ev);
    return e == cudaSuccess ? ADPSGD_OK : cuda_fail(e, "cudaEventCreate");
}

// Add up the elapsed times of all recorded launches (all of them must have completed).
int harvest_times(adpsgd_ctx* ctx)
{
    if (ctx->pending.empty()) return ADPSGD_OK;
    int st = wait_event(ctx, ctx->pending.back().stop);
    if (st != ADPSGD_OK) return st;
    for (const TimedLaunch& t : ctx->pending) {
        float ms = 0.0f;
        cudaError_t e = cudaEventElapsedTime(&ms, t.start, t.stop);
        if (e != cudaSuccess) return cuda_fail(e, "cudaEventElapsedTime");
        ctx->ms[t.kind] += ms;
        ctx->timed_launches[t.kind] += 1;
        ctx->free_events.push_back(t.start);
        ctx->free_events.push_back(t.stop);
    }
    ctx->pending.clear();
    return ADPSGD_OK;
}

template <typename Launch>
int timed(adpsgd_ctx* ctx, int kind, Launch launch, const char* what)
{
    cudaEvent_t a = nullptr, b = nullptr;
    // time_kernels = N > 0: bracket every N-th launch of each kind with events.
    const bool sample = ctx->cfg.time_kernels > 0 && ctx->launches[kind] % ctx->cfg.time_kernels == 0;
    if (sample) {
        if (ctx->pending.size() >= 16384) {
            int st = harvest_times(ctx);
            if (st != ADPSGD_OK) return st;
        }
        int st = take_event(ctx, &a);
        if (st != ADPSGD_OK) return st;
        st = take_event(ctx, &b);
        if (st != ADPSGD_OK) {
            ctx->free_events.push_back(a);
            return st;
        }
        cudaError_t e = cudaEventRecord(a, ctx->stream);
        if (e != cudaSuccess) {
            ctx->free_events.push_back(a);
            ctx->free_events.push_back(b);
            return cuda_fail(e, "cudaEventRecord");
        }
    }
    cudaError_t e = launch();
    if (e != cudaSuccess) {
        if (sample) {
            ctx->free_events.push_back(a);
            ctx->free_events.push_back(b);
        }
        return cuda_fail(e, what);
    }
    ctx->launches[kind] += 1;
    if (sample) {
        e = cudaEventRecord(b, ctx->stream);
        if (e != cudaSuccess) {
            ctx->free_events.push_back(a);
            ctx->free_events.push_back(b);
            return cuda_fail(e, "cudaEventRecord");
        }
        ctx->pending.push_back({a, b, kind});
    }
    return ADPSGD_OK;
}

int local_step(adpsgd_ctx* ctx, int64_t k, float gamma)
{
    adpsgd::LocalStepArgs a;
    a.x = ctx->x;
    a.v = ctx->v;
    a.h = ctx->h;
    a.c = ctx->c;
    a.noise_bf16 = ctx->cfg.noise_mode == ADPSGD_NOISE_BF16 ? ctx->noise : nullptr;
    a.keys = &ctx->keys;
    a.n = ctx->cfg.n;
    a.P = ctx->cfg.P;
    a.k = (uint32_t)k;
    a.q0 = ctx->q0;
    a.r0 = ctx->r0;
    a.gamma = gamma;
    a.mu = ctx->cfg.momentum;
    a.wd = ctx->cfg.weight_decay;
    a.sigma = ctx->cfg.noise_sigma;
    return timed(ctx, 0, [&] { return adpsgd::launch_local_step(a, ctx->stream); }, "local step");
}

// A replica split's sync: the caller's all-to-all into the chunk, the averaging (or variance)
// kernel on the chunk of all replicas, the copy of its two sums into ctx->h_out and ctx->done, and
// (write_back) the caller's all-gather of the chunks' means into x.
int replica_average_enqueue(adpsgd_ctx* ctx, bool write_back, bool loss)
{
    const adpsgd_replica_split& rs = ctx->split;
    if (rs.collective(ADPSGD_SCATTER_COLUMNS, rs.user) != 0) {
        g_last_error = "the replica split's all-to-all failed";
        return ADPSGD_E_PEER;
    }
    adpsgd::AverageArgs a;
    a.x = rs.chunk_x;
    a.h = loss ? ctx->h + rs.col0 : nullptr;
    a.c = loss ? ctx->c + rs.col0 : nullptr;
    a.n = rs.n_total;
    a.P = rs.P_chunk;
    a.write_back = write_back;
    a.partials = ctx->d_partials;
    a.out = ctx->d_out;
    a.counter = reinterpret_cast<unsigned int*>(ctx->d_out + 2);
    a.grid = !write_back ? ctx->grid_chunk_var : (loss ? ctx->grid_chunk_loss : ctx->grid_chunk);
    int st = timed(ctx, 1, [&] { return adpsgd::launch_average(a, ctx->stream); }, "average");
    if (st != ADPSGD_OK) return st;
    cudaError_t e = cudaMemcpyAsync(ctx->h_out, ctx->d_out, 2 * sizeof(double), cudaMemcpyDeviceToHost,
                                    ctx->stream);
    if (e == cudaSuccess) e = cudaEventRecord(ctx->done, ctx->stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync");
    if (write_back && rs.collective(ADPSGD_GATHER_AVERAGE, rs.user) != 0) {
        g_last_error = "the replica split's all-gather failed";
        return ADPSGD_E_PEER;
    }
    return ADPSGD_OK;
}

// Enqueue the averaging (write_back) or variance-only kernel and the copy of its two sums
// into ctx->h_out, then record ctx->done.
int average_enqueue(adpsgd_ctx* ctx, bool write_back, bool loss)
{
    if (ctx->replica) return replica_average_enqueue(ctx, write_back, loss);
    adpsgd::AverageArgs a;
    a.x = ctx->x;
    a.h = loss ? ctx->h : nullptr;
    a.c = loss ? ctx->c : nullptr;
    a.n = ctx->cfg.n;
    a.P = ctx->cfg.P;
    a.write_back = write_back;
    a.partials = ctx->d_partials;
    a.out = ctx->d_out;
    a.counter = reinterpret_cast<unsigned int*>(ctx->d_out + 2);
    a.grid = !write_back ? ctx->grid_var : (loss ? ctx->grid_avg_loss : ctx->grid_avg);
    int st = timed(ctx, 1, [&] { return adpsgd::launch_average(a, ctx->stream); }, "average");
    if (st != ADPSGD_OK) return st;
    cudaError_t e = cudaMemcpyAsync(ctx->h_out, ctx->d_out, 2 * sizeof(double), cudaMemcpyDeviceToHost,
                                    ctx->stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync");
    e = cudaEventRecord(ctx->done, ctx->stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
    return ADPSGD_OK;
}

// Variance of the current state into device slot k of ctx->d_var (no host round trip).
int variance_into_slot(adpsgd_ctx* ctx, int64_t k)
{
    adpsgd::AverageArgs a;
    a.x = ctx->x;
    a.h = nullptr;
    a.c = nullptr;
    a.n = ctx->cfg.n;
    a.P = ctx->cfg.P;
    a.write_back = false;
    a.partials = ctx->d_partials;
    a.out = ctx->d_var + 2 * k;
    a.counter = reinterpret_cast<unsigned int*>(ctx->d_out + 2);
    a.grid = ctx->grid_var;
    return timed(ctx, 1, [&] { return adpsgd::launch_average(a, ctx->stream); }, "variance");
}

// Averaging (write_back) or variance only; results land in ctx->h_out after a bounded wait.
int average(adpsgd_ctx* ctx, bool write_back, bool loss)
{
    int st = average_enqueue(ctx, write_back, loss);
    if (st != ADPSGD_OK) return st;
    return wait_event(ctx, ctx->done);
}

// D and the loss of the last averaging (ctx->h_out): this context's own sums, or for a shard of a
// column-split problem the totals over all shards in shard order.
int sync_sums(adpsgd_ctx* ctx, double* D, double* loss)
{
    if (!ctx->sharded) {
        *D = ctx->h_out[0];
        *loss = ctx->h_out[1];
        return ADPSGD_OK;
    }
    double total[2];
    const int st = shard_combine(&ctx->shard, ctx->h_out, 2, total);
    if (st != ADPSGD_OK) return st;
    *D = total[0];
    *loss = total[1];
    return ADPSGD_OK;
}

// Enqueue one fused interval: m local steps from step k0 (step sizes gamma[0..m)) and, if
// `average`, the averaging with the copy of its sums and ctx->done.
int interval(adpsgd_ctx* ctx, int64_t k0, int32_t m, const float* gamma, bool average, bool loss)
{
    adpsgd::IntervalArgs a;
    a.x = ctx->x;
    a.v = ctx->v;
    a.h = ctx->h;
    a.c = ctx->c;
    a.noise_bf16 = ctx->cfg.noise_mode == ADPSGD_NOISE_BF16 ? ctx->noise : nullptr;
    a.keys = &ctx->keys;
    a.n = ctx->cfg.n;
    a.P = ctx->cfg.P;
    a.k0 = (uint32_t)k0;
    a.q0 = ctx->q0;
    a.m = m;
    a.gamma = gamma;
    a.mu = ctx->cfg.momentum;
    a.wd = ctx->cfg.weight_decay;
    a.sigma = ctx->cfg.noise_sigma;
    a.average = average;
    a.loss = average && loss;
    a.partials = ctx->d_partials;
    a.out = ctx->d_out;
    a.counter = reinterpret_cast<unsigned int*>(ctx->d_out + 2);
    a.grid = ctx->grid_interval;
    int st = timed(ctx, 2, [&] { return adpsgd::launch_interval(a, ctx->stream); }, "interval");
    if (st != ADPSGD_OK || !average) return st;
    cudaError_t e = cudaMemcpyAsync(ctx->h_out, ctx->d_out, 2 * sizeof(double), cudaMemcpyDeviceToHost,
                                    ctx->stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync");
    e = cudaEventRecord(ctx->done, ctx->stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
    return ADPSGD_OK;
}

// Enqueue the local step of iteration k fused with the averaging that ends it (needs
// ctx->grid_sync > 0), the copy of the two sums into ctx->h_out, and ctx->done.
int sync_step_enqueue(adpsgd_ctx* ctx, int64_t k, float gamma, bool loss)
{
    adpsgd::SyncStepArgs a;
    a.x = ctx->x;
    a.v = ctx->v;
    a.h = ctx->h;
    a.c = ctx->c;
    a.noise_bf16 = ctx->noise;
    a.keys = &ctx->keys;
    a.n = ctx->cfg.n;
    a.P = ctx->cfg.P;
    a.k = (uint32_t)k;
    a.q0 = ctx->q0;
    a.gamma = gamma;
    a.mu = ctx->cfg.momentum;
    a.wd = ctx->cfg.weight_decay;
    a.sigma = ctx->cfg.noise_sigma;
    a.loss = loss;
    a.partials = ctx->d_partials;
    a.out = ctx->d_out;
    a.counter = reinterpret_cast<unsigned int*>(ctx->d_out + 2);
    a.grid = ctx->grid_sync;
    int st = timed(ctx, 3, [&] { return adpsgd::launch_sync_step(a, ctx->stream); }, "sync step");
    if (st != ADPSGD_OK) return st;
    cudaError_t e = cudaMemcpyAsync(ctx->h_out, ctx->d_out, 2 * sizeof(double), cudaMemcpyDeviceToHost,
                                    ctx->stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync");
    e = cudaEventRecord(ctx->done, ctx->stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
    return ADPSGD_OK;
}

int check_schedule(const adpsgd_schedule* s)
{
    if (s == nullptr) return ADPSGD_E_INVAL;
    if (s->kind != ADPSGD_CPSGD && s->kind != ADPSGD_ADPSGD && s->kind != ADPSGD_PIECEWISE) return ADPSGD_E_INVAL;
    if (s->kind == ADPSGD_PIECEWISE) {
        if (s->n_period_changes < 0 || s->literal_phase) return ADPSGD_E_INVAL;
        if (s->n_period_changes > 0 && (s->period_change_k == nullptr || s->period_values == nullptr))
            return ADPSGD_E_INVAL;
        for (int32_t t = 0; t < s->n_period_changes; ++t) {
            if (s->period_values[t] < 1) return ADPSGD_E_INVAL;
            if (t > 0 && s->period_change_k[t] <= s->period_change_k[t - 1]) return ADPSGD_E_INVAL;
        }
    }
    if (s->p_init < 1 || s->K < 0 || s->K > kMaxK || s->K_w < 0 || s->K_s < 0) return ADPSGD_E_INVAL;
    if (s->p_min < 1 || s->p_max < 0 || (s->p_max > 0 && s->p_max < s->p_min)) return ADPSGD_E_INVAL;
    if (s->n_milestones < 0 || (s->n_milestones > 0 && s->milestones == nullptr)) return ADPSGD_E_INVAL;
    if (!(s->lr0 > 0.0) || !(s->lr_factor > 0.0)) return ADPSGD_E_INVAL;
    if (s->lr_warmup_steps < 0 || (s->lr_warmup_steps > 0 && s->lr_warmup_len < 1)) return ADPSGD_E_INVAL;
    if (s->kind == ADPSGD_ADPSGD) {
        if (s->literal_phase) return ADPSGD_E_INVAL;
        if (!(s->lo > 0.0) || !(s->hi >= s->lo)) return ADPSGD_E_INVAL;
        // C_2 must receive at least one sample before the rule first compares against it.
        if (s->K_s < s->K_w + s->p_init) return ADPSGD_E_INVAL;
    }
    return ADPSGD_OK;
}

float gamma_of(const adpsgd_schedule* s, int64_t k)
{
    double g = s->lr0;
    if (s->lr_warmup_steps > 0) {
        const int64_t stair = std::min<int64_t>(k / s->lr_warmup_len, s->lr_warmup_steps - 1);
        g = g * (double)(stair + 1);
    }
    for (int32_t t = 0; t < s->n_milestones; ++t)
        if (k >= s->milestones[t]) g = g * s->lr_factor;
    return (float)g;
}

// Period of a piecewise-constant schedule at iteration k.
int32_t period_at(const adpsgd_schedule* s, int64_t k)
{
    int32_t p = s->p_init;
    for (int32_t t = 0; t < s->n_period_changes; ++t)
        if (k >= s->period_change_k[t]) p = s->period_values[t];
    return p;
}

// Does iteration k end with a sync?  Advances cnt like Algorithm 2.
bool sync_after(const adpsgd_schedule* s, adpsgd_state* st, int64_t k)
{
    if (k < s->K_w) {
        st->cnt = 0;
        return true;
    }
    if (s->kind == ADPSGD_PIECEWISE) st->p = period_at(s, k);
    if (s->kind == ADPSGD_CPSGD && s->literal_phase) return (k % st->p) == 0;
    st->cnt += 1;
    if (st->cnt >= st->p) {
        st->cnt = 0;
        return true;
    }
    return false;
}

int32_t rule(const adpsgd_schedule* s, adpsgd_state* st, int64_t k, double S, double gamma)
{
    if (k < s->K_w) return 1;                 // warm-up
    if (s->kind == ADPSGD_CPSGD || s->kind == ADPSGD_PIECEWISE) return 0;    // set by the schedule
    if (k < s->K_s) {                         // sampling C_2 (cumulative mean)
        st->m += 1;
        st->C2 += (S / gamma - st->C2) / (double)st->m;
        return 2;
    }
    const double target = gamma * st->C2;
    if (S < s->lo * target) st->p += 1;
    else if (S > s->hi * target) st->p -= 1;
    if (st->p < s->p_min) st->p = s->p_min;
    if (s->p_max > 0 && st->p > s->p_max) st->p = s->p_max;
    return 3;
}

void wire(int32_t n, int64_t P, int64_t rounds, bool with_scalar, double* per_node, double* total)
{
    const double ring = 2.0 * (double)(n - 1) / (double)n;
    double per_round = ring * 4.0 * (double)P;
    if (with_scalar) per_round += ring * 4.0;
    *per_node = per_round * (double)rounds;
    *total = *per_node * (double)n;
}

}  // namespace

extern "C" {

const char* adpsgd_strerror(int status)
{
    switch (status) {
    case ADPSGD_OK: return "ok";
    case ADPSGD_E_INVAL: return "invalid argument";
    case ADPSGD_E_ALIGN: return "device pointer not 16-byte aligned";
    case ADPSGD_E_CUDA: return "CUDA error";
    case ADPSGD_E_TIMEOUT: return "bounded wait timed out";
    case ADPSGD_E_NOMEM: return "out of memory";
    case ADPSGD_E_STATE: return "invalid state for this call";
    case ADPSGD_E_PEER: return "the shard exchange failed";
    default: return "unknown status";
    }
}

const char* adpsgd_last_error(void) { return g_last_error.c_str(); }

int adpsgd_init(const adpsgd_config* cfg, float* x, float* v, const float* h, const float* c,
                const uint16_t* noise_bf16, void* stream, adpsgd_ctx** out)
{
    if (out == nullptr) return ADPSGD_E_INVAL;
    *out = nullptr;
    if (cfg == nullptr || x == nullptr || v == nullptr || h == nullptr || c == nullptr) return ADPSGD_E_INVAL;
    if (cfg->n < 1 || cfg->P < 1) return ADPSGD_E_INVAL;
    if (cfg->P > (int64_t(1) << 34) || (int64_t)cfg->n * cfg->P > (int64_t(1) << 40)) return ADPSGD_E_INVAL;
    if (cfg->noise_mode != ADPSGD_NOISE_PHILOX && cfg->noise_mode != ADPSGD_NOISE_BF16) return ADPSGD_E_INVAL;
    if (cfg->noise_mode == ADPSGD_NOISE_BF16 && noise_bf16 == nullptr) return ADPSGD_E_INVAL;
    if (!aligned16(x) || !aligned16(v) || !aligned16(h) || !aligned16(c)) return ADPSGD_E_ALIGN;
    if (noise_bf16 != nullptr && !aligned16(noise_bf16)) return ADPSGD_E_ALIGN;
    if (cfg->fuse_intervals && cfg->n > adpsgd::interval_max_replicas()) return ADPSGD_E_INVAL;

    adpsgd_ctx* ctx = new (std::nothrow) adpsgd_ctx();
    if (ctx == nullptr) return ADPSGD_E_NOMEM;
    ctx->cfg = *cfg;
    ctx->x = x;
    ctx->v = v;
    ctx->h = h;
    ctx->c = c;
    ctx->noise = cfg->noise_mode == ADPSGD_NOISE_BF16 ? noise_bf16 : nullptr;
    ctx->stream = static_cast<cudaStream_t>(stream);
    ctx->n_total = cfg->n;
    adpsgd::make_philox_keys(cfg->seed, &ctx->keys);

    cudaError_t e = cudaGetDevice(&ctx->device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&ctx->sms, cudaDevAttrMultiProcessorCount, ctx->device);
    if (e != cudaSuccess) {
        delete ctx;
        return cuda_fail(e, "device query");
    }
    ctx->grid_avg = adpsgd::average_grid(cfg->n, cfg->P, false, true, ctx->sms);
    ctx->grid_avg_loss = adpsgd::average_grid(cfg->n, cfg->P, true, true, ctx->sms);
    ctx->grid_var = adpsgd::average_grid(cfg->n, cfg->P, false, false, ctx->sms);
    if (cfg->fuse_intervals) ctx->grid_interval = adpsgd::interval_grid(cfg->n, cfg->P, ctx->sms);
    if (cfg->fuse_sync_step && adpsgd::sync_step_supported(cfg->n, cfg->P, x, v, h, c, ctx->noise))
        ctx->grid_sync = adpsgd::sync_step_grid(cfg->n, cfg->P, ctx->noise != nullptr, cfg->want_loss != 0, ctx->sms);
    const int max_grid = std::max(adpsgd::average_grid_max(ctx->sms), adpsgd::interval_grid_max(ctx->sms));
    const size_t partial_bytes = 2 * sizeof(double) * (size_t)max_grid;
    e = cudaMalloc(reinterpret_cast<void**>(&ctx->d_partials), partial_bytes);
    if (e == cudaSuccess) e = cudaMalloc(reinterpret_cast<void**>(&ctx->d_out), 4 * sizeof(double));
    if (e == cudaSuccess) e = cudaMemset(ctx->d_out, 0, 4 * sizeof(double));
    if (e == cudaSuccess) e = cudaMallocHost(reinterpret_cast<void**>(&ctx->h_out), 2 * sizeof(double));
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ctx->done, cudaEventDisableTiming);
    if (e != cudaSuccess) {
        adpsgd_destroy(ctx);
        cudaGetLastError();
        g_last_error = std::string("context allocation: ") + cudaGetErrorString(e);
        return e == cudaErrorMemoryAllocation ? ADPSGD_E_NOMEM : ADPSGD_E_CUDA;
    }
    *out = ctx;
    return ADPSGD_OK;
}

void adpsgd_destroy(adpsgd_ctx* ctx)
{
    if (ctx == nullptr) return;
    if (ctx->done != nullptr && cudaEventRecord(ctx->done, ctx->stream) == cudaSuccess) {
        bool forced = ctx->force_incomplete;
        ctx->force_incomplete = false;
        wait_event(ctx, ctx->done);
        ctx->force_incomplete = forced;
    }
    for (const TimedLaunch& t : ctx->pending) {
        cudaEventDestroy(t.start);
        cudaEventDestroy(t.stop);
    }
    for (cudaEvent_t ev : ctx->free_events) cudaEventDestroy(ev);
    if (ctx->done != nullptr) cudaEventDestroy(ctx->done);
    if (ctx->d_partials != nullptr) cudaFree(ctx->d_partials);
    if (ctx->d_out != nullptr) cudaFree(ctx->d_out);
    if (ctx->d_var != nullptr) cudaFree(ctx->d_var);
    if (ctx->h_out != nullptr) cudaFreeHost(ctx->h_out);
    delete ctx;
}

int adpsgd_local_steps(adpsgd_ctx* ctx, int64_t k0, int32_t m, const float* lr)
{
    if (ctx == nullptr || m < 0 || k0 < 0 || k0 + m > kMaxK || (m > 0 && lr == nullptr)) return ADPSGD_E_INVAL;
    NvtxRange range("adpsgd_local_steps");
    if (ctx->cfg.fuse_intervals) {
        for (int32_t t = 0; t < m; t += adpsgd::kMaxFusedSteps) {
            const int32_t chunk = std::min<int32_t>(adpsgd::kMaxFusedSteps, m - t);
            int st = interval(ctx, k0 + t, chunk, lr + t, false, false);
            if (st != ADPSGD_OK) return st;
        }
        return ADPSGD_OK;
    }
    for (int32_t t = 0; t < m; ++t) {
        int st = local_step(ctx, k0 + t, lr[t]);
        if (st != ADPSGD_OK) return st;
    }
    return ADPSGD_OK;
}

int adpsgd_average_and_variance(adpsgd_ctx* ctx, double* D_out, double* loss_out)
{
    if (ctx == nullptr || D_out == nullptr) return ADPSGD_E_INVAL;
    NvtxRange range("adpsgd_average_and_variance");
    if (loss_out != nullptr && !ctx->cfg.want_loss) return ADPSGD_E_STATE;
    int st = average(ctx, true, loss_out != nullptr);
    if (st != ADPSGD_OK) return st;
    double D = 0.0, loss = 0.0;
    st = sync_sums(ctx, &D, &loss);
    if (st != ADPSGD_OK) return st;
    *D_out = D;
    if (loss_out != nullptr) *loss_out = loss;
    return ADPSGD_OK;
}

int adpsgd_variance(adpsgd_ctx* ctx, double* D_out)
{
    if (ctx == nullptr || D_out == nullptr) return ADPSGD_E_INVAL;
    int st = average(ctx, false, false);
    if (st != ADPSGD_OK) return st;
    double D = 0.0, loss = 0.0;
    st = sync_sums(ctx, &D, &loss);
    if (st != ADPSGD_OK) return st;
    *D_out = D;
    return ADPSGD_OK;
}

int adpsgd_state_init(const adpsgd_schedule* sched, adpsgd_state* state)
{
    if (state == nullptr || check_schedule(sched) != ADPSGD_OK) return ADPSGD_E_INVAL;
    state->k_next = 0;
    state->cnt = 0;
    state->p = sched->p_init;
    state->C2 = 0.0;
    state->m = 0;
    state->rounds = 0;
    return ADPSGD_OK;
}

int adpsgd_sched_on_sync(const adpsgd_schedule* sched, adpsgd_state* state, int64_t k, double S,
                         double gamma, int32_t* phase)
{
    if (state == nullptr || check_schedule(sched) != ADPSGD_OK || !(gamma > 0.0)) return ADPSGD_E_INVAL;
    int32_t ph = rule(sched, state, k, S, gamma);
    if (phase != nullptr) *phase = ph;
    return ADPSGD_OK;
}

int adpsgd_gamma(const adpsgd_schedule* sched, int64_t k, float* gamma_out)
{
    if (gamma_out == nullptr || check_schedule(sched) != ADPSGD_OK || k < 0) return ADPSGD_E_INVAL;
    *gamma_out = gamma_of(sched, k);
    return ADPSGD_OK;
}

int adpsgd_wire_bytes(int32_t n, int64_t P, int64_t rounds, int32_t with_scalar, double* per_node,
                      double* total)
{
    if (n < 1 || P < 0 || rounds < 0 || per_node == nullptr || total == nullptr) return ADPSGD_E_INVAL;
    wire(n, P, rounds, with_scalar != 0, per_node, total);
    return ADPSGD_OK;
}

int adpsgd_run(adpsgd_ctx* ctx, const adpsgd_schedule* sched, adpsgd_state* state, int64_t k_end,
               adpsgd_trace* trace, adpsgd_stats* stats)
{
    if (ctx == nullptr || state == nullptr) return ADPSGD_E_INVAL;
    NvtxRange range("adpsgd_run");
    int st = check_schedule(sched);
    if (st != ADPSGD_OK) return st;
    if (state->p < 1 || state->k_next < 0 || state->cnt < 0) return ADPSGD_E_INVAL;
    if (trace != nullptr && (trace->cap < 0 || (trace->cap > 0 && (trace->k == nullptr || trace->p == nullptr ||
                                                                    trace->S == nullptr || trace->C2 == nullptr ||
                                                                    trace->loss == nullptr || trace->phase == nullptr))))
        return ADPSGD_E_INVAL;
    const bool loss = ctx->cfg.want_loss != 0;
    const int64_t stop = k_end < sched->K ? k_end : sched->K;
    const bool track = trace != nullptr && trace->var != nullptr && trace->var_cap > 0;
    if (track && (ctx->cfg.fuse_intervals || ctx->replica)) return ADPSGD_E_INVAL;
    if (track && stop > ctx->d_var_cap) {
        if (ctx->d_var != nullptr) {
            cudaError_t e = cudaStreamSynchronize(ctx->stream);
            if (e == cudaSuccess) e = cudaFree(ctx->d_var);
            if (e != cudaSuccess) return cuda_fail(e, "cudaFree");
            ctx->d_var = nullptr;
        }
        cudaError_t e = cudaMalloc(reinterpret_cast<void**>(&ctx->d_var), 2 * sizeof(double) * (size_t)stop);
        if (e != cudaSuccess) {
            ctx->d_var_cap = 0;
            return e == cudaErrorMemoryAllocation ? ADPSGD_E_NOMEM : cuda_fail(e, "cudaMalloc");
        }
        ctx->d_var_cap = stop;
    }
    const int64_t k_first = state->k_next;
    // The local step of iteration k, preceded (when recording) by the variance of W_k.
    auto step = [&](int64_t k) -> int {
        if (track && k < trace->var_cap) {
            int rs = variance_into_slot(ctx, k);
            if (rs != ADPSGD_OK) return rs;
        }
        return local_step(ctx, k, gamma_of(sched, k));
    };
    const int64_t launches0[4] = {ctx->launches[0], ctx->launches[1], ctx->launches[2], ctx->launches[3]};
    bool launched_ahead = false;  // the local step of iteration k is already enqueued
    if (ctx->cfg.fuse_intervals) {
        // One kernel per stretch of iterations up to and including the next sync (at most
        // kMaxFusedSteps); sync_after advances cnt exactly as in the unfused loop below.
        float gam[adpsgd::kMaxFusedSteps];
        int64_t k = state->k_next;
        while (k < stop) {
            int32_t m = 0;
            bool sync = false;
            while (k + m < stop && m < adpsgd::kMaxFusedSteps) {
                gam[m] = gamma_of(sched, k + m);
                const bool s_now = sync_after(sched, state, k + m);
                ++m;
                if (s_now) {
                    sync = true;
                    break;
                }
            }
            st = interval(ctx, k, m, gam, sync, loss);
            if (st != ADPSGD_OK) return st;
            state->k_next = k + m;
            if (sync) {
                {
                    NvtxRange wait_range("adpsgd_sync_wait");
                    st = wait_event(ctx, ctx->done);
                }
                if (st != ADPSGD_OK) return st;
                double D = 0.0, L = 0.0;
                st = sync_sums(ctx, &D, &L);
                if (st != ADPSGD_OK) return st;
                const int64_t ks = k + m - 1;
                const double S = D / (double)ctx->n_total;
                const int32_t phase = rule(sched, state, ks, S, (double)gam[m - 1]);
                if (trace != nullptr && trace->len < trace->cap) {
                    const int64_t t = trace->len;
                    trace->k[t] = ks;
                    trace->p[t] = state->p;
                    trace->S[t] = S;
                    trace->C2[t] = state->C2;
                    trace->loss[t] = loss ? L : 0.0;
                    trace->phase[t] = phase;
                    trace->len = t + 1;
                }
                state->rounds += 1;
            }
            k += m;
        }
    }
    for (int64_t k = state->k_next; k < stop; ++k) {
        // Whether iteration k ends with a sync depends only on the schedule state, not on the
        // step, so it is known before the step is enqueued.
        // If enqueuing fails, the state goes back to the start of iteration k.
        const adpsgd_state before = *state;
        const bool sync = sync_after(sched, state, k);
        if (sync && !launched_ahead && ctx->grid_sync > 0) {
            // the step and the averaging as one kernel
            if (track && k < trace->var_cap) st = variance_into_slot(ctx, k);
            if (st == ADPSGD_OK) st = sync_step_enqueue(ctx, k, gamma_of(sched, k), loss);
        } else {
            if (!launched_ahead) st = step(k);
            if (st == ADPSGD_OK && sync) st = average_enqueue(ctx, true, loss);
        }
        if (st != ADPSGD_OK) {
            *state = before;
            return st;
        }
        launched_ahead = false;
        state->k_next = k + 1;
        if (!sync) continue;
        // Whatever the rule decides, iteration k + 1 starts with a local step (p >= 1), so it is
        // enqueued behind the averaging before the host waits for S: the GPU stays busy while
        // the scalars travel to the host and the rule runs.
        if (k + 1 < stop) {
            st = step(k + 1);
            if (st != ADPSGD_OK) return st;
            launched_ahead = true;
        }
        {
            NvtxRange wait_range("adpsgd_sync_wait");
            st = wait_event(ctx, ctx->done);
        }
        if (st != ADPSGD_OK) return st;
        double D = 0.0, L = 0.0;
        st = sync_sums(ctx, &D, &L);
        if (st != ADPSGD_OK) return st;
        const double S = D / (double)ctx->n_total;
        const int32_t phase = rule(sched, state, k, S, (double)gamma_of(sched, k));
        if (trace != nullptr) {
            if (trace->len < trace->cap) {
                const int64_t t = trace->len;
                trace->k[t] = k;
                trace->p[t] = state->p;
                trace->S[t] = S;
                trace->C2[t] = state->C2;
                trace->loss[t] = loss ? L : 0.0;
                trace->phase[t] = phase;
                trace->len = t + 1;
            }
        }
        state->rounds += 1;
    }
    if (track) {
        const int64_t last = std::min(stop, trace->var_cap);
        if (last > k_first) {
            std::vector<double> slots(2 * (size_t)(last - k_first));
            cudaError_t e = cudaMemcpyAsync(slots.data(), ctx->d_var + 2 * k_first, slots.size() * sizeof(double),
                                            cudaMemcpyDeviceToHost, ctx->stream);
            if (e == cudaSuccess) e = cudaEventRecord(ctx->done, ctx->stream);
            if (e != cudaSuccess) return cuda_fail(e, "variance copy");
            st = wait_event(ctx, ctx->done);
            if (st != ADPSGD_OK) return st;
            std::vector<double> D((size_t)(last - k_first));
            for (int64_t k = k_first; k < last; ++k) D[(size_t)(k - k_first)] = slots[2 * (size_t)(k - k_first)];
            if (ctx->sharded) {
                std::vector<double> local = D;
                st = shard_combine(&ctx->shard, local.data(), (int64_t)local.size(), D.data());
                if (st != ADPSGD_OK) return st;
            }
            for (int64_t k = k_first; k < last; ++k) trace->var[k] = D[(size_t)(k - k_first)] / (double)ctx->n_total;
        }
    }
    if (stats != nullptr) {
        stats->rounds = state->rounds;
        stats->equiv_period = state->rounds > 0 ? (double)state->k_next / (double)state->rounds : 0.0;
        double total = 0.0;
        const int64_t P_all = ctx->sharded ? ctx->shard.P_total : ctx->cfg.P;
        wire(ctx->n_total, P_all, state->rounds, true, &stats->wire_bytes_per_node, &stats->wire_bytes_total);
        wire(ctx->n_total, P_all, state->k_next, false, &stats->fullsgd_wire_bytes_per_node, &total);
        stats->local_step_launches = ctx->launches[0] - launches0[0];
        stats->average_launches = ctx->launches[1] - launches0[1];
        stats->interval_launches = ctx->launches[2] - launches0[2];
        stats->sync_step_launches = ctx->launches[3] - launches0[3];
    }
    return ADPSGD_OK;
}

int adpsgd_average_and_variance_static(float* x, const float* h, const float* c, int32_t n, int64_t P,
                                       double* D_out, double* loss_out, int64_t wait_timeout_ms, void* stream)
{
    if (x == nullptr || D_out == nullptr || n < 1 || P < 1) return ADPSGD_E_INVAL;
    if (P > (int64_t(1) << 34) || (int64_t)n * P > (int64_t(1) << 40)) return ADPSGD_E_INVAL;
    const bool loss = loss_out != nullptr;
    if (loss && (h == nullptr || c == nullptr)) return ADPSGD_E_INVAL;
    if (!aligned16(x) || (loss && (!aligned16(h) || !aligned16(c)))) return ADPSGD_E_ALIGN;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int device = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
    if (e != cudaSuccess) return cuda_fail(e, "device query");
    const int grid = adpsgd::average_grid(n, P, loss, true, sms);
    if (grid > adpsgd::static_scratch_max_blocks()) {
        g_last_error = "the averaging grid needs " + std::to_string(grid) + " partial-sum slots; the fixed scratch holds " +
                       std::to_string(adpsgd::static_scratch_max_blocks());
        return ADPSGD_E_INVAL;
    }
    adpsgd::AverageArgs a;
    a.x = x;
    a.h = loss ? h : nullptr;
    a.c = loss ? c : nullptr;
    a.n = n;
    a.P = P;
    a.write_back = true;
    a.grid = grid;
    e = adpsgd::static_scratch_address(&a.partials, &a.out, &a.counter);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress");
    // The array keeps the previous call's contents; the completion counter must start at zero.
    e = cudaMemsetAsync(a.counter, 0, sizeof(unsigned int), s);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync");
    e = adpsgd::launch_average(a, s);
    if (e != cudaSuccess) return cuda_fail(e, "average");
    // Bounded wait for the stream, then a 16-byte copy from an idle stream.
    const auto t0 = std::chrono::steady_clock::now();
    const auto limit = std::chrono::milliseconds(wait_timeout_ms > 0 ? wait_timeout_ms : 60000);
    int spins = 0;
    for (;;) {
        e = cudaStreamQuery(s);
        if (e == cudaSuccess) break;
        if (e != cudaErrorNotReady) return cuda_fail(e, "cudaStreamQuery");
        if (std::chrono::steady_clock::now() - t0 > limit) {
            g_last_error = "bounded wait ran out";
            return ADPSGD_E_TIMEOUT;
        }
        if (++spins > 2000) std::this_thread::sleep_for(std::chrono::microseconds(20));
    }
    double result[2] = {0.0, 0.0};
    e = cudaMemcpyAsync(result, a.out, sizeof(result), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync");
    *D_out = result[0];
    if (loss) *loss_out = result[1];
    return ADPSGD_OK;
}

int adpsgd_philox_fill(uint64_t seed, uint32_t tag, int32_t n, int64_t nq, int64_t k, uint32_t* out, void* stream)
{
    if (out == nullptr || n < 0 || nq < 0 || nq > kMaxK || k < 0 || k >= kMaxK) return ADPSGD_E_INVAL;
    if ((int64_t)n * nq > (int64_t(1) << 38)) return ADPSGD_E_INVAL;  // keeps the grid below 2^31 blocks
    if (!aligned16(out)) return ADPSGD_E_ALIGN;
    cudaError_t e = adpsgd::launch_philox_fill(seed, tag, n, nq, (uint32_t)k, out, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ADPSGD_OK : cuda_fail(e, "philox fill");
}

int adpsgd_noise_fill_f32(uint64_t seed, uint32_t tag, int32_t n, int64_t P, int64_t k, float* out, void* stream)
{
    if (out == nullptr || n < 0 || P < 0 || P > (int64_t(1) << 34) || k < 0 || k >= kMaxK) return ADPSGD_E_INVAL;
    if ((int64_t)n * P > (int64_t(1) << 40)) return ADPSGD_E_INVAL;
    if (!aligned16(out)) return ADPSGD_E_ALIGN;
    cudaError_t e = adpsgd::launch_noise_f32(seed, tag, n, P, (uint32_t)k, out, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ADPSGD_OK : cuda_fail(e, "noise fill");
}

int adpsgd_noise_fill_bf16(uint64_t seed, int32_t n, int64_t P, uint16_t* out, void* stream)
{
    if (out == nullptr || n < 0 || P < 0 || P > (int64_t(1) << 34)) return ADPSGD_E_INVAL;
    if ((int64_t)n * P > (int64_t(1) << 40)) return ADPSGD_E_INVAL;
    if (!aligned16(out)) return ADPSGD_E_ALIGN;
    cudaError_t e = adpsgd::launch_noise_bf16(seed, n, P, 0u, 0u, out, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ADPSGD_OK : cuda_fail(e, "bf16 noise fill");
}

int adpsgd_noise_fill_bf16_part(uint64_t seed, int32_t n, int64_t P, int32_t replica0, int64_t col0, uint16_t* out,
                                void* stream)
{
    if (out == nullptr || n < 0 || P < 0 || P > (int64_t(1) << 34) || replica0 < 0) return ADPSGD_E_INVAL;
    if (col0 < 0 || col0 % 4 != 0 || (col0 + P + 3) / 4 > kMaxK) return ADPSGD_E_INVAL;
    if ((int64_t)n * P > (int64_t(1) << 40)) return ADPSGD_E_INVAL;
    if (!aligned16(out)) return ADPSGD_E_ALIGN;
    cudaError_t e = adpsgd::launch_noise_bf16(seed, n, P, (uint32_t)replica0, (uint32_t)(col0 / 4), out,
                                              static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ADPSGD_OK : cuda_fail(e, "bf16 noise fill");
}

int adpsgd_set_shard(adpsgd_ctx* ctx, const adpsgd_shard* shard)
{
    if (ctx == nullptr || ctx->replica || check_shard(shard) != ADPSGD_OK) return ADPSGD_E_INVAL;
    if (shard->P_total < shard->col0 + ctx->cfg.P) return ADPSGD_E_INVAL;
    if ((shard->col0 + ctx->cfg.P + 3) / 4 > kMaxK) return ADPSGD_E_INVAL;  // Philox blocks are 32-bit words
    ctx->shard = *shard;
    ctx->sharded = true;
    ctx->q0 = (uint32_t)(shard->col0 / 4);
    return ADPSGD_OK;
}

int adpsgd_set_replica_split(adpsgd_ctx* ctx, const adpsgd_replica_split* rs)
{
    if (ctx == nullptr || rs == nullptr || ctx->sharded) return ADPSGD_E_INVAL;
    if (rs->processes < 1 || rs->rank < 0 || rs->rank >= rs->processes || rs->collective == nullptr) return ADPSGD_E_INVAL;
    if (rs->processes > 1 && rs->gather == nullptr) return ADPSGD_E_INVAL;
    if (rs->replica0 < 0 || rs->n_total < 1 || (int64_t)rs->replica0 + ctx->cfg.n > rs->n_total) return ADPSGD_E_INVAL;
    if (rs->col0 < 0 || rs->col0 % 4 != 0 || rs->P_chunk < 0 || rs->col0 + rs->P_chunk > ctx->cfg.P) return ADPSGD_E_INVAL;
    if ((int64_t)rs->n_total * rs->P_chunk > (int64_t(1) << 40)) return ADPSGD_E_INVAL;
    if (rs->chunk_x == nullptr || ctx->cfg.fuse_intervals || ctx->cfg.fuse_sync_step) return ADPSGD_E_INVAL;
    if (!aligned16(rs->chunk_x) || !aligned16(ctx->h + rs->col0) || !aligned16(ctx->c + rs->col0)) return ADPSGD_E_ALIGN;
    ctx->split = *rs;
    ctx->replica = true;
    ctx->r0 = (uint32_t)rs->replica0;
    ctx->n_total = rs->n_total;
    ctx->grid_chunk = adpsgd::average_grid(rs->n_total, rs->P_chunk, false, true, ctx->sms);
    ctx->grid_chunk_loss = adpsgd::average_grid(rs->n_total, rs->P_chunk, true, true, ctx->sms);
    ctx->grid_chunk_var = adpsgd::average_grid(rs->n_total, rs->P_chunk, false, false, ctx->sms);
    // the chunk sums are exchanged like a column shard's (process order); x keeps every column
    ctx->shard = adpsgd_shard{rs->processes, rs->rank, 0, ctx->cfg.P, rs->gather, rs->user};
    ctx->sharded = true;
    return ADPSGD_OK;
}

int adpsgd_shard_combine(const adpsgd_shard* shard, const double* local, int64_t count, double* out)
{
    if (check_shard(shard) != ADPSGD_OK || count < 0 || (count > 0 && (local == nullptr || out == nullptr)))
        return ADPSGD_E_INVAL;
    return shard_combine(shard, local, count, out);
}

namespace {

// The kind of memory p points into (cudaMemoryTypeUnregistered for plain host memory) and,
// for device memory, the device it lives on.
cudaError_t memory_type(const void* p, cudaMemoryType* type, int* device)
{
    cudaPointerAttributes attr;
    const cudaError_t e = cudaPointerGetAttributes(&attr, p);
    if (e != cudaSuccess) return e;
    *type = attr.type;
    *device = attr.device;
    return cudaSuccess;
}

// One host <-> device copy: `host` is the host side, `device` the device side; to_device
// gives the direction.
int transfer(void* dst, const void* src, int64_t bytes, void* stream, bool to_device)
{
    if (bytes < 0 || (bytes > 0 && (dst == nullptr || src == nullptr))) return ADPSGD_E_INVAL;
    if (bytes == 0) return ADPSGD_OK;
    if (!aligned16(dst) || !aligned16(src)) return ADPSGD_E_ALIGN;
    const void* host = to_device ? src : dst;
    const void* device = to_device ? dst : src;
    cudaMemoryType host_type, device_type;
    int host_dev = -1, device_dev = -1, current = 0;
    cudaError_t e = memory_type(device, &device_type, &device_dev);
    if (e == cudaSuccess) e = memory_type(host, &host_type, &host_dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaPointerGetAttributes");
    if (device_type != cudaMemoryTypeDevice && device_type != cudaMemoryTypeManaged) {
        g_last_error = "the device side of the copy is not device memory";
        return ADPSGD_E_INVAL;
    }
    if (host_type == cudaMemoryTypeDevice) {
        g_last_error = "the host side of the copy is device memory";
        return ADPSGD_E_INVAL;
    }
    e = cudaGetDevice(&current);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    void* mapped = nullptr;
    // The copy kernel runs on the current device, so it takes only device memory of that device;
    // managed memory and another device's memory go through cudaMemcpyAsync, which needs no peer
    // mapping and migrates managed pages itself.
    const bool kernel_route = device_type == cudaMemoryTypeDevice && device_dev == current &&
                              host_type == cudaMemoryTypeHost &&
                              cudaHostGetDevicePointer(&mapped, const_cast<void*>(host), 0) == cudaSuccess &&
                              aligned16(mapped);
    if (kernel_route) {
        int sms = 0;
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, current);
        if (e != cudaSuccess) return cuda_fail(e, "device query");
        e = to_device ? adpsgd::launch_copy(dst, mapped, bytes, sms, s) : adpsgd::launch_copy(mapped, src, bytes, sms, s);
        return e == cudaSuccess ? ADPSGD_OK : cuda_fail(e, "copy kernel");
    }
    cudaGetLastError();  // a failed cudaHostGetDevicePointer leaves no sticky error; clear the last one
    e = cudaMemcpyAsync(dst, src, (size_t)bytes, to_device ? cudaMemcpyHostToDevice : cudaMemcpyDeviceToHost, s);
    return e == cudaSuccess ? ADPSGD_OK : cuda_fail(e, "cudaMemcpyAsync");
}

}  // namespace

int adpsgd_init_replicas(adpsgd_ctx* ctx, const float* w0)
{
    if (ctx == nullptr || w0 == nullptr) return ADPSGD_E_INVAL;
    NvtxRange range("adpsgd_init_replicas");
    const int32_t n = ctx->cfg.n;
    const int64_t P = ctx->cfg.P;
    const size_t row_bytes = (size_t)P * sizeof(float);
    cudaMemoryType type;
    int dev = -1;
    cudaError_t e = memory_type(w0, &type, &dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaPointerGetAttributes");
    // The kernel reads w0 where it is device memory of this device or page-locked host memory
    // (through its mapped address); anything else is first copied into row 0 of x.
    const float* src = nullptr;
    int32_t first = 0;
    void* mapped = nullptr;
    if (type == cudaMemoryTypeDevice && dev == ctx->device) {
        src = w0;
    } else if (type == cudaMemoryTypeHost &&
               cudaHostGetDevicePointer(&mapped, const_cast<float*>(w0), 0) == cudaSuccess) {
        src = static_cast<const float*>(mapped);
    } else {
        cudaGetLastError();  // a failed cudaHostGetDevicePointer leaves no sticky error
        e = cudaMemcpyAsync(ctx->x, w0, row_bytes, cudaMemcpyDefault, ctx->stream);
        if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync");
        src = ctx->x;
        first = 1;
    }
    e = adpsgd::launch_broadcast_rows(ctx->x + (int64_t)first * P, src, n - first, P, ctx->sms, ctx->stream);
    if (e != cudaSuccess) return cuda_fail(e, "broadcast kernel");
    e = cudaMemsetAsync(ctx->v, 0, (size_t)n * row_bytes, ctx->stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync");
    return ADPSGD_OK;
}

int adpsgd_copy_h2d(void* dst, const void* src, int64_t bytes, void* stream)
{
    return transfer(dst, src, bytes, stream, true);
}

int adpsgd_copy_d2h(void* dst, const void* src, int64_t bytes, void* stream)
{
    return transfer(dst, src, bytes, stream, false);
}

int adpsgd_kernel_times(adpsgd_ctx* ctx, adpsgd_kernel_timing* out)
{
    if (ctx == nullptr || out == nullptr) return ADPSGD_E_INVAL;
    if (!ctx->cfg.time_kernels) return ADPSGD_E_STATE;
    int st = harvest_times(ctx);
    if (st != ADPSGD_OK) return st;
    out->local_step_ms = ctx->ms[0];
    out->local_step_launches = ctx->timed_launches[0];
    out->average_ms = ctx->ms[1];
    out->average_launches = ctx->timed_launches[1];
    out->interval_ms = ctx->ms[2];
    out->interval_launches = ctx->timed_launches[2];
    out->sync_step_ms = ctx->ms[3];
    out->sync_step_launches = ctx->timed_launches[3];
    return ADPSGD_OK;
}

int adpsgd_reset_kernel_times(adpsgd_ctx* ctx)
{
    if (ctx == nullptr) return ADPSGD_E_INVAL;
    if (ctx->cfg.time_kernels) {
        int st = harvest_times(ctx);
        if (st != ADPSGD_OK) return st;
    }
    ctx->ms[0] = ctx->ms[1] = ctx->ms[2] = ctx->ms[3] = 0.0;
    ctx->timed_launches[0] = ctx->timed_launches[1] = ctx->timed_launches[2] = ctx->timed_launches[3] = 0;
    return ADPSGD_OK;
}

int adpsgd_test_force_incomplete(adpsgd_ctx* ctx, int32_t force_incomplete)
{
    if (ctx == nullptr) return ADPSGD_E_INVAL;
    ctx->force_incomplete = force_incomplete != 0;
    return ADPSGD_OK;
}

}  // extern "C"
