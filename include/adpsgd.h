/*
 * adpsgd.h -- C ABI of the GB300 (sm_103a) data-parallel hot path of ADPSGD,
 * adaptive periodic parameter averaging SGD (Jiang & Agrawal, "Adaptive
 * Periodic Averaging: A Practical Approach to Reducing Communication in
 * Distributed Learning", arXiv 2007.06134).
 *
 * n worker replicas ("nodes" in the paper) live on one GPU as an [n, P] fp32
 * row-major tensor x (replica i at x + i*P) with momentum buffers v of the
 * same shape.  The objective is the separable quadratic
 *     f(x) = 1/2 sum_j h_j (x_j - c_j)^2
 * standing in for the paper's CNN losses (Sec. II-A, Eq. obj1), with additive
 * Gaussian gradient noise standing in for mini-batch sampling (Eq. eg).
 *
 * Conventions for every entry point:
 *   - Pointers named x, v, h, c, noise, out are DEVICE pointers the caller owns
 *     (allocated by the caller, e.g. through PyTorch); the library never frees
 *     them and keeps only borrowed references inside a context.
 *   - Pointers to structs and scalars (cfg, schedule, state, trace, stats,
 *     D_out, lr, ...) are HOST pointers.
 *   - `stream` is a cudaStream_t passed as void* (NULL = the legacy default
 *     stream).  All device work is enqueued on it in order.
 *   - Every call returns an adpsgd_status; no C++ exception crosses the ABI.
 *     On ADPSGD_E_CUDA, adpsgd_last_error() gives the CUDA error text of the
 *     calling thread.  Calls that return scalars to the host wait for them
 *     with a bounded poll (cfg.wait_timeout_ms) and return ADPSGD_E_TIMEOUT
 *     instead of blocking forever.
 *   - Device pointers must be 16-byte aligned (ADPSGD_E_ALIGN otherwise);
 *     P need not be a multiple of 4 (a scalar kernel variant handles that).
 *   - A context is not thread-safe: use each one from one host thread at a time.  Separate
 *     contexts on separate streams are independent.
 */
#ifndef ADPSGD_H
#define ADPSGD_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    ADPSGD_OK = 0,
    ADPSGD_E_INVAL = -1,   /* an argument is out of range or NULL where it may not be */
    ADPSGD_E_ALIGN = -2,   /* a device pointer is not 16-byte aligned */
    ADPSGD_E_CUDA = -3,    /* a CUDA runtime call failed (see adpsgd_last_error) */
    ADPSGD_E_TIMEOUT = -4, /* a bounded host wait ran out; the work may still be in flight */
    ADPSGD_E_NOMEM = -5,   /* the context's own scratch could not be allocated */
    ADPSGD_E_STATE = -6,   /* call not valid in the current state (e.g. no noise tensor) */
    ADPSGD_E_PEER = -7     /* the shard exchange (adpsgd_shard.gather) reported a failure */
} adpsgd_status;

/* Opaque context: borrowed pointers to x, v, h, c (and the noise tensor),
 * the stream, and the only memory the library allocates itself: per-block
 * fp64 partial sums on the device, two pinned host doubles, CUDA events. */
typedef struct adpsgd_ctx adpsgd_ctx;

enum { ADPSGD_NOISE_PHILOX = 0, ADPSGD_NOISE_BF16 = 1 };

typedef struct {
    int32_t n;               /* replicas, >= 1 (the paper's n nodes) */
    int32_t noise_mode;      /* ADPSGD_NOISE_PHILOX: z drawn per step from Philox4x32-10;
                                ADPSGD_NOISE_BF16: z read from a caller tensor [n, P] bf16 */
    int64_t P;               /* parameters per replica, >= 1 */
    float momentum;          /* mu (Sec. IV-A uses 0.9) */
    float weight_decay;      /* wd, added to the gradient as wd * x (0 = off) */
    float noise_sigma;       /* sigma: g = h (x - c) + sigma z */
    int32_t want_loss;       /* nonzero: averaging also returns 1/2 sum_j h_j (xbar_j - c_j)^2 */
    uint64_t seed;           /* Philox key (low word, high word) */
    int64_t wait_timeout_ms; /* bound on every host wait; <= 0 means 60000 */
    int32_t time_kernels;    /* N > 0: bracket every N-th launch of each kernel kind with CUDA
                                events (1: every launch); 0: no timing */
    int32_t fuse_intervals;  /* nonzero (needs n <= 32): adpsgd_run and adpsgd_local_steps run each
                                stretch of local steps up to the next sync (at most 256 steps), and
                                the sync's averaging, as ONE kernel that keeps x and v in registers
                                between steps.  Results are bit-identical to the unfused path.  Valid
                                only because the surrogate objective is separable per column. */
    int32_t fuse_sync_step;  /* nonzero: in adpsgd_run's per-iteration path, the local step of each
                                iteration that ends with a sync and that averaging run as ONE
                                kernel (x is not written and read back in between: 17 instead of
                                25 bytes per replica-param).  Bit-identical results (D and the
                                loss up to the order of fp64 additions).  Valid for any objective
                                whose gradient is computed per element in the step; nothing is
                                carried across steps.  Used where it measured faster: n <= 16,
                                P % 4 == 0, every array 16-byte aligned (bf16 noise: 8-byte);
                                elsewhere ignored. */
} adpsgd_config;

/* Schedules (Algorithm 1: kind 0; Algorithm 2: kind 1; kind 2: a piecewise-constant period,
 * such as the four strategies of Sec. III-A and the decreasing period of Sec. V-B). */
enum { ADPSGD_CPSGD = 0, ADPSGD_ADPSGD = 1, ADPSGD_PIECEWISE = 2 };

typedef struct {
    int32_t kind;            /* ADPSGD_CPSGD (constant p), ADPSGD_ADPSGD or ADPSGD_PIECEWISE */
    int32_t p_init;          /* the constant period, or Algorithm 2's p_init; >= 1 */
    int64_t K;               /* total iterations of the schedule */
    int64_t K_s;             /* Algorithm 2: syncs at iterations k < K_s sample C_2;
                                must be >= p_init (+ K_w) so that C_2 gets a sample */
    int64_t K_w;             /* warm-up: iterations k < K_w sync every iteration and are
                                not sampled (Sec. IV-B warm-up epoch); 0 = none */
    double lo, hi;           /* Algorithm 2 thresholds, 0.7 and 1.3 in the paper */
    int32_t p_min, p_max;    /* clamp of p after the rule; p_max = 0: no upper bound */
    double lr0;              /* step size at k = 0 */
    double lr_factor;        /* step size multiplied by this at each milestone */
    int32_t n_milestones;    /* length of milestones[] (host array) */
    int32_t literal_phase;   /* kind 0 only: sync when k mod p == 0 (Algorithm 1 as printed)
                                instead of when cnt reaches p */
    const int64_t* milestones; /* iterations from which the step size changes */
    int32_t n_period_changes;  /* kind 2: the period is p_init, then period_values[t] from iteration */
    int32_t reserved;          /* period_change_k[t] on (increasing k, values >= 1; host arrays) */
    const int64_t* period_change_k;
    const int32_t* period_values;
    int32_t lr_warmup_steps;   /* step-size warm-up of Sec. IV-C (0 = none): on stair
                                  s = min(k div lr_warmup_len, lr_warmup_steps - 1) the step size is
                                  lr0 * (s + 1) before the milestone factors */
    int32_t reserved2;
    int64_t lr_warmup_len;     /* iterations per stair (the paper: one epoch), >= 1 */
} adpsgd_schedule;

/* Scheduler state (everything besides x and v that a checkpoint needs). */
typedef struct {
    int64_t k_next;          /* next iteration to run */
    int32_t cnt;             /* iterations since the last sync (Algorithm 2's cnt) */
    int32_t p;               /* current period */
    double C2;               /* sampled C_2 (cumulative mean of S_k / gamma_k) */
    int64_t m;               /* number of samples in C2 */
    int64_t rounds;          /* syncs so far */
} adpsgd_state;

/* Per-sync trace, caller-allocated host arrays of capacity cap. */
typedef struct {
    int64_t cap;             /* capacity of every array */
    int64_t len;             /* entries written (<= cap); syncs beyond cap are counted, not stored */
    int64_t* k;              /* iteration of the sync */
    int32_t* p;              /* period after the rule ran */
    double* S;               /* S_k = D / n */
    double* C2;              /* C_2 after the rule ran */
    double* loss;            /* 1/2 sum_j h_j (xbar_j - c_j)^2 (0 if want_loss == 0) */
    int32_t* phase;          /* 0 constant, 1 warm-up, 2 sampling, 3 adapting */
    int64_t var_cap;         /* entries of var (0: not recorded) */
    double* var;             /* var[k] = Var[W_k] = D / n at the start of iteration k, k < var_cap
                                (Sec. II-B; the series behind V_t of Eq. vt and the weighted variance
                                of Eq. metric2).  Costs one variance pass (4 B per replica-param) per
                                iteration; not available with cfg.fuse_intervals */
} adpsgd_trace;

typedef struct {
    int64_t rounds;                  /* syncs so far (state.rounds) */
    double equiv_period;             /* k_next / rounds */
    double wire_bytes_per_node;      /* ring allreduce of P fp32 + one fp32 S_k, per sync */
    double wire_bytes_total;         /* times n */
    double fullsgd_wire_bytes_per_node; /* one P-fp32 allreduce per iteration (FULLSGD) */
    int64_t local_step_launches;     /* kernel launches issued by this call: local steps, */
    int64_t average_launches;        /* averagings, */
    int64_t interval_launches;       /* fused intervals (cfg.fuse_intervals), */
    int64_t sync_step_launches;      /* and fused sync steps (cfg.fuse_sync_step) */
} adpsgd_stats;

/* Device time of the kernels launched through a context, from CUDA events on its stream. */
typedef struct {
    double local_step_ms;
    int64_t local_step_launches;
    double average_ms;
    int64_t average_launches;
    double interval_ms;
    int64_t interval_launches;
    double sync_step_ms;
    int64_t sync_step_launches;
} adpsgd_kernel_timing;

/* Create a context over caller-owned device arrays.
 * x, v: [n, P] fp32 (read/write); h, c: [P] fp32 (read only);
 * noise_bf16: [n, P] bf16 (read only) when cfg->noise_mode == ADPSGD_NOISE_BF16, else NULL.
 * The pointers must stay valid until adpsgd_destroy.  Errors: E_INVAL (bad n, P, NULL
 * pointer, P*n overflow, fuse_intervals with n > 32), E_ALIGN, E_NOMEM, E_CUDA.  On error
 * *out is NULL. */
int adpsgd_init(const adpsgd_config* cfg, float* x, float* v, const float* h, const float* c,
                const uint16_t* noise_bf16, void* stream, adpsgd_ctx** out);

/* m local steps of every replica (Algorithm 1 and 2, the local update;
 * Sec. IV-A momentum): for t in [0, m), step k = k0 + t with step size lr[t] (host array):
 *   g = h (x - c) + sigma z[i, j, k];  if wd != 0: g += wd x;  v = mu v + g;  x -= lr[t] v
 * each a separately rounded fp32 operation.  z is word (j mod 4) of Philox4x32-10 with counter
 * (j div 4, i, k, 0) and key (seed lo, seed hi), mapped through Box-Muller.  Enqueued only;
 * does not wait.  Errors: E_INVAL (m < 0, k0 < 0, k0 + m > 2^32), E_CUDA. */
int adpsgd_local_steps(adpsgd_ctx* ctx, int64_t k0, int32_t m, const float* lr);

/* Synchronisation (Algorithm 2 averaging and S_k lines; Sec. II-B definition of Var[W_k]):
 * for every column j, xbar_j = x_0j + (sum_{i>=1} (x_ij - x_0j)) / n in fp32, written back to
 * all n replicas, and *D_out = sum_j sum_i (x_ij - xbar_j)^2 over the pre-average values
 * (n * Var[W]), accumulated in fp64.  If loss_out != NULL (needs cfg.want_loss),
 * *loss_out = 1/2 sum_j h_j (xbar_j - c_j)^2.  Blocks (bounded) until the scalars arrive.
 * Accuracy (every averaging entry point, and the syncs of adpsgd_run): xbar as written above,
 * bit for bit.  D and the loss are within 1e-4 relative of the fp64 definitions, over the
 * whole fp32 range, for h_j >= 0.  Squares are taken in fp32 where their column sums lie in
 * [2^-100, 2^100].  Elsewhere the columns are redone in fp64: subnormal or huge deviations,
 * inf, NaN.  A NaN or inf in x gives a NaN or inf D, as the definition does.
 * Errors: E_INVAL (D_out NULL), E_STATE (loss requested without want_loss), E_TIMEOUT, E_CUDA. */
int adpsgd_average_and_variance(adpsgd_ctx* ctx, double* D_out, double* loss_out);

/* The same averaging as adpsgd_average_and_variance, for callers that cannot allocate device
 * memory: code running inside a host framework whose pool allocator owns the GPU's memory
 * (a cudaMalloc of its own would bypass or fragment that pool), and code on a latency-critical
 * path where cudaMalloc / cudaFree would synchronise the device.  The paper has no counterpart:
 * this is an interface variant, not part of the method.
 *
 * It needs no context and allocates nothing.  Its scratch is a fixed array inside the library,
 * 2 * 2048 + 4 doubles (32.8 KB), which every GPU that loads the library holds until the process
 * exits.  The per-block partial sums for up to 2048 blocks live there.  A shape whose averaging
 * grid would need more blocks is rejected with ADPSGD_E_INVAL; on GB300 the grid is at most
 * 1216 blocks.
 *
 * x: device fp32 [n, P], read, then xbar written to every row.  h, c: device fp32 [P], needed
 * only when loss_out != NULL.  D_out, loss_out: host doubles; loss_out may be NULL.
 * stream: cudaStream_t as void*.  wait_timeout_ms bounds the wait for the stream (<= 0: 60000).
 *
 * The first call on each device looks up the scratch array's device address
 * (cudaGetSymbolAddress) with that device current.  Make that first call before any stream
 * capture.  The address is cached with the id of the CUDA context it was looked up in; a call from
 * a different context (after cudaDeviceReset, or with another context current) looks it up again.
 * Every call uses the same array, which keeps the last call's contents.  Each call clears the
 * completion counter in it on the stream before the launch, and writes every other slot before
 * reading it.  Calls that overlap on the GPU (several host threads, or streams that run
 * concurrently) race on the array and must be serialised by the caller.
 * The call returns once the stream has passed the averaging (a bounded poll, then a 16-byte copy
 * of the two sums).  After ADPSGD_E_TIMEOUT the averaging may still be running on the shared
 * array: wait for that stream to finish before calling again, on any stream.
 * Errors: E_INVAL, E_ALIGN, E_TIMEOUT, E_CUDA. */
int adpsgd_average_and_variance_static(float* x, const float* h, const float* c, int32_t n, int64_t P,
                                       double* D_out, double* loss_out, int64_t wait_timeout_ms, void* stream);

/* D = sum_j sum_i (x_ij - xbar_j)^2 without averaging (the per-iteration Var[W_k] of
 * Sec. II-B and Eq. vt, times n).  Blocks (bounded).  Errors: as above. */
int adpsgd_variance(adpsgd_ctx* ctx, double* D_out);

/* Initial scheduler state of a schedule: k_next 0, cnt 0, p = p_init, C2 0.  Errors: E_INVAL. */
int adpsgd_state_init(const adpsgd_schedule* sched, adpsgd_state* state);

/* Run iterations [state->k_next, min(k_end, sched->K)) of a schedule (Algorithm 2, or
 * Algorithm 1 when kind == ADPSGD_CPSGD): each iteration one local step with gamma_k, then
 * cnt += 1 and, when cnt reaches p, one averaging, S = D / n, and the period rule
 * (adpsgd_sched_on_sync).  Updates *state so that a later call resumes bit-identically.
 * With cfg.fuse_intervals each stretch of steps up to a sync runs as one kernel; with
 * cfg.fuse_sync_step the step of each iteration that ends with a sync, and that averaging, run
 * as one kernel (except where that step was already enqueued ahead of the previous sync's wait,
 * which happens only when p = 1).  Both give the same x, v and schedule as the separate kernels;
 * D, and so S, may differ in the last bits of its fp64 sum when the kernels' grids differ.  A
 * call that resumes right after a sync with p = 1 may therefore fuse an iteration that an
 * uninterrupted run ran as two kernels: x and v stay bit-identical, S may differ in its last bits.
 * trace and stats may be NULL.  Blocks (bounded) at every sync.  Errors: E_INVAL (bad
 * schedule, K_s < p_init + K_w for kind 1, p < 1, trace->var with fuse_intervals), E_TIMEOUT,
 * E_CUDA.  After an error the state is not resumable (restore a checkpoint). */
int adpsgd_run(adpsgd_ctx* ctx, const adpsgd_schedule* sched, adpsgd_state* state, int64_t k_end,
               adpsgd_trace* trace, adpsgd_stats* stats);

/* Column sharding: one problem split by columns over g processes (one per GPU).
 *
 * The local step is elementwise and the averaging reduces over replicas column by column, so a
 * problem can be cut into contiguous column ranges: shard r holds x and v as [n, P_r] (its
 * columns of every replica), its slice of h and c, and of the bf16 noise tensor.  Each shard runs
 * the same schedule.  At every sync the only exchange is the shard's two fp64 partial sums
 * (D and the loss; Algorithm 2's S_k line needs their totals): `gather` collects them from every
 * shard, and every shard adds them in shard order starting from 0, so all shards see the same S
 * and take the same decisions (16 bytes per shard per sync; no parameter traffic).
 *
 * gather(local, count, gathered, user) must place every shard's `count` doubles in shard order,
 * gathered[r * count + t] = local of shard r, and return 0 (nonzero: ADPSGD_E_PEER).  It is
 * called from the thread that called the library, on every shard at the same syncs.  With
 * shards == 1 it may be NULL.
 *
 * The noise of global column col0 + j is drawn with Philox block (col0 + j) div 4, so a sharded
 * run gives every column the same x and v as the unsharded run, bit for bit; D and the loss
 * differ from the unsharded run's only in the order of their fp64 additions. */
typedef int (*adpsgd_gather_fn)(const double* local, int64_t count, double* gathered, void* user);

typedef struct {
    int32_t shards;          /* g >= 1 */
    int32_t index;           /* this shard, 0 <= index < shards */
    int64_t col0;            /* global column of this shard's first column; a multiple of 4 */
    int64_t P_total;         /* columns of the whole problem (wire accounting); >= col0 + P */
    adpsgd_gather_fn gather; /* the exchange (see above) */
    void* user;              /* passed to gather */
} adpsgd_shard;

/* Make ctx one shard of a column-split problem (before its first step).  From then on the sums
 * that adpsgd_run, adpsgd_average_and_variance and adpsgd_variance report (and the per-iteration
 * variance record) are the totals over all shards, and the wire accounting uses P_total.
 * Errors: E_INVAL (shards < 1, index out of range, col0 not a multiple of 4 or negative,
 * P_total < col0 + P, (col0 + P) / 4 >= 2^32, gather NULL with shards > 1). */
int adpsgd_set_shard(adpsgd_ctx* ctx, const adpsgd_shard* shard);

/* Replica split: the paper's own mapping (Sec. IV-A), one process per node holding whole
 * replicas, averaging by an allreduce over the processes.  Process r holds cfg.n = n_local
 * replicas, the global replicas [replica0, replica0 + n_local) (Philox counter word 1 is the
 * global replica index), and owns one column chunk [col0, col0 + P_chunk) of the averaging.
 *
 * A sync runs as an allreduce split into its two halves, with the averaging kernel between them,
 * so that the mean is the one of Algorithm 2 formed column by column over all n_total replicas in
 * replica order (bit-identical to a single process holding them all):
 *   1. collective(ADPSGD_SCATTER_COLUMNS, user): the caller's all-to-all, enqueued on the context's
 *      stream, that leaves in chunk_x [n_total, P_chunk] every replica's values of this process's
 *      chunk, in global replica order (reduce-scatter's traffic: (g - 1)/g of the parameters);
 *   2. the averaging kernel on chunk_x (the chunk's mean, written to every row of chunk_x), its D
 *      and loss over the chunk;
 *   3. collective(ADPSGD_GATHER_AVERAGE, user): the caller's all-gather, enqueued on the stream,
 *      of every chunk's mean (row 0 of each process's chunk_x) into every row of x;
 *   4. the chunk sums through `gather`, added in process order (as for column shards).
 * A collective returns 0, or nonzero for ADPSGD_E_PEER.  Every process calls them at the same
 * syncs.  Not available with cfg.fuse_intervals, cfg.fuse_sync_step or the variance record. */
enum { ADPSGD_SCATTER_COLUMNS = 0, ADPSGD_GATHER_AVERAGE = 1 };
typedef int (*adpsgd_collective_fn)(int32_t op, void* user);

typedef struct {
    int32_t processes;       /* g >= 1 */
    int32_t rank;            /* this process, 0 <= rank < processes */
    int32_t replica0;        /* global index of this process's first replica */
    int32_t n_total;         /* replicas of the whole problem (>= replica0 + cfg.n) */
    int64_t col0;            /* this process's chunk of the averaging: columns [col0, col0 + P_chunk), */
    int64_t P_chunk;         /* col0 a multiple of 4, col0 + P_chunk <= cfg.P */
    float* chunk_x;          /* device [n_total, P_chunk], 16-byte aligned */
    adpsgd_collective_fn collective;
    adpsgd_gather_fn gather; /* every process's chunk sums, in process order (NULL with one process) */
    void* user;              /* passed to collective and gather */
} adpsgd_replica_split;

/* Make ctx one process of a replica split (before its first step).  chunk_x and the chunk's
 * slices of h and c (h + col0, c + col0) must stay valid until adpsgd_destroy.
 * Errors: E_INVAL (ranges, NULL collective, gather NULL with processes > 1, fuse_intervals or
 * fuse_sync_step set), E_ALIGN (chunk_x, or col0 leaving h + col0 unaligned). */
int adpsgd_set_replica_split(adpsgd_ctx* ctx, const adpsgd_replica_split* split);

/* The exchange alone, for tests and for callers that run their own averaging (pure host code):
 * gathers `count` doubles from every shard through shard->gather and writes their sums in shard
 * order, out[t] = ((0 + local_0[t]) + local_1[t]) + ...  Errors: E_INVAL, E_PEER. */
int adpsgd_shard_combine(const adpsgd_shard* shard, const double* local, int64_t count, double* out);

/* A part of the bf16 noise tensor that adpsgd_noise_fill_bf16 fills: rows (replicas)
 * [replica0, replica0 + n) and columns [col0, col0 + P) of the whole [n_total, P_total] tensor, as an
 * [n, P] array -- a column shard's slice (replica0 = 0) or a process's replicas (adpsgd_replica_split).
 * col0 a multiple of 4.  Enqueued only.  Errors: as adpsgd_noise_fill_bf16, and E_INVAL for a
 * negative replica0 or col0 not a multiple of 4. */
int adpsgd_noise_fill_bf16_part(uint64_t seed, int32_t n, int64_t P, int32_t replica0, int64_t col0, uint16_t* out,
                                void* stream);

/* The period rule alone (Algorithm 2, after the sync at iteration k; pure host code):
 * warm-up (k < K_w) and kind 0 leave the state unchanged; k < K_s: m += 1,
 * C2 += (S / gamma - C2) / m; otherwise p += 1 if S < lo * (gamma * C2), else p -= 1 if
 * S > hi * (gamma * C2), then p is clamped to [p_min, p_max].  *phase (may be NULL)
 * receives the phase code.  Errors: E_INVAL. */
int adpsgd_sched_on_sync(const adpsgd_schedule* sched, adpsgd_state* state, int64_t k, double S,
                         double gamma, int32_t* phase);

/* Step size of iteration k: (float)(lr0 * w_k * lr_factor^(number of milestones <= k)), the product
 * taken in fp64, with the warm-up multiple w_k = min(k div lr_warmup_len + 1, lr_warmup_steps)
 * (w_k = 1 without warm-up).  Errors: E_INVAL. */
int adpsgd_gamma(const adpsgd_schedule* sched, int64_t k, float* gamma_out);

/* Bytes a ring allreduce would move per node and in total for `rounds` syncs of P fp32
 * values, 2 (n-1)/n * 4P each (plus 2 (n-1)/n * 4 for the fp32 S_k if with_scalar): the
 * communication Algorithm 2 saves (Sec. IV-B).  Errors: E_INVAL. */
int adpsgd_wire_bytes(int32_t n, int64_t P, int64_t rounds, int32_t with_scalar,
                      double* per_node, double* total);

/* Raw Philox4x32-10 words of the noise stream: out[(i * nq + q) * 4 + r] = word r of
 * Philox(counter (q, i, k, tag), key (seed lo, seed hi)), i < n, q < nq.  out: device
 * uint32 [n, nq, 4].  Enqueued only.  Errors: E_INVAL (n * nq > 2^38, k >= 2^32), E_ALIGN, E_CUDA. */
int adpsgd_philox_fill(uint64_t seed, uint32_t tag, int32_t n, int64_t nq, int64_t k,
                       uint32_t* out, void* stream);

/* The fp32 normals the local step uses: out[i * P + j] = z[i, j] of stream `tag` at step k
 * (Box-Muller of words (0,1) -> elements 4q, 4q+1 and (2,3) -> 4q+2, 4q+3).  out: device fp32
 * [n, P].  Enqueued only.  Errors: E_INVAL (n * P > 2^40, P > 2^34), E_ALIGN, E_CUDA. */
int adpsgd_noise_fill_f32(uint64_t seed, uint32_t tag, int32_t n, int64_t P, int64_t k,
                          float* out, void* stream);

/* A pre-materialised bf16 noise tensor [n, P]: the step-0 normals of stream tag 1, rounded
 * to nearest-even bf16.  out: device, raw bf16 bits.  Enqueued only.  Errors: as above. */
int adpsgd_noise_fill_bf16(uint64_t seed, int32_t n, int64_t P, uint16_t* out, void* stream);

/* Moving a run's inputs and results between host and device: the state x, v and the
 * objective h, c in, the averaged parameters out.  The paper has no counterpart (it trains on
 * one machine per replica); these carry the end-to-end path from host buffers.
 *
 * adpsgd_copy_h2d copies `bytes` from host memory src to device memory dst, and
 * adpsgd_copy_d2h from device memory src to host memory dst, enqueued on `stream`.  When the
 * host buffer is page-locked (cudaHostAlloc, cudaHostRegister, PyTorch pinned memory), the
 * library's copy kernel moves the bytes through the buffer's mapped device address.  That
 * holds its throughput when other work loads the host memory, where the copy engines slow
 * down.  The kernel is used only when the device side is device memory of the current device;
 * managed memory, another device's memory, and host memory that is not page-locked go through
 * cudaMemcpyAsync.  The device side must be device (or managed) memory.  Both pointers 16-byte
 * aligned; bytes need not be a multiple of 16.
 * bytes == 0 does nothing.  Both buffers must hold `bytes` bytes from the given addresses: the
 * library cannot check a buffer's length, and a page-locked host buffer shorter than `bytes`
 * makes the copy kernel read or write past its mapping (a device fault).  The caller keeps both
 * buffers alive until the stream has passed the copy.
 * Errors: E_INVAL (NULL pointer with bytes > 0, bytes < 0, the device side not device memory,
 * the host side device memory), E_ALIGN, E_CUDA. */
int adpsgd_copy_h2d(void* dst, const void* src, int64_t bytes, void* stream);

/* The initialisation of Algorithms 1 and 2: every replica starts from the same model,
 * w_{0,i} = w_0, with zero momentum.  Sets each of the context's n rows of x to the P floats at
 * w0 and v to zero, enqueued on the context's stream (a column shard passes its own P columns of
 * w_0).  w0: fp32 [P], host or device memory, kept alive by the caller until the stream has
 * passed the call; it may be a row of x.  Device memory of the current device and page-locked
 * host memory are read once by a broadcast kernel (host memory through its mapped address, so a
 * run's initial model crosses the host link once, not n times); other memory is first copied
 * into row 0 of x by cudaMemcpyAsync.  Errors: E_INVAL (NULL), E_CUDA. */
int adpsgd_init_replicas(adpsgd_ctx* ctx, const float* w0);
int adpsgd_copy_d2h(void* dst, const void* src, int64_t bytes, void* stream);

/* Device time of the kernels launched through ctx while cfg.time_kernels was set, summed from
 * CUDA events on ctx's stream since init or the last reset (waits for them, bounded), over the
 * timed launches only (every time_kernels-th); *_launches counts those timed launches.
 * Errors: E_INVAL (out NULL), E_STATE (timing off), E_TIMEOUT, E_CUDA. */
int adpsgd_kernel_times(adpsgd_ctx* ctx, adpsgd_kernel_timing* out);
int adpsgd_reset_kernel_times(adpsgd_ctx* ctx);

/* Test hook: when force_incomplete is nonzero every bounded wait of ctx behaves as if the
 * awaited work never finished, so the wait returns ADPSGD_E_TIMEOUT after
 * cfg.wait_timeout_ms.  Only for exercising the timeout path. */
int adpsgd_test_force_incomplete(adpsgd_ctx* ctx, int32_t force_incomplete);

/* Synchronise the context's stream (bounded) and release the context.  NULL is a no-op. */
void adpsgd_destroy(adpsgd_ctx* ctx);

/* Static text for a status code, and the calling thread's last CUDA error detail. */
const char* adpsgd_strerror(int status);
const char* adpsgd_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* ADPSGD_H */
