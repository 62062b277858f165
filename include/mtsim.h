/*
 * mtsim.h -- C ABI of libmtsim, a batched GPU simulation of the multi-tier
 * Llumnix-style LLM-serving scheduler of "Beyond Binary Priorities:
 * Multi-Tier SLA Scheduling for LLM Serving" (Sec. 3).
 *
 * One simulation object holds R independent replicas.  A replica is a
 * serving cluster of N instances ("Llumlets", Sec. 3.1) with M KV-cache blocks
 * of T tokens each and a maximum running batch of Bmax requests, fed by its
 * own request trace.  Each simulation step of a replica processes every event
 * at the replica's next event time t, in this order:
 *   1. iteration ends at instances whose batch finishes at t (token
 *      accounting, request completion, one copy stage of an outbound
 *      migration, Sec. 3.5 Fig. 4);
 *   2. dispatch of the requests arriving at t, tier 0 first and FCFS within a
 *      tier, each to the instance of highest freeness F (Sec. 3.4), where
 *      F = (M - sum_r V(r)) / B (Sec. 3.2 Eq. 1-2) and the virtual usage
 *      includes the per-tier headroom H_k of every tier present, charged once
 *      per tier (Sec. 3.3 Eq. 3-4); an instance that is draining (see
 *      sim_set_drain) has infinite virtual usage and gets no request unless
 *      every instance drains, then the freest of them does (Sec. 3.4-3.5);
 *   3. at every interval ("tick"): the auto-scaling signal when enabled
 *      (mean normal-priority freeness against two thresholds, Sec. 3.6), then
 *      pairing of low- and high-freeness instances while max F - min F >=
 *      theta, draining instances first and without the threshold (Sec. 3.5);
 *   4. batch formation at idle instances (continuous batching with
 *      priority-ordered queues, KV growth and preemption, Sec. 2.2, 3.1) under
 *      the integer iteration-time model base + a*prefill_tokens + b*decodes.
 * All quantities are integers (blocks, tokens, microseconds); freeness is
 * compared exactly.  Results are deterministic and independent of how the
 * replicas are batched or how a run is split into sim_run calls.
 *
 * Conventions for every entry point:
 *  - Return value: SIM_OK (0) or a negative SIM_ERR_* code; sim_last_error()
 *    then describes the failure.  A failed call leaves the object usable
 *    unless the code is SIM_ERR_CUDA.
 *  - Pointers named "host" are host memory; pointers documented as
 *    "host or device" follow the call's on_device flag (0 = host, 1 = device
 *    memory of the simulation's GPU).  Input buffers are copied; the caller
 *    keeps ownership of every buffer it passes.  The sim_t object owns all of
 *    its device memory.
 *  - Work is queued on the CUDA stream given to sim_create.  Calls that return
 *    data to the host (sim_load_trace's validation, sim_run with a non-NULL
 *    num_unfinished, sim_metrics) synchronise that stream; nothing else does.
 *  - An object must not be used from two host threads at once.
 */
#ifndef MTSIM_H
#define MTSIM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ------------------------------------------------------------- limits --- */
#define SIM_MAX_TIERS 16        /* K <= 16 priority tiers, tier 0 highest (Sec. 4.2) */
#define SIM_MAX_INSTANCES 256   /* N */
#define SIM_MAX_BATCH 64        /* Bmax */
#define SIM_MAX_BLOCKS 65535    /* M */

/* --------------------------------------------------------- return codes --- */
#define SIM_OK 0
#define SIM_ERR_ARG (-1)        /* invalid argument or limit exceeded */
#define SIM_ERR_TRACE (-2)      /* malformed trace (see sim_load_trace) */
#define SIM_ERR_STATE (-3)      /* call out of order (e.g. sim_run before sim_load_trace) */
#define SIM_ERR_OOM (-4)        /* device allocation failed */
#define SIM_ERR_OVERFLOW (-5)   /* a time or counter would exceed its 32-bit field */
#define SIM_ERR_CUDA (-7)       /* CUDA runtime error; the object should be destroyed */
#define SIM_ERR_INTERNAL (-8)   /* a device-side consistency check failed */
#define SIM_ERR_DEADLOCK (-10)  /* no event left while requests are unfinished */
#define SIM_ERR_UNFINISHED (-11) /* sim_run_static: some replica did not reach SIM_REPLICA_DONE */

/* Per-replica status (sim_replica_stats_t.status). */
#define SIM_REPLICA_DONE 0      /* every request of the replica has finished */
#define SIM_REPLICA_RUNNING 1   /* stopped by the step limit; sim_run resumes it */
/* negative values: SIM_ERR_OVERFLOW, SIM_ERR_INTERNAL, SIM_ERR_DEADLOCK */

#define SIM_POLICY_LLUMNIX_MT 0 /* multi-tier Llumnix global scheduler (Sec. 3) */

/* Migration log record kinds (Sec. 3.5). */
#define SIM_EV_QUEUED 0  /* a queued request moved to the destination at once (0 blocks) */
#define SIM_EV_START 1   /* staged copy of a running request began (blocks = its KV size) */
#define SIM_EV_COMMIT 2  /* the request committed to the destination (blocks = its KV size) */
#define SIM_EV_ABORT 3   /* staged copy abandoned (blocks = blocks copied so far) */
/* Auto-scaling signal records (Sec. 3.6): request = SIM_NONE32, src = dst = 255, blocks = 0. */
#define SIM_EV_SCALE_OUT 4  /* mean F_normal below the scale-out threshold at this tick */
#define SIM_EV_SCALE_IN 5   /* mean F_normal above the scale-in threshold at this tick */

#define SIM_NONE32 0xFFFFFFFFu  /* "not set" for 32-bit times */
#define SIM_NONE16 0xFFFFu      /* "not set" for 16-bit instance ids */

/* ---------------------------------------------------------------- types --- */
typedef struct sim sim_t; /* opaque, owned by the library */

typedef struct {
    int32_t num_replicas;        /* R >= 1 */
    int32_t num_instances;       /* N in [1, SIM_MAX_INSTANCES] */
    int32_t blocks_per_instance; /* M in [1, SIM_MAX_BLOCKS] KV blocks per instance */
    int32_t tokens_per_block;    /* T in [1, 64] tokens per KV block */
    int32_t max_batch;           /* Bmax in [1, SIM_MAX_BATCH] running requests per instance */
} sim_cluster_t;

/* Per-tier headroom H_k in blocks (Sec. 3.3 Eq. 3), one table per distinct
 * tier setting; every replica names its table.  All pointers are host. */
typedef struct {
    int32_t num_tables;             /* >= 1 */
    int32_t max_tiers;              /* row stride of headroom_blocks, in [1, SIM_MAX_TIERS] */
    const int32_t *num_tiers;       /* [num_tables]: K of each table, in [1, max_tiers] */
    const int32_t *headroom_blocks; /* [num_tables * max_tiers]: H_k >= 0 for k < K */
    const int32_t *replica_table;   /* [num_replicas]: table index of each replica */
} sim_tier_table_t;

typedef struct {
    int32_t policy;                     /* SIM_POLICY_LLUMNIX_MT */
    int32_t enable_migration;           /* 0 or 1 */
    int64_t iter_base_us;               /* iteration time = base, in [1, 2^24] */
    int64_t iter_us_per_prefill_token;  /*   + a * prefill tokens in the batch */
    int64_t iter_us_per_decode_seq;     /*   + b * decode requests in the batch; a, b in [0, 2^24] */
    int32_t migrate_blocks_per_iter;    /* S: KV blocks copied per source iteration, in [1, 65535] */
    int32_t theta_num, theta_den;       /* imbalance threshold theta = num/den (0.3 = 3/10) */
    int32_t event_log_capacity;         /* migration-log records kept per replica, in [0, 2^24] */
    int64_t migrate_interval_us;        /* tick period, in [1, 2^31] (50 ms in Sec. 3.5) */
    /* Auto-scaling signal (Sec. 3.4, 3.6), evaluated at every tick when
     * autoscale = 1: the mean over non-draining instances of the
     * normal-priority freeness F_normal = (M - running KV - HoL demand -
     * inbound reservation) / max(B, 1), i.e. Eq. 1 without the headroom
     * term, is compared exactly with scale_out_num / scale_den (strictly
     * below: scale-out) and scale_in_num / scale_den (strictly above:
     * scale-in).  The paper's thresholds are -1/2 and 3/2.  The signal is
     * reported (counters and log records); it adds or removes no instance.
     * With autoscale = 1 ticks happen even when migration is off.
     * autoscale = 0 ignores the three thresholds. */
    int32_t autoscale;                  /* 0 or 1 */
    int32_t scale_out_num, scale_in_num; /* in [-4096, 4096], scale_out_num < scale_in_num */
    int32_t scale_den;                  /* in [1, 64] */
} sim_policy_t;

/* Per-request outcome, 16 bytes.  Times are microseconds from the replica's
 * start; TTFT = first_token_us - arrival, E2E = finish_us - arrival.  The
 * preemption and migration counters are kept modulo 2^16 (each exactly: they
 * share the last 32-bit word, preemptions in the low half). */
typedef struct {
    uint16_t dispatch_instance;  /* instance chosen at arrival (SIM_NONE16 if not yet arrived) */
    uint16_t final_instance;     /* instance it finished on (SIM_NONE16 if unfinished) */
    uint32_t first_token_us;     /* SIM_NONE32 if no token yet */
    uint32_t finish_us;          /* SIM_NONE32 if unfinished */
    uint16_t n_preemptions;
    uint16_t n_migrations;       /* queued moves + committed running migrations */
} sim_request_result_t;

typedef struct {
    uint64_t steps;              /* distinct event times processed */
    uint64_t iterations;         /* batches formed */
    uint64_t member_iterations;  /* sum of batch sizes over all iterations */
    uint64_t events;             /* arrivals + first tokens + finishes + migrations + preemptions */
    uint32_t migrations;         /* queued moves + commits */
    uint32_t preemptions;
    uint32_t migration_starts;
    uint32_t migration_aborts;
    uint32_t log_events;         /* migration-log records produced (may exceed the capacity) */
    uint32_t finished;           /* requests finished */
    uint32_t last_time_us;       /* time of the last processed step */
    int32_t status;              /* SIM_REPLICA_* or a negative SIM_ERR_* code */
    uint32_t scale_out_signals;  /* ticks with a scale-out signal (Sec. 3.6) */
    uint32_t scale_in_signals;   /* ticks with a scale-in signal */
} sim_replica_stats_t;

typedef struct {
    uint32_t time_us;
    uint32_t request;            /* index within the replica's trace */
    uint16_t blocks;
    uint8_t src, dst;            /* instance indices (N <= 256) */
    uint8_t kind;                /* SIM_EV_* */
    uint8_t pad[3];
} sim_migration_event_t;

/* Per-tier latency statistics of one measure (Sec. 5.1, Sec. 5.3: the paper
 * reports TTFT, time between tokens and end-to-end latency per priority tier,
 * as distributions, means and P50 / P90 / P99).  992 bytes. */
#define SIM_HIST_BUCKETS 240
#define SIM_LAT_TTFT 0  /* first_token - arrival (prefill latency) */
#define SIM_LAT_TBT 1   /* floor((finish - first_token) / (O - 1)), requests with O >= 2 */
#define SIM_LAT_E2E 2   /* finish - arrival */
typedef struct {
    uint32_t count;              /* finished requests of the tier counted */
    uint32_t max_us;             /* exact maximum (0 if count = 0) */
    uint64_t sum_us;             /* exact sum; mean = sum_us / count */
    uint32_t p50_us, p90_us, p99_us; /* nearest-rank percentiles: exactly the value of rank
                                        ceil(p * count / 100) in ascending order; 0 if count = 0 */
    uint32_t pad;
    /* hist[b]: requests whose value v falls in bucket b: b = v for v < 8,
     * else b = 8 * (e - 3) + floor(v / 2^(e-3)) with e = floor(log2 v):
     * eight equal buckets per power of two, floors 0..7, 8, 9, .., 15, 16,
     * 18, .., 30, 32, 36, ... */
    uint32_t hist[SIM_HIST_BUCKETS];
} sim_latency_stats_t;

/* Optional device allocator, e.g. a framework's caching allocator.  alloc
 * returns a device pointer (16-byte aligned at least) or NULL; free releases
 * one.  Both are called on the calling host thread with the simulation's
 * stream.  NULL allocator: the library uses cudaMallocAsync / cudaFreeAsync
 * on that stream. */
typedef void *(*sim_alloc_fn)(void *ctx, size_t bytes, void *cuda_stream);
typedef void (*sim_free_fn)(void *ctx, void *ptr, size_t bytes, void *cuda_stream);
typedef struct {
    void *ctx;
    sim_alloc_fn alloc;
    sim_free_fn free;
} sim_allocator_t;

/* ---------------------------------------------------------- entry points --- */

/* Creates a simulation of cluster->num_replicas replicas on the current CUDA
 * device.  The cluster, tier tables and policy are validated (limits above;
 * additionally M + sum_k H_k must stay below 2^19 for every table) and
 * copied.  cuda_stream is a cudaStream_t (NULL = legacy default stream);
 * allocator may be NULL.  Allocates the per-replica and per-instance state
 * (about N * (67 + 14 * K + T) + N * Bmax * 16 + 16 * log capacity + 4 * K +
 * 500 bytes per replica).  On success *out receives the object and SIM_OK is returned;
 * on failure *out is NULL and sim_last_error(NULL) describes the error. */
int sim_create(const sim_cluster_t *cluster, const sim_tier_table_t *tiers, const sim_policy_t *policy,
               void *cuda_stream, const sim_allocator_t *allocator, sim_t **out);

/* Loads the request traces and resets every replica to t = 0.
 * replica_offsets (host, [R + 1]): replica r owns trace records
 * [replica_offsets[r], replica_offsets[r+1]); offsets[0] = 0, non-decreasing,
 * at most 2^32 - 2 records per replica.  arrival_us, prompt_len, output_len,
 * tier ([total] each, host or device per on_device): arrival times in
 * microseconds from the replica's start, sorted non-decreasing within a
 * replica (requests with equal times are dispatched tier-major, then in trace
 * order), prompt length P >= 1 and output length O >= 1 in tokens with
 * P + O <= min(M * T, 65536), and tier < the replica's K.  Violations return
 * SIM_ERR_TRACE and leave no trace loaded.  Synchronises the stream. */
int sim_load_trace(sim_t *sim, const int64_t *replica_offsets, const uint32_t *arrival_us,
                   const uint16_t *prompt_len, const uint16_t *output_len, const uint8_t *tier, int on_device);

/* Resets every replica of the loaded trace to t = 0 (asynchronous). */
int sim_reset(sim_t *sim);

/* Sets the drain schedule (Sec. 3.4-3.5; the last case of Eq. 2): instance i
 * of replica r is draining at every step whose time is >=
 * drain_start_us[r * N + i] (SIM_NONE32 = never).  A draining instance keeps
 * running its own batches and queue, but its virtual usage is infinite: it
 * receives no dispatch while some instance of its replica is not draining,
 * it is the first migration source at every tick (no imbalance threshold)
 * and never a destination, and it is left out of the auto-scaling mean.
 * drain_start_us: [R * N] times, host or device per on_device, copied (a host
 * buffer may be reused when the call returns); NULL removes the schedule.
 * The schedule takes effect at the next sim_load_trace or sim_reset.
 * Returns SIM_ERR_OOM if its device copy (4 * R * N bytes) cannot be
 * allocated.  sim_run_static has no drain schedule. */
int sim_set_drain(sim_t *sim, const uint32_t *drain_start_us, int on_device);

/* Replaces the headroom tables (adaptive headroom, Sec. 6 "Adaptive
 * headroom allocation": H_p adjusted while the system runs).
 * headroom_blocks: host, [num_tables * max_tiers] in the layout of
 * sim_tier_table_t.headroom_blocks (entries k >= the table's K are ignored),
 * H_k >= 0 and M + sum_k H_k below 2^19 for every table, else SIM_ERR_ARG and
 * nothing changes.  Every replica then uses its table's new values from the
 * next step it processes (the next sim_run); each instance's headroom of the
 * tiers present on it is recomputed.  The tables stay in force for later
 * sim_reset and sim_load_trace calls.  Copied (the buffer may be reused
 * when the call returns); queues a small kernel on the stream.  A replica
 * stopped by a sim_run step limit has processed exactly that many steps, so
 * a caller that changes the tables between calls of max_steps_per_replica E
 * applies them at step indices E, 2E, ...: the same schedule runs the same
 * way in every chunking. */
int sim_set_headroom(sim_t *sim, const int32_t *headroom_blocks);

/* Sets the order in which sim_run starts replicas: the persistent grid takes
 * replicas from a counter, and with an order set the k-th replica taken is
 * order[k].  Starting the replicas with the most work first shortens the
 * tail of a launch that runs more replicas than fit on the GPU at once.
 * Results never depend on the order.  order: host, [R], a permutation of
 * 0..R-1 (checked: anything else returns SIM_ERR_ARG and keeps the previous
 * order); copied, so the buffer may be reused when the call returns.  NULL
 * restores trace order.  Takes effect at the next sim_run.  The paper has no
 * counterpart; this is a scheduling aid of the batched simulation. */
int sim_set_order(sim_t *sim, const int32_t *order);

/* Advances every unfinished replica by at most max_steps_per_replica steps
 * (>= 1) in one persistent kernel launch; a later call resumes where this one
 * stopped.  If num_unfinished (host) is non-NULL the call synchronises and
 * stores the number of replicas not yet SIM_REPLICA_DONE; otherwise it
 * returns as soon as the work is queued.  Returns SIM_ERR_STATE without a
 * loaded trace. */
int sim_run(sim_t *sim, int64_t max_steps_per_replica, int64_t *num_unfinished);

/* Copies results out (host or device per on_device; any pointer may be NULL
 * to skip that output) and synchronises the stream.
 * per_request [total records], in trace order; per_replica [R];
 * events [R * event_log_capacity]: replica r's first
 * min(log_events, capacity) records start at r * capacity, in the order the
 * simulation produced them. */
int sim_metrics(sim_t *sim, sim_request_result_t *per_request, sim_replica_stats_t *per_replica,
                sim_migration_event_t *events, int on_device);

/* Per-tier latency statistics of the current results, computed on the device:
 * out[(r * max_tiers + k) * 3 + m] for replica r, tier k < max_tiers (tiers
 * beyond a replica's K have count 0) and measure m = SIM_LAT_*.  Counts only
 * requests that have finished, so it may be called between sim_run calls.
 * out is host or device per on_device, [R * max_tiers * 3] records.  Host
 * output synchronises the stream (and allocates a device staging buffer of
 * the same size on first use); device output is asynchronous.  The first
 * call also allocates the percentile selection scratch, 3,120 bytes per
 * (replica, tier, measure).  Returns SIM_ERR_STATE before sim_load_trace. */
int sim_latency_stats(sim_t *sim, sim_latency_stats_t *out, int on_device);

/* Releases everything the object owns (synchronises the stream first).
 * NULL is ignored. */
void sim_destroy(sim_t *sim);

/* Text of the last error on this object, or of the last failed sim_create on
 * this thread when sim is NULL.  Valid until the next call on the object. */
const char *sim_last_error(const sim_t *sim);

/* Static description of a return code. */
const char *sim_strerror(int code);

/* Device bytes the object holds (0 for NULL). */
size_t sim_device_bytes(const sim_t *sim);

/* Launch configuration of the simulation kernel that the next sim_run on
 * this object will use (a measurement aid: with it, kernel time, SM clock and
 * step counts give cycles per replica-step per resident warp).  The paper has
 * no counterpart.  One warp simulates one replica; the grid is persistent
 * and takes replicas from a work counter. */
typedef struct {
    int32_t grid_blocks;        /* blocks of one sim_run launch */
    int32_t block_threads;      /* threads per block (32 per replica in flight) */
    int32_t blocks_per_sm;      /* resident blocks per SM that registers and shared memory allow */
    int32_t instances_per_lane; /* instances each lane of a replica's warp owns */
    int32_t slots_in_shared;    /* 1: running-request records stay in shared memory while a warp owns a replica */
    int32_t extended;           /* 1: the variant with draining and the auto-scaling signal */
    int64_t shared_bytes;       /* dynamic shared memory per block */
} sim_launch_info_t;

/* Fills *out (host) for the kernel variant sim_run would launch now (it
 * depends on whether a drain schedule is set or the auto-scaling signal is
 * on).  Returns SIM_ERR_ARG for NULL arguments. */
int sim_launch_info(const sim_t *sim, sim_launch_info_t *out);

/* Scratch memory behind sim_run_static: one fixed device array per GPU. */
#define SIM_STATIC_SCRATCH_BYTES (32u << 20)

/* Allocation-free variant of a whole simulation (the paper has no
 * counterpart; this is a library service).  For callers that cannot call
 * cudaMalloc: code running inside a process whose device memory is entirely
 * owned by another allocator or budget, plugins and hooks that must not touch
 * the CUDA allocator at all, or contexts where an allocation's implicit
 * synchronisation is not allowed.  It simulates every replica of the given
 * trace from t = 0 to completion, exactly like sim_create + sim_load_trace +
 * sim_run + sim_metrics, but allocates nothing: the simulation state lives in
 * a file-scope device array of SIM_STATIC_SCRATCH_BYTES (32 MiB) that every
 * GPU which loads the library holds until the process exits.
 *
 * cluster, tiers, policy: as for sim_create (host).  replica_offsets: host,
 * [R + 1], as for sim_load_trace.  arrival_us, prompt_len, output_len, tier:
 * DEVICE pointers to the trace, as for sim_load_trace.  per_request
 * ([total records]) and per_replica ([R]) are DEVICE output buffers owned by
 * the caller; events is a DEVICE buffer of R * policy->event_log_capacity
 * records or NULL (then no log is written).  cuda_stream is a cudaStream_t
 * (NULL = legacy default stream).
 *
 * Limits: the state of all replicas must fit in the scratch array, about
 * R * (N * (67 + 14 * K + T) + N * Bmax * 16 + 600) + 16 * total records bytes;
 * a larger problem returns SIM_ERR_ARG with the size it needed.  Every call
 * looks up the array's device address (cudaGetSymbolAddress) with the
 * caller's device current, so the address stays right after a
 * cudaDeviceReset; the first call on a device also loads the library's
 * kernels there, so make the first call before any stream capture.
 * Every call uses the same array and overwrites what the previous call left
 * there; two calls whose work overlaps on the GPU (other streams, other host
 * threads) race and corrupt each other's results.  Validates the trace
 * (SIM_ERR_TRACE) and synchronises the stream before returning.  Returns
 * SIM_ERR_UNFINISHED, with every output written, when some replica did not
 * finish: per_replica[r].status then gives each replica's outcome (a
 * negative SIM_ERR_* code, or SIM_REPLICA_RUNNING if it reached 2^32 - 1
 * steps).  Errors are described by sim_last_error(NULL). */
int sim_run_static(const sim_cluster_t *cluster, const sim_tier_table_t *tiers, const sim_policy_t *policy,
                   const int64_t *replica_offsets, const uint32_t *arrival_us, const uint16_t *prompt_len,
                   const uint16_t *output_len, const uint8_t *tier, sim_request_result_t *per_request,
                   sim_replica_stats_t *per_replica, sim_migration_event_t *events, void *cuda_stream);

#ifdef __cplusplus
}
#endif

#endif /* MTSIM_H */
