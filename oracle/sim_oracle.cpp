/*
 * sim_oracle.cpp -- reference CPU simulator (TEST INFRASTRUCTURE ONLY).
 *
 * Only the test suite, the package smoke check and the benchmark's CPU
 * baseline may load this library.  It is a plain, single-threaded,
 * event-driven simulation of one serving cluster ("replica") under the
 * multi-tier Llumnix-style global scheduler of "Beyond Binary Priorities:
 * Multi-Tier SLA Scheduling for LLM Serving".  It is written for clarity, not
 * speed: std::vector / std::deque containers, linear scans, and freeness
 * compared exactly by 64-bit cross-multiplication of (numerator, denominator)
 * pairs.  It shares no code with the CUDA simulator.
 *
 * Model (all integers; time in microseconds):
 *  - N instances per replica, each with M KV blocks of T tokens and a maximum
 *    batch of Bmax running requests; K priority tiers, tier 0 highest
 *    (Sec. 4.2); per-tier headroom H_k in blocks (Sec. 3.3, Eq. 3).
 *  - Freeness F = (M - sum_r V(r)) / B (Sec. 3.2, Eq. 1) where the virtual
 *    usage (Sec. 3.2, Eq. 2) is the KV blocks of running requests, plus the
 *    block demand of the head-of-line queued request, plus the headroom H_k of
 *    every tier k present on the instance, charged once per tier (Sec. 3.3,
 *    Eq. 4), plus blocks already copied in by an inbound migration.  B is the
 *    number of running requests, taken as 1 when it is 0.
 *  - Dispatch (Sec. 3.4): arrivals go, tier 0 first and FCFS within a tier,
 *    to the instance of highest freeness (ties: lowest index).
 *  - Migration (Sec. 3.5): every interval, while max F - min F >= theta over
 *    instances not already migrating, pair the least free instance (source)
 *    with the freest (destination); the source moves its lowest-priority
 *    queued request at once, or else starts a staged copy of a low-priority,
 *    small-KV running request: each source iteration end copies up to S
 *    blocks; the request commits to the destination when all of its blocks
 *    are copied.
 *  - Draining (Sec. 3.4, Sec. 3.5, the last case of Eq. 2): from its drain
 *    start time on, an instance's virtual usage is infinite.  It gets no
 *    dispatch unless every instance drains (then the least loaded draining
 *    one, by ordinary freeness, gets it), it is the first migration source at
 *    every tick (no threshold: its freeness is minus infinity) and never a
 *    destination.  Its own batches keep running.
 *  - Auto-scaling signal (Sec. 3.4, Sec. 3.6): at every tick, the mean of the
 *    normal-priority freeness F_normal (Eq. 1 without the headroom term) over
 *    the instances that are not draining is compared, exactly, with the
 *    scale-out and scale-in thresholds (-1/2 and 3/2 in the paper); each
 *    signal is counted and logged.  Nothing is added or removed: the signal
 *    is an output.
 *  - Local scheduling (Sec. 2.2, Sec. 3.1): continuous batching with
 *    priority-ordered queues (one FCFS bucket per tier), block-level KV
 *    allocation (ceil((P+g)/T) blocks for P prompt and g generated tokens),
 *    recompute preemption of the lowest-priority newest request, strict
 *    head-of-line admission, and iteration time
 *    base + a * prefill_tokens + b * decode_requests.
 * Every reading taken where the paper is silent is listed beside the code
 * that takes it.
 */
#include <algorithm>
#include <atomic>
#include <cstdint>
#include <cstring>
#include <deque>
#include <thread>
#include <vector>

namespace {

constexpr uint32_t NONE32 = 0xFFFFFFFFu;
constexpr int MAXK = 16;

enum Status { ST_DONE = 0, ST_INCOMPLETE = 1, ST_ARG = -1, ST_TRACE = -2, ST_OVERFLOW = -5,
              ST_INVARIANT = -9, ST_DEADLOCK = -10 };
enum EvKind { EV_QUEUED = 0, EV_START = 1, EV_COMMIT = 2, EV_ABORT = 3, EV_SCALE_OUT = 4, EV_SCALE_IN = 5 };
enum ReqState { PENDING = 0, WAITING = 1, RUNNING = 2, DONE = 3 };
enum MigRole { MIG_NONE = 0, MIG_SRC = 1, MIG_DST = 2 };

}  // namespace

extern "C" {

typedef struct {
    int32_t num_instances;       /* N */
    int32_t blocks_per_instance; /* M */
    int32_t tokens_per_block;    /* T */
    int32_t max_batch;           /* Bmax */
    int32_t num_tiers;           /* K */
    int32_t headroom[MAXK];      /* H_k in blocks */
    int64_t iter_base_us, iter_us_per_prefill_token, iter_us_per_decode_seq;
    int32_t migrate_blocks_per_iter; /* S */
    int32_t enable_migration;
    int64_t migrate_interval_us;
    int32_t theta_num, theta_den;
    int32_t check_invariants;
    int32_t autoscale;               /* evaluate the auto-scaling signal at every tick */
    int32_t scale_out_num, scale_in_num, scale_den;  /* thresholds on the mean F_normal */
    int32_t pad_;
    const uint32_t *drain_start_us;  /* [num_instances] or NULL: instance i drains from that time on */
    /* Headroom schedule (adaptive headroom, Sec. 6 "Adaptive headroom
     * allocation"): change j replaces the table H by
     * headroom_change_table[j * MAXK .. + num_tiers) just before the step of
     * index headroom_change_step[j] (0-based count of the steps processed so
     * far) is processed.  Steps non-decreasing; 0 changes = the static table. */
    int32_t n_headroom_changes;
    int32_t pad2_;
    const int64_t *headroom_change_step;   /* [n_headroom_changes] */
    const int32_t *headroom_change_table;  /* [n_headroom_changes * MAXK] */
} oracle_config_t;

typedef struct {
    int64_t steps;               /* distinct event times processed */
    int64_t iterations;          /* batches formed */
    int64_t member_iterations;   /* sum of batch sizes over iterations */
    int64_t events;              /* arrivals + first tokens + finishes + migrations + preemptions */
    int64_t migrations;          /* queued moves + committed running migrations */
    int64_t preemptions;
    int64_t migration_starts;
    int64_t migration_aborts;
    int64_t log_events;          /* migration-log records produced (may exceed capacity) */
    int64_t finished;
    uint32_t last_time;
    int32_t status;
    int64_t scale_out_signals;   /* ticks at which the mean F_normal was below the scale-out threshold */
    int64_t scale_in_signals;    /* ticks at which it was above the scale-in threshold */
} oracle_stats_t;

typedef struct {
    int64_t nreq;
    const uint32_t *arrival_us;
    const uint16_t *prompt_len;
    const uint16_t *output_len;
    const uint8_t *tier;
    /* outputs, [nreq] each */
    int32_t *dispatch_instance;
    int32_t *final_instance;
    uint32_t *first_token_us;
    uint32_t *finish_us;
    int32_t *n_migrations;
    int32_t *n_preemptions;
    /* migration log, [log_capacity] each; may be NULL when capacity is 0 */
    int64_t log_capacity;
    uint32_t *ev_time;
    uint32_t *ev_req;
    int32_t *ev_src;
    int32_t *ev_dst;
    int32_t *ev_blocks;
    int32_t *ev_kind;
} oracle_io_t;

}  // extern "C"

namespace {

struct Req {
    uint32_t arrival = 0;
    int P = 0, O = 0, tier = 0;
    int g = 0;       /* tokens generated so far */
    int blocks = 0;  /* KV blocks held while running */
    int where = -1;  /* instance holding it (waiting or running) */
    int state = PENDING;
};

struct Inst {
    int free_blocks = 0;
    int reserved_in = 0;            /* blocks copied in for an in-flight inbound migration */
    std::vector<int> running;       /* admission order */
    std::vector<std::deque<int>> waiting;  /* one FCFS bucket per tier */
    std::vector<int> cnt;           /* requests of each tier present (running or waiting) */
    bool busy = false;
    uint32_t busy_until = 0;
    int batch_size = 0;             /* the current iteration runs running[0 .. batch_size) */
    int mig_role = MIG_NONE, mig_peer = -1, mig_req = -1, mig_copied = 0;
};

struct Sim {
    const oracle_config_t &c;
    oracle_io_t &io;
    oracle_stats_t &st;
    std::vector<Req> req;
    std::vector<Inst> inst;
    int64_t cursor = 0;           /* next request not yet arrived */
    int64_t next_tick = 0;
    uint32_t now = 0;
    int32_t H[MAXK];              /* the headroom table in force (c.headroom, then the schedule's) */
    int32_t next_change = 0;      /* next entry of the headroom schedule */

    Sim(const oracle_config_t &cfg, oracle_io_t &o, oracle_stats_t &s) : c(cfg), io(o), st(s) {}

    /* ---- helpers ------------------------------------------------------- */
    int need_blocks(const Req &r) const {  /* KV needed to run the next iteration */
        return (r.P + r.g + c.tokens_per_block - 1) / c.tokens_per_block;
    }
    int hol_request(const Inst &in) const {  /* front of the highest-priority non-empty bucket */
        for (int k = 0; k < c.num_tiers; ++k)
            if (!in.waiting[k].empty()) return in.waiting[k].front();
        return -1;
    }
    /* Freeness as an exact fraction num/den (Sec. 3.2 Eq. 1-2, Sec. 3.3 Eq. 4). */
    void freeness(const Inst &in, int64_t &num, int64_t &den) const {
        int64_t usage = 0;
        for (int r : in.running) usage += req[r].blocks;               /* physUsage of running requests */
        int h = hol_request(in);
        if (h >= 0) usage += need_blocks(req[h]);                      /* HoL demand; other queued: 0 */
        for (int k = 0; k < c.num_tiers; ++k)
            if (in.cnt[k] > 0) usage += H[k];                          /* H_k once per present tier */
        usage += in.reserved_in;                                       /* inbound migration copy */
        num = (int64_t)c.blocks_per_instance - usage;
        den = in.running.empty() ? 1 : (int64_t)in.running.size();
    }
    /* Normal-priority freeness (Sec. 3.4): the same fraction without the headroom term. */
    void normal_freeness(const Inst &in, int64_t &num, int64_t &den) const {
        int64_t usage = 0;
        for (int r : in.running) usage += req[r].blocks;
        int h = hol_request(in);
        if (h >= 0) usage += need_blocks(req[h]);
        usage += in.reserved_in;
        num = (int64_t)c.blocks_per_instance - usage;
        den = in.running.empty() ? 1 : (int64_t)in.running.size();
    }
    /* An instance drains from its drain start time on (Sec. 3.5). */
    bool draining(int i) const { return c.drain_start_us != nullptr && now >= c.drain_start_us[i]; }
    /* true when F_a > F_b */
    bool freer(int a, int b) const {
        int64_t na, da, nb, db;
        freeness(inst[a], na, da);
        freeness(inst[b], nb, db);
        return na * db > nb * da;
    }

    void log_event(int kind, int r, int src, int dst, int blocks) {
        int64_t k = st.log_events++;
        if (k < io.log_capacity) {
            io.ev_time[k] = now;
            io.ev_req[k] = (uint32_t)r;
            io.ev_src[k] = src;
            io.ev_dst[k] = dst;
            io.ev_blocks[k] = blocks;
            io.ev_kind[k] = kind;
        }
    }
    void remove_running(Inst &in, int r) {
        auto it = std::find(in.running.begin(), in.running.end(), r);
        in.running.erase(it);
    }

    /* ---- migration (Sec. 3.5) ------------------------------------------ */
    void clear_migration(Inst &s, Inst &d) {
        s.mig_role = d.mig_role = MIG_NONE;
        s.mig_peer = d.mig_peer = -1;
        s.mig_req = -1;
        s.mig_copied = 0;
    }
    void abort_migration(int si) {
        Inst &s = inst[si];
        Inst &d = inst[s.mig_peer];
        d.free_blocks += s.mig_copied;   /* copied blocks are released on the destination */
        d.reserved_in -= s.mig_copied;
        log_event(EV_ABORT, s.mig_req, si, s.mig_peer, s.mig_copied);
        st.migration_aborts++;
        clear_migration(s, d);
    }
    void commit_migration(int si) {
        Inst &s = inst[si];
        int di = s.mig_peer;
        Inst &d = inst[di];
        Req &r = req[s.mig_req];
        s.free_blocks += r.blocks;
        remove_running(s, s.mig_req);
        d.reserved_in -= s.mig_copied;   /* the copied blocks now belong to r */
        d.running.push_back(s.mig_req);  /* joins the destination's next batch */
        s.cnt[r.tier]--;
        d.cnt[r.tier]++;
        r.where = di;
        io.n_migrations[s.mig_req]++;
        st.migrations++;
        st.events++;
        log_event(EV_COMMIT, s.mig_req, si, di, r.blocks);
        clear_migration(s, d);
    }
    /* One copy stage at the end of a source iteration (Fig. 4). */
    void migration_stage(int si) {
        Inst &s = inst[si];
        Inst &d = inst[s.mig_peer];
        Req &r = req[s.mig_req];
        int c_blocks = std::min(c.migrate_blocks_per_iter, r.blocks - s.mig_copied);
        if (d.free_blocks < c_blocks) { abort_migration(si); return; }
        d.free_blocks -= c_blocks;
        d.reserved_in += c_blocks;
        s.mig_copied += c_blocks;
        if (s.mig_copied == r.blocks && (int)d.running.size() < c.max_batch) commit_migration(si);
    }

    /* ---- local scheduler ----------------------------------------------- */
    void finish_request(int i, int r) {
        Inst &in = inst[i];
        Req &q = req[r];
        io.finish_us[r] = now;
        io.final_instance[r] = i;
        in.free_blocks += q.blocks;
        q.blocks = 0;
        remove_running(in, r);
        in.cnt[q.tier]--;
        q.state = DONE;
        q.where = -1;
        st.finished++;
        st.events++;
        if (in.mig_role == MIG_SRC && in.mig_req == r) abort_migration(i);
    }
    void preempt(int i, int v) {  /* recompute-style: keeps g, frees KV, back to the queue front */
        Inst &in = inst[i];
        Req &q = req[v];
        in.free_blocks += q.blocks;
        q.blocks = 0;
        remove_running(in, v);
        in.waiting[q.tier].push_front(v);
        q.state = WAITING;
        io.n_preemptions[v]++;
        st.preemptions++;
        st.events++;
        if (in.mig_role == MIG_SRC && in.mig_req == v) abort_migration(i);
    }

    /* Phase 1: iteration ends at instances whose batch completes at `now`. */
    void phase_completions() {
        for (int i = 0; i < c.num_instances; ++i) {
            Inst &in = inst[i];
            if (!in.busy || in.busy_until != now) continue;
            in.busy = false;
            std::vector<int> members(in.running.begin(), in.running.begin() + in.batch_size);
            in.batch_size = 0;
            for (int r : members) {
                Req &q = req[r];
                q.g += 1;  /* a prefill yields the first token, a decode one more */
                if (io.first_token_us[r] == NONE32) {
                    io.first_token_us[r] = now;
                    st.events++;
                }
                if (q.g == q.O) finish_request(i, r);
            }
            if (in.mig_role == MIG_SRC) migration_stage(i);
        }
    }

    /* Phase 2: dispatch of the arrivals at `now` (Sec. 3.4). */
    void phase_dispatch() {
        std::vector<int> arr;
        while (cursor < io.nreq && io.arrival_us[cursor] == now) arr.push_back((int)cursor++);
        std::stable_sort(arr.begin(), arr.end(), [&](int a, int b) { return req[a].tier < req[b].tier; });
        for (int r : arr) {
            int best = -1;  /* freest instance that is not draining, lowest index on ties */
            for (int i = 0; i < c.num_instances; ++i)
                if (!draining(i) && (best < 0 || freer(i, best))) best = i;
            if (best < 0)   /* every instance drains: the least loaded of them */
                for (int i = 0; i < c.num_instances; ++i)
                    if (best < 0 || freer(i, best)) best = i;
            Req &q = req[r];
            inst[best].waiting[q.tier].push_back(r);
            inst[best].cnt[q.tier]++;
            q.state = WAITING;
            q.where = best;
            io.dispatch_instance[r] = best;
            st.events++;
        }
    }

    /* Phase 3: periodic rebalancing (Sec. 3.5). */
    void phase_migration_tick() {
        std::vector<bool> eligible(c.num_instances);
        int n_el = 0;
        for (int i = 0; i < c.num_instances; ++i) {
            eligible[i] = inst[i].mig_role == MIG_NONE;
            n_el += eligible[i];
        }
        while (n_el >= 2) {
            /* A draining instance has infinite virtual usage, so it is the least free
             * (lowest index among several) and passes the threshold against any other. */
            int s = -1;
            for (int i = 0; i < c.num_instances; ++i)
                if (eligible[i] && draining(i)) { s = i; break; }
            const bool drain_source = s >= 0;
            if (!drain_source)
                for (int i = 0; i < c.num_instances; ++i)
                    if (eligible[i] && (s < 0 || freer(s, i))) s = i;     /* least free, lowest index */
            int d = -1;
            for (int i = 0; i < c.num_instances; ++i)
                if (eligible[i] && i != s && !draining(i) && (d < 0 || freer(i, d))) d = i;  /* freest, lowest index */
            if (d < 0) break;  /* nothing but draining instances left to receive */
            if (!drain_source) {
                int64_t ns, ds, nd, dd;
                freeness(inst[s], ns, ds);
                freeness(inst[d], nd, dd);
                /* F_d - F_s >= theta_num / theta_den, exactly */
                if ((int64_t)c.theta_den * (nd * ds - ns * dd) < (int64_t)c.theta_num * dd * ds) break;
            }
            Inst &S = inst[s];
            Inst &D = inst[d];
            bool moved = false;
            int kq = -1;
            for (int k = c.num_tiers - 1; k >= 0; --k)
                if (!S.waiting[k].empty()) { kq = k; break; }
            if (kq >= 0) {
                /* queued candidate: newest request of the lowest-priority bucket, no KV to copy */
                int r = S.waiting[kq].back();
                S.waiting[kq].pop_back();
                D.waiting[kq].push_back(r);
                S.cnt[kq]--;
                D.cnt[kq]++;
                req[r].where = d;
                io.n_migrations[r]++;
                st.migrations++;
                st.events++;
                log_event(EV_QUEUED, r, s, d, 0);
                moved = true;
            } else if (!S.running.empty()) {
                /* running candidate: lowest priority, then fewest blocks, then newest */
                int best = -1;
                for (int r : S.running) {
                    if (best < 0) { best = r; continue; }
                    const Req &a = req[r], &b = req[best];
                    if (a.tier != b.tier ? a.tier > b.tier : (a.blocks != b.blocks ? a.blocks < b.blocks : r > best))
                        best = r;
                }
                if (D.free_blocks >= req[best].blocks) {
                    S.mig_role = MIG_SRC;
                    S.mig_peer = d;
                    S.mig_req = best;
                    S.mig_copied = 0;
                    D.mig_role = MIG_DST;
                    D.mig_peer = s;
                    st.migration_starts++;
                    log_event(EV_START, best, s, d, req[best].blocks);
                    moved = true;
                }
            }
            eligible[s] = false;
            --n_el;
            if (moved) { eligible[d] = false; --n_el; }
        }
    }

    /* Auto-scaling signal at a tick (Sec. 3.6).  The mean is kept as an exact
     * fraction p/q (q > 0, reduced): every F_normal has a denominator of at
     * most Bmax, so q divides lcm(1..Bmax) < 2^91 and 128-bit integers hold
     * every product below. */
    static __int128 gcd128(__int128 a, __int128 b) {
        if (a < 0) a = -a;
        while (b != 0) {
            __int128 t = a % b;
            a = b;
            b = t;
        }
        return a;
    }
    void phase_autoscale() {
        __int128 p = 0, q = 1;
        int64_t n = 0;
        for (int i = 0; i < c.num_instances; ++i) {
            if (draining(i)) continue;  /* an instance that is leaving does not count */
            int64_t num, den;
            normal_freeness(inst[i], num, den);
            p = p * den + (__int128)num * q;
            q = q * den;
            __int128 g = gcd128(p, q);
            p /= g;
            q /= g;
            ++n;
        }
        if (n == 0) return;
        /* mean = p / (q n) against threshold x / scale_den  <=>  p * scale_den against x * n * q */
        if (p * c.scale_den < (__int128)c.scale_out_num * n * q) {
            st.scale_out_signals++;
            log_event(EV_SCALE_OUT, -1, 255, 255, 0);
        } else if (p * c.scale_den > (__int128)c.scale_in_num * n * q) {
            st.scale_in_signals++;
            log_event(EV_SCALE_IN, -1, 255, 255, 0);
        }
    }

    /* Phase 4: batch formation at idle instances (Sec. 2.2 continuous batching). */
    bool phase_batch_formation() {
        for (int i = 0; i < c.num_instances; ++i) {
            Inst &in = inst[i];
            if (in.busy) continue;
            bool any_waiting = hol_request(in) >= 0;
            if (in.running.empty() && !any_waiting) continue;
            /* (i) grow the KV of running requests in running order; preempt when out of blocks */
            size_t idx = 0;
            while (idx < in.running.size()) {
                int r = in.running[idx];
                bool self_preempted = false;
                while (need_blocks(req[r]) > req[r].blocks) {
                    if (in.free_blocks > 0) {
                        in.free_blocks--;
                        req[r].blocks++;
                        continue;
                    }
                    int v = -1;  /* victim: lowest priority, then newest */
                    for (int x : in.running)
                        if (v < 0 || req[x].tier > req[v].tier || (req[x].tier == req[v].tier && x > v)) v = x;
                    size_t vpos = std::find(in.running.begin(), in.running.end(), v) - in.running.begin();
                    preempt(i, v);
                    if (v == r) { self_preempted = true; break; }
                    if (vpos < idx) --idx;
                }
                if (!self_preempted) ++idx;
            }
            /* (ii) admission in (tier, FCFS) order, stopping at the first misfit */
            int64_t n_decode = (int64_t)in.running.size();
            int64_t prefill_tokens = 0;
            while ((int)in.running.size() < c.max_batch) {
                int h = hol_request(in);
                if (h < 0) break;
                Req &q = req[h];
                if (c.check_invariants)
                    for (int k = 0; k < q.tier; ++k)
                        if (!in.waiting[k].empty()) return false;  /* tier isolation */
                int need = need_blocks(q);
                if (need > in.free_blocks) break;
                in.waiting[q.tier].pop_front();
                in.free_blocks -= need;
                q.blocks = need;
                q.state = RUNNING;
                in.running.push_back(h);
                prefill_tokens += q.P + q.g;
            }
            /* (iii) start the iteration */
            if (!in.running.empty()) {
                int64_t dur = c.iter_base_us + c.iter_us_per_prefill_token * prefill_tokens +
                              c.iter_us_per_decode_seq * n_decode;
                int64_t end = (int64_t)now + dur;
                if (end > 0xFFFFFFFEll) { st.status = ST_OVERFLOW; return true; }
                in.busy = true;
                in.busy_until = (uint32_t)end;
                in.batch_size = (int)in.running.size();
                st.iterations++;
                st.member_iterations += in.batch_size;
            }
        }
        return true;
    }

    bool check_invariants_now() const {
        int64_t placed = 0;
        for (int i = 0; i < c.num_instances; ++i) {
            const Inst &in = inst[i];
            int64_t held = 0;
            std::vector<int> recount(c.num_tiers, 0);
            for (int r : in.running) {
                const Req &q = req[r];
                if (q.state != RUNNING || q.where != i) return false;
                held += q.blocks;
                recount[q.tier]++;
            }
            for (int k = 0; k < c.num_tiers; ++k)
                for (int r : in.waiting[k]) {
                    const Req &q = req[r];
                    if (q.state != WAITING || q.where != i || q.tier != k || q.blocks != 0) return false;
                    recount[k]++;
                }
            for (int k = 0; k < c.num_tiers; ++k)
                if (recount[k] != in.cnt[k]) return false;
            placed += (int64_t)in.running.size();
            for (int k = 0; k < c.num_tiers; ++k) placed += (int64_t)in.waiting[k].size();
            /* KV block conservation */
            if (in.free_blocks < 0 || in.reserved_in < 0) return false;
            if (in.free_blocks + held + in.reserved_in != c.blocks_per_instance) return false;
            if ((int)in.running.size() > c.max_batch) return false;
            if (in.busy) {
                if (in.batch_size < 1 || in.batch_size > (int)in.running.size()) return false;
                for (int j = 0; j < in.batch_size; ++j)
                    if (req[in.running[j]].blocks < need_blocks(req[in.running[j]])) return false;
            }
            if (in.mig_role == MIG_SRC) {
                const Inst &d = inst[in.mig_peer];
                if (d.mig_role != MIG_DST || d.mig_peer != i) return false;
                if (std::find(in.running.begin(), in.running.end(), in.mig_req) == in.running.end()) return false;
                if (d.reserved_in != in.mig_copied) return false;
                if (in.mig_copied > req[in.mig_req].blocks) return false;
            } else if (in.mig_role == MIG_DST) {
                const Inst &s = inst[in.mig_peer];
                if (s.mig_role != MIG_SRC || s.mig_peer != i) return false;
            } else if (in.reserved_in != 0) {
                return false;
            }
        }
        if (placed + st.finished + (io.nreq - cursor) != io.nreq) return false;
        return true;
    }

    bool validate() const {
        if (c.num_instances < 1 || c.blocks_per_instance < 1 || c.tokens_per_block < 1 || c.max_batch < 1) return false;
        if (c.num_tiers < 1 || c.num_tiers > MAXK || c.migrate_blocks_per_iter < 1) return false;
        if (c.migrate_interval_us < 1 || c.theta_den < 1 || c.theta_num < 0) return false;
        if (c.iter_base_us < 0 || c.iter_us_per_prefill_token < 0 || c.iter_us_per_decode_seq < 0) return false;
        if (c.autoscale != 0 && c.autoscale != 1) return false;
        if (c.autoscale && (c.scale_den < 1 || c.scale_den > 64 || c.scale_out_num >= c.scale_in_num ||
                            c.scale_out_num < -4096 || c.scale_in_num > 4096 || c.max_batch > 64))
            return false;
        for (int k = 0; k < c.num_tiers; ++k)
            if (c.headroom[k] < 0) return false;
        if (c.n_headroom_changes < 0 || (c.n_headroom_changes > 0 && (!c.headroom_change_step || !c.headroom_change_table)))
            return false;
        for (int j = 0; j < c.n_headroom_changes; ++j) {
            if (c.headroom_change_step[j] < 0 || (j > 0 && c.headroom_change_step[j] < c.headroom_change_step[j - 1]))
                return false;
            for (int k = 0; k < c.num_tiers; ++k)
                if (c.headroom_change_table[j * MAXK + k] < 0) return false;
        }
        return true;
    }
    bool validate_trace() const {
        for (int64_t r = 0; r < io.nreq; ++r) {
            if (r > 0 && io.arrival_us[r] < io.arrival_us[r - 1]) return false;
            if (io.arrival_us[r] == NONE32) return false;
            if (io.tier[r] >= c.num_tiers || io.prompt_len[r] < 1 || io.output_len[r] < 1) return false;
            if ((int64_t)io.prompt_len[r] + io.output_len[r] > (int64_t)c.blocks_per_instance * c.tokens_per_block)
                return false;
        }
        return true;
    }

    void run(int64_t max_steps) {
        std::memset(&st, 0, sizeof st);
        if (!validate()) { st.status = ST_ARG; return; }
        if (!validate_trace()) { st.status = ST_TRACE; return; }
        req.assign(io.nreq, Req());
        for (int64_t r = 0; r < io.nreq; ++r) {
            req[r].arrival = io.arrival_us[r];
            req[r].P = io.prompt_len[r];
            req[r].O = io.output_len[r];
            req[r].tier = io.tier[r];
            io.dispatch_instance[r] = -1;
            io.final_instance[r] = -1;
            io.first_token_us[r] = NONE32;
            io.finish_us[r] = NONE32;
            io.n_migrations[r] = 0;
            io.n_preemptions[r] = 0;
        }
        inst.assign(c.num_instances, Inst());
        for (auto &in : inst) {
            in.free_blocks = c.blocks_per_instance;
            in.waiting.assign(c.num_tiers, std::deque<int>());
            in.cnt.assign(c.num_tiers, 0);
        }
        next_tick = c.migrate_interval_us;
        for (int k = 0; k < MAXK; ++k) H[k] = k < c.num_tiers ? c.headroom[k] : 0;
        st.status = ST_INCOMPLETE;
        while (st.finished < io.nreq) {
            if (st.steps >= max_steps) return;
            /* headroom changes due before this step (adaptive headroom) */
            while (next_change < c.n_headroom_changes && c.headroom_change_step[next_change] <= st.steps) {
                for (int k = 0; k < c.num_tiers; ++k) H[k] = c.headroom_change_table[next_change * MAXK + k];
                ++next_change;
            }
            const int64_t INF = INT64_MAX;
            int64_t t = cursor < io.nreq ? (int64_t)io.arrival_us[cursor] : INF;
            for (const Inst &in : inst)
                if (in.busy) t = std::min<int64_t>(t, in.busy_until);
            if (t == INF) { st.status = ST_DEADLOCK; return; }
            bool tick = false;
            if ((c.enable_migration || c.autoscale) && next_tick <= t) { t = next_tick; tick = true; }
            now = (uint32_t)t;
            st.steps++;
            st.last_time = now;
            phase_completions();
            phase_dispatch();
            if (tick) {
                next_tick += c.migrate_interval_us;
                if (c.autoscale) phase_autoscale();
                if (c.enable_migration) phase_migration_tick();
            }
            if (!phase_batch_formation()) { st.status = ST_INVARIANT; return; }
            if (st.status == ST_OVERFLOW) return;
            if (c.check_invariants && !check_invariants_now()) { st.status = ST_INVARIANT; return; }
        }
        st.status = ST_DONE;
    }
};

}  // namespace

extern "C" {

/* Simulates one replica from t = 0 for at most max_steps event times. */
int oracle_run_replica(const oracle_config_t *cfg, oracle_io_t *io, int64_t max_steps, oracle_stats_t *stats) {
    if (!cfg || !io || !stats) return ST_ARG;
    Sim sim(*cfg, *io, *stats);
    sim.run(max_steps);
    return stats->status;
}

/* Freeness of a hand-built instance state (for unit tests of Eq. 1-2, 4).
 * running_blocks[n_running]; cnt[num_tiers]; headroom taken from cfg. */
int oracle_freeness(const oracle_config_t *cfg, int32_t n_running, const int32_t *running_blocks,
                    int32_t hol_demand, const int32_t *cnt, int32_t reserved_in, int64_t *num, int64_t *den) {
    if (!cfg || !num || !den || n_running < 0) return ST_ARG;
    int64_t usage = 0;
    for (int j = 0; j < n_running; ++j) usage += running_blocks[j];
    usage += hol_demand;
    for (int k = 0; k < cfg->num_tiers; ++k)
        if (cnt[k] > 0) usage += cfg->headroom[k];
    usage += reserved_in;
    *num = (int64_t)cfg->blocks_per_instance - usage;
    *den = n_running > 0 ? n_running : 1;
    return 0;
}

/* Runs many independent replicas on `nthreads` host threads (one replica per
 * thread at a time; each replica is still the single-threaded simulation). */
int oracle_run_many(int32_t nrep, const oracle_config_t *cfgs /*[nrep]*/, oracle_io_t *ios /*[nrep]*/,
                    int64_t max_steps, oracle_stats_t *stats /*[nrep]*/, int32_t nthreads) {
    if (nrep < 0 || (nrep > 0 && (!cfgs || !ios || !stats))) return ST_ARG;
    if (nthreads < 1) nthreads = 1;
    std::atomic<int> next(0);
    auto work = [&]() {
        for (;;) {
            int r = next.fetch_add(1);
            if (r >= nrep) break;
            oracle_run_replica(&cfgs[r], &ios[r], max_steps, &stats[r]);
        }
    };
    std::vector<std::thread> th;
    for (int i = 1; i < nthreads; ++i) th.emplace_back(work);
    work();
    for (auto &t : th) t.join();
    return 0;
}

}  // extern "C"
