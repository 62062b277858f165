// mtsim.cu -- batched simulation of the multi-tier Llumnix-style scheduler
// ("Beyond Binary Priorities: Multi-Tier SLA Scheduling for LLM Serving",
// Sec. 3) for sm_103a, behind the C ABI declared in mtsim.h.
//
// Execution model
//   One warp simulates one replica.  A persistent grid pulls replicas from an
//   atomic work counter.  While a warp owns a replica, the replica's instance
//   state (per-instance scalars, per-(instance, tier) queue heads/tails and
//   request counts, headroom table) lives in shared memory, and so do the
//   running-request slots when they fit; everything is written back to HBM
//   when the warp stops (step limit or completion), so sim_run can be resumed.
//   Instances are spread over lanes in contiguous blocks of C = ceil(N/32) per
//   lane (C is a template parameter), so "lowest lane" order is "lowest
//   instance" order.  Per-request state stays in HBM: the read-only trace
//   (SoA), the 16-byte result record and a 16-byte queue node that threads a
//   waiting request into its (instance, tier) FCFS bucket.  A running request
//   is a 16-byte slot record that is written when it joins a batch and read
//   only on events; batch advance is lazy (see the slot record below), so an
//   iteration end and a batch formation without events cost O(1).
//   Between global events (arrivals, migration ticks) the instances that are
//   in no migration do not interact, so each lane advances its own instances
//   through a window in which each ends at most one iteration; migrations and
//   global events are stepped by the whole warp in the oracle's order.  The
//   next 32 arrivals are held in registers, one per lane.
//
// Exactness
//   Everything is integer.  Freeness F = (M - U) / max(B, 1) (Sec. 3.2 Eq. 1-2)
//   is kept per instance as an order-preserving 32-bit key
//   floor((M - U) * 4096 / max(B, 1)): for batch sizes up to 64, two distinct
//   fractions differ by at least 1/4032, so the floored keys order every pair
//   of freeness values exactly as the fractions do and equal fractions get
//   equal keys.  The floor division by B is the high half of the product
//   with a per-block table entry ceil(2^64 / B), exact for every 32-bit
//   numerator.  The
//   arg-max/arg-min of dispatch and migration pairing are therefore one warp
//   __reduce_{max,min}_sync plus a ballot (lowest index on ties).  The
//   migration threshold max F - min F >= theta is checked exactly by 64-bit
//   cross-multiplication.  Since free + sum(running blocks) + inbound
//   reservation = M on every instance, M - U reduces to
//   free - HoL demand - sum of present-tier headroom.
//
// Safety
//   No kernel waits on another warp, block or launch: there are no spin
//   loops.  Every loop is bounded by the trace length, the batch size, or the
//   per-call step limit.  Index checks on queue links and slot positions turn
//   an inconsistency into SIM_ERR_INTERNAL for that replica instead of an
//   out-of-bounds access.
#include "mtsim.h"
#include "latency.cuh"

#include <cuda_runtime.h>

#include <algorithm>
#include <climits>
#include <cstddef>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

namespace mt {

constexpr uint32_t kNone = 0xFFFFFFFFu;  // idle instance / no pending event / nil link
constexpr uint32_t kFull = 0xFFFFFFFFu;
constexpr int kKeyShift = 12;            // keys are floor(num * 4096 / den)
constexpr int kMaxKeyRange = 1 << 19;    // |num| < 2^19 keeps num * 4096 below 2^31
constexpr int kMagicShift = 40;          // floor(n / T) = (n * ceil(2^40 / T)) >> 40 for n < 2^20, T <= 65535
constexpr int kWarpsPerBlock = 2;
constexpr int kMaxBlockTokens = 64;      // T limit of the per-instance growth histogram
constexpr uint32_t kMagicBytes = 528;    // ceil(2^64 / d) for d = 0..64, rounded up to 16 bytes
constexpr uint32_t kHashSlots = 512;     // per-warp set of event times (C > 1 variants)

enum : int { MIG_NONE = 0, MIG_SRC = 1, MIG_DST = 2 };

// A running request is a 16-byte slot record, written when it joins an
// instance's running list and read only on events (finish, preemption,
// migration, first token):
//   x = request id (index in the replica's trace)
//   y = phi: number of the instance's first formation that includes it
//   z = c | left << 16: its context length P + g and its remaining output O - g at formation phi
//   w = tier | rho << 16, rho = (c - phi) mod T
// With nf formations done and pc = 1 after the iteration that followed the
// last one (0 before), the request has advanced adv = nf - phi + pc tokens
// (0 if phi > nf) and holds ceil((c + nf - phi) / T) KV blocks: every
// formation grows each surviving request to exactly its need, one block at a
// time because contexts grow by one token per iteration.  So the number of
// requests that need a new block at the next formation is the count of
// running requests with rho == -nf (mod T), and a request finishes at the
// iteration that follows formation phi + left - 1.

// A waiting request's queue node (16 bytes, indexed by request) carries what
// admitting it needs: x = next, y = info of next, z = prev, w = own info, with
// info = context (P + g) | remaining output (O - g) << 16.  The info of each
// bucket's head is also kept in shared memory, so admission and the HoL demand
// need no dependent HBM reads.

// An instance's scalars, one record per instance: every field sits at a
// fixed offset from the record, so the accesses to one instance share one
// address.  13 words: lanes reading one field of consecutive instances hit
// distinct shared-memory banks.
struct InstRec {
    uint32_t busy;                // end of the running iteration, or kNone when idle
    int free_, resv, hol, hr;     // free KV blocks; reserved for inbound copies; HoL demand; present headroom
    int key;                      // freeness key (dispatch, rebalancing)
    uint32_t mreq;                // request being copied out (migration source)
    int mcopied;                  // its blocks copied so far
    uint32_t nf, minfin, drain;   // formations done; next finishing formation; drain start
    uint16_t wmask;               // non-empty tier buckets
    uint8_t nrun, pc, phase;      // running requests; iteration-ended flag; nf mod T
    uint8_t mrole, mpeer, pad;    // migration role and peer
};
static_assert(sizeof(InstRec) == 52, "InstRec is 13 words");

// x.busy[i] and the like: field F of instance i's record.
template <typename T, int OFF>
struct Field {
    unsigned char *base;  // the replica's record array
    __device__ __forceinline__ T &operator[](int i) const {
        return *reinterpret_cast<T *>(base + i * (int)sizeof(InstRec) + OFF);
    }
};
#define MT_FIELD(T, f) Field<T, (int)offsetof(InstRec, f)> f

struct Layout {
    uint32_t inst;                                                       // [N] x InstRec
    uint32_t cnt;                                                        // [N*K] x 2 B
    uint32_t head, tail, hinfo;                                          // [N*K] x 4 B
    uint32_t h;                                                          // [K] x 4 B
    uint32_t hist;                                                       // [N*TH] x 1 B
    uint32_t mslot;                                                      // [N] x 16 B
    uint32_t bytes;
};

// Per-replica scalars persisted between sim_run calls.
struct RepState {
    uint32_t t, cursor, finished, log_events;
    uint32_t next_tick, pad0;
    uint64_t steps, iterations, member_iterations, events;
    uint32_t migrations, preemptions, starts, aborts;
    uint32_t scale_out, scale_in;
    int32_t status;
    uint32_t pad1;
};

struct Params {
    int R, N, M, T, TH, Bmax, K, S, cap, enable_mig, theta_num, theta_den;
    uint32_t interval, max_steps;
    unsigned long long magT;      // ceil(2^40 / T)
    int base, a, b;
    int ticks;                    // ticks happen (migration or the auto-scaling signal is on)
    int autoscale, scale_out_num, scale_in_num, scale_den;
    int drains;                   // a drain schedule is loaded
    unsigned long long lcm_lo, lcm_hi;  // lcm(1, ..., Bmax) as two 64-bit halves
    Layout L;
    uint32_t hash_bytes;          // per-warp event-time set (C > 1 variants), else 0
    const long long *offsets;
    const uint32_t *drain_src;    // [R][N] drain start times, or NULL
    const uint32_t *arrival;
    const uint16_t *plen, *olen;
    const uint8_t *tier;
    uint4 *node;                  // queue node per request: next, info of next, prev, own info
    sim_request_result_t *res;
    unsigned char *blobs;
    uint4 *slots;                 // [R][N][Bmax]
    RepState *rep;
    sim_migration_event_t *log;
    int *work;
    const int *order;             // [R] start order of the replicas, or NULL (trace order)
};

// Per-warp view of the replica being simulated: instance state in shared
// memory, request state in HBM, slot records in either; scalars are warp-uniform
// except t while lanes advance their own instances.
struct Ctx {
    MT_FIELD(uint32_t, busy);
    MT_FIELD(int, free_);
    MT_FIELD(int, resv);
    MT_FIELD(int, hol);
    MT_FIELD(int, hr);
    MT_FIELD(int, key);
    MT_FIELD(uint32_t, mreq);
    MT_FIELD(int, mcopied);
    MT_FIELD(uint32_t, nf);
    MT_FIELD(uint32_t, minfin);
    MT_FIELD(uint32_t, drain);
    MT_FIELD(uint16_t, wmask);
    MT_FIELD(uint8_t, nrun);
    MT_FIELD(uint8_t, pc);
    MT_FIELD(uint8_t, phase);
    MT_FIELD(uint8_t, mrole);
    MT_FIELD(uint8_t, mpeer);
    uint32_t *head, *tail, *hinfo;
    int *h;
    uint16_t *cnt;
    uint8_t *hist;
    uint4 *mslot;                     // record of the request a migration source is copying out
    uint4 *slots;
    uint32_t *tset;                   // event-time set (C > 1)
    const unsigned long long *magic;  // [65]: ceil(2^64 / d) for d >= 2
    const uint32_t *arrival;
    const uint16_t *plen, *olen;
    const uint8_t *tier;
    uint4 *node;
    sim_request_result_t *res;
    sim_migration_event_t *log;
    unsigned long long magT;
    int N, K, T, TH, Bmax, S, cap, lane, drains;
    uint32_t Q, t;
};

// Counters.  Lane 0's copy carries the replica's totals; the other lanes'
// copies collect what they add while advancing their own instances and are
// folded into lane 0's when the warp leaves the replica (`finished` after
// every window).
struct Cnt {
    uint32_t finished, log_events, migrations, preemptions, starts, aborts, steps, iterations;
    uint32_t scale_out, scale_in;  // lane 0 only
    uint64_t member_iterations, events;
    int status;
};

__device__ __forceinline__ int blocks_for(const Ctx &x, uint32_t tokens) {
    return (int)(((unsigned long long)(tokens + (uint32_t)x.T - 1u) * x.magT) >> kMagicShift);
}
__device__ __forceinline__ uint32_t mod_t(const Ctx &x, uint32_t v) {  // v mod T for v < 2^20
    const uint32_t q = (uint32_t)(((unsigned long long)v * x.magT) >> kMagicShift);
    const uint32_t r = v - q * (uint32_t)x.T;
    return r >= (uint32_t)x.T ? r - (uint32_t)x.T : r;
}

// floor(v / d) for v < 2^32 and 1 <= d <= 64: the high half of v * ceil(2^64 / d).
__device__ __forceinline__ uint32_t div_small(const Ctx &x, uint32_t v, int d) {
    return d == 1 ? v : (uint32_t)__umul64hi((unsigned long long)v, x.magic[d]);
}

__device__ __forceinline__ int make_key(const Ctx &x, int num, int nrun) {
    const int d = nrun > 0 ? nrun : 1;
    if (num >= 0) return (int)div_small(x, (uint32_t)num << kKeyShift, d);
    return -(int)div_small(x, ((uint32_t)(-num) << kKeyShift) + (uint32_t)(d - 1), d);
}

__device__ __forceinline__ int fnum(const Ctx &x, int i) { return x.free_[i] - x.hol[i] - x.hr[i]; }

__device__ __forceinline__ void set_key(const Ctx &x, int i) { x.key[i] = make_key(x, fnum(x, i), x.nrun[i]); }

template <int C>
__device__ __forceinline__ void refresh_keys(const Ctx &x) {
#pragma unroll
    for (int j = 0; j < C; ++j) {
        const int i = x.lane * C + j;
        if (i < x.N) set_key(x, i);
    }
    __syncwarp();
}

template <int C>
__device__ __forceinline__ uint32_t own_mask(const Ctx &x) {
    uint32_t m = 0;
#pragma unroll
    for (int j = 0; j < C; ++j)
        if (x.lane * C + j < x.N) m |= 1u << j;
    return m;
}

// Arg-max (want_max) or arg-min of the freeness key over the instances whose
// bit is set in `el` (bit j = instance lane*C + j), excluding `excl`; lowest
// index on ties; -1 if none.  Collective.
template <int C>
__device__ __forceinline__ int arg_ext(const Ctx &x, uint32_t el, bool want_max, int excl) {
    int bv = want_max ? INT_MIN : INT_MAX, bi = -1;
#pragma unroll
    for (int j = 0; j < C; ++j) {
        const int i = x.lane * C + j;
        if (((el >> j) & 1u) && i != excl) {
            const int k = x.key[i];
            if (bi < 0 || (want_max ? k > bv : k < bv)) { bv = k; bi = i; }
        }
    }
    const int m = want_max ? __reduce_max_sync(kFull, bv) : __reduce_min_sync(kFull, bv);
    // lowest instance among those at the extreme (INT_MAX: none)
    const int best = __reduce_min_sync(kFull, (bi >= 0 && bv == m) ? bi : INT_MAX);
    return best == INT_MAX ? -1 : best;
}

// ---- single-thread instance logic (no collectives inside) -------------------
__device__ __forceinline__ void cnt_inc(const Ctx &x, int i, int k) {
    if (x.cnt[i * x.K + k]++ == 0) x.hr[i] += x.h[k];
}
__device__ __forceinline__ void cnt_dec(const Ctx &x, int i, int k) {
    if (--x.cnt[i * x.K + k] == 0) x.hr[i] -= x.h[k];
}
__device__ __forceinline__ void push_back(const Ctx &x, int i, int k, uint32_t r, uint32_t info) {
    const int b = i * x.K + k;
    const uint32_t tl = x.tail[b];
    x.node[r] = make_uint4(kNone, 0u, tl, info);
    if (tl != kNone) *reinterpret_cast<uint2 *>(&x.node[tl]) = make_uint2(r, info);
    else { x.head[b] = r; x.hinfo[b] = info; }
    x.tail[b] = r;
    x.wmask[i] |= (uint16_t)(1u << k);
}
__device__ __forceinline__ void push_front(const Ctx &x, int i, int k, uint32_t r, uint32_t info) {
    const int b = i * x.K + k;
    const uint32_t hd = x.head[b];
    x.node[r] = make_uint4(hd, hd != kNone ? x.hinfo[b] : 0u, kNone, info);
    if (hd != kNone) x.node[hd].z = r; else x.tail[b] = r;
    x.head[b] = r;
    x.hinfo[b] = info;
    x.wmask[i] |= (uint16_t)(1u << k);
}
// Removes the tail of bucket (i, k) and returns its info in `info`.
__device__ __forceinline__ uint32_t pop_back(const Ctx &x, int i, int k, uint32_t &info, int &status) {
    const int b = i * x.K + k;
    const uint32_t r = x.tail[b];
    if (r >= x.Q) { status = SIM_ERR_INTERNAL; return kNone; }
    const uint4 nd = x.node[r];
    info = nd.w;
    x.tail[b] = nd.z;
    if (nd.z != kNone) *reinterpret_cast<uint2 *>(&x.node[nd.z]) = make_uint2(kNone, 0u);
    else { x.head[b] = kNone; x.wmask[i] &= (uint16_t)~(1u << k); }
    return r;
}
// HoL demand: KV blocks the head of the highest-priority non-empty bucket needs.
__device__ __forceinline__ void refresh_hol(const Ctx &x, int i) {
    const uint32_t wm = x.wmask[i];
    x.hol[i] = wm ? blocks_for(x, x.hinfo[i * x.K + (__ffs(wm) - 1)] & 0xFFFFu) : 0;
}
__device__ __forceinline__ void log_ev(const Ctx &x, Cnt &cn, int kind, uint32_t r, int s, int d, int blocks) {
    const uint32_t k = cn.log_events++;
    if (k < (uint32_t)x.cap) {
        uint4 w;
        w.x = x.t;
        w.y = r;
        w.z = (uint32_t)(blocks & 0xFFFF) | ((uint32_t)s << 16) | ((uint32_t)d << 24);
        w.w = (uint32_t)kind;
        reinterpret_cast<uint4 *>(x.log)[k] = w;
    }
}
// The result record's last word holds n_preemptions (low half) and
// n_migrations (high half), both modulo 2^16.  A migration adds 1 << 16: a
// wrap carries out of the word, so nothing waits on the add.  A preemption
// adds 1 to the low half and gets the old word back; when the low half
// wrapped, the carry into n_migrations is taken back (pre_fix).
__device__ __forceinline__ unsigned int *count_word(const Ctx &x, uint32_t r) {
    return reinterpret_cast<unsigned int *>(reinterpret_cast<unsigned char *>(x.res + r) + 12);
}
__device__ __forceinline__ void bump_mig(const Ctx &x, uint32_t r) { atomicAdd(count_word(x, r), 1u << 16); }
__device__ __forceinline__ unsigned int bump_pre(const Ctx &x, uint32_t r) { return atomicAdd(count_word(x, r), 1u); }
__device__ __forceinline__ void pre_fix(const Ctx &x, uint32_t r, unsigned int old) {
    if ((old & 0xFFFFu) == 0xFFFFu) atomicSub(count_word(x, r), 1u << 16);
}
__device__ __forceinline__ void clear_mig(const Ctx &x, int s, int d) {
    x.mrole[s] = MIG_NONE;
    x.mrole[d] = MIG_NONE;
    x.mreq[s] = kNone;
    x.mcopied[s] = 0;
}
// Abandon the staged copy out of source s: the destination releases what was copied.
__device__ __forceinline__ void abort_mig(const Ctx &x, Cnt &cn, int s) {
    const int d = x.mpeer[s];
    const int cp = x.mcopied[s];
    x.free_[d] += cp;
    x.resv[d] -= cp;
    log_ev(x, cn, SIM_EV_ABORT, x.mreq[s], s, d, cp);
    cn.aborts++;
    clear_mig(x, s, d);
}

// Derived quantities of a slot record on instance i.
__device__ __forceinline__ uint32_t sl_c(const uint4 &sl) { return sl.z & 0xFFFFu; }
__device__ __forceinline__ uint32_t sl_left(const uint4 &sl) { return sl.z >> 16; }
__device__ __forceinline__ uint32_t sl_tier(const uint4 &sl) { return sl.w & 0xFFu; }
__device__ __forceinline__ uint32_t sl_rho(const uint4 &sl) { return sl.w >> 16; }
__device__ __forceinline__ uint32_t sl_fin(const uint4 &sl) { return sl.y + sl_left(sl) - 1u; }
__device__ __forceinline__ uint32_t sl_adv(const Ctx &x, int i, const uint4 &sl) {
    const uint32_t nf = x.nf[i];
    return sl.y <= nf ? nf - sl.y + x.pc[i] : 0u;
}
__device__ __forceinline__ int sl_blocks(const Ctx &x, int i, const uint4 &sl) {
    return blocks_for(x, sl_c(sl) + x.nf[i] - sl.y);
}
__device__ __forceinline__ uint4 *slot_ptr(const Ctx &x, int i, int s) { return x.slots + i * x.Bmax + s; }

// A request joins instance i's running list at position n with context c and
// remaining output left; its first formation there will be number nf + 1.
__device__ __forceinline__ void slot_join_at(const Ctx &x, int i, int n, uint32_t r, uint32_t c, uint32_t left,
                                             uint32_t tier, uint32_t nf, uint32_t ph) {
    const uint32_t phi = nf + 1u;
    const uint32_t pm = ph + 1u == (uint32_t)x.T ? 0u : ph + 1u;  // phi mod T
    const uint32_t cm = mod_t(x, c);
    const uint32_t rho = cm >= pm ? cm - pm : cm + (uint32_t)x.T - pm;
    *slot_ptr(x, i, n) = make_uint4(r, phi, c | (left << 16), tier | (rho << 16));
    x.hist[i * x.TH + rho]++;
    x.minfin[i] = min(x.minfin[i], phi + left - 1u);
}
__device__ __forceinline__ void slot_join(const Ctx &x, int i, int n, uint32_t r, uint32_t c, uint32_t left,
                                          uint32_t tier) {
    slot_join_at(x, i, n, r, c, left, tier, x.nf[i], x.phase[i]);
}

// Lane 0's part of committing a fully copied running request `sl` of source s
// to its destination (Sec. 3.5, Fig. 4).  The warp has already taken the
// slot out of s's running list (order kept); fm is the new minimum finishing
// formation of what is left there.
__device__ __forceinline__ void commit_book(const Ctx &x, Cnt &cn, int s, const uint4 &sl, uint32_t fm) {
    const int d = x.mpeer[s];
    const int blocks = sl_blocks(x, s, sl);
    const uint32_t adv = sl_adv(x, s, sl);
    x.nrun[s] = (uint8_t)(x.nrun[s] - 1);
    x.hist[s * x.TH + sl_rho(sl)]--;
    x.minfin[s] = fm;
    x.free_[s] += blocks;
    x.resv[d] -= x.mcopied[s];
    const uint32_t tr = sl_tier(sl);
    cnt_dec(x, s, (int)tr);
    cnt_inc(x, d, (int)tr);
    const int nd = x.nrun[d];
    slot_join(x, d, nd, sl.x, sl_c(sl) + adv, sl_left(sl) - adv, tr);
    x.nrun[d] = (uint8_t)(nd + 1);
    bump_mig(x, sl.x);
    cn.migrations++;
    cn.events++;
    log_ev(x, cn, SIM_EV_COMMIT, sl.x, s, d, blocks);
    clear_mig(x, s, d);
}

// Phase 1, first part, single thread: the iteration of instance i ends at
// x.t (Sec. 2.1 token accounting; first tokens were recorded when the
// prefill iteration was scheduled).  Returns whether some running request
// finishes now (then coop_finish must run before anything else touches i).
__device__ __forceinline__ bool inst_complete_head(const Ctx &x, int i) {
    x.busy[i] = kNone;
    x.pc[i] = 1;
    return x.minfin[i] == x.nf[i];
}

// Phase 1, second part, whole warp: the requests of instance i whose output
// is complete finish at x.t and free their KV (an in-flight migration of one
// of them is abandoned).  Lane l looks at slots l and 32 + l.
__device__ __forceinline__ void coop_finish(const Ctx &x, Cnt &cn, int i) {
    const int n = x.nrun[i];
    const uint32_t nf = x.nf[i];
    uint4 *p = slot_ptr(x, i, 0);
    const int q0 = x.lane, q1 = x.lane + 32;
    const bool v0 = q0 < n, v1 = q1 < n;
    const uint4 a0 = v0 ? p[q0] : make_uint4(0, 0, 0, 0);
    const uint4 a1 = v1 ? p[q1] : make_uint4(0, 0, 0, 0);
    const bool f0 = v0 && sl_fin(a0) == nf, f1 = v1 && sl_fin(a1) == nf;
    if (f0) { x.res[a0.x].finish_us = x.t; x.res[a0.x].final_instance = (uint16_t)i; }
    if (f1) { x.res[a1.x].finish_us = x.t; x.res[a1.x].final_instance = (uint16_t)i; }
    const int freed = __reduce_add_sync(kFull, (f0 ? sl_blocks(x, i, a0) : 0) + (f1 ? sl_blocks(x, i, a1) : 0));
    const uint32_t m0 = __ballot_sync(kFull, f0), m1 = __ballot_sync(kFull, f1);
#pragma unroll
    for (int j = 0; j < 2; ++j) {
        uint32_t lanes = j ? m1 : m0;
        while (lanes) {
            const int l = __ffs(lanes) - 1;
            lanes &= lanes - 1;
            const uint32_t rid = __shfl_sync(kFull, j ? a1.x : a0.x, l);
            const uint32_t w = __shfl_sync(kFull, j ? a1.w : a0.w, l);
            if (x.lane == 0) {
                cnt_dec(x, i, (int)(w & 0xFFu));
                x.hist[i * x.TH + (w >> 16)]--;
                if (x.mrole[i] == MIG_SRC && x.mreq[i] == rid) abort_mig(x, cn, i);
            }
        }
    }
    const bool k0 = v0 && !f0, k1 = v1 && !f1;
    const uint32_t e0 = __ballot_sync(kFull, k0), e1 = __ballot_sync(kFull, k1);
    const uint32_t below = (1u << x.lane) - 1u;
    const int p0 = __popc(e0 & below), p1 = __popc(e0) + __popc(e1 & below);
    const uint32_t fm = __reduce_min_sync(kFull, min(k0 ? sl_fin(a0) : kNone, k1 ? sl_fin(a1) : kNone));
    __syncwarp();
    if (k0 && p0 != q0) p[p0] = a0;  // only the records that move are written
    if (k1 && p1 != q1) p[p1] = a1;
    if (x.lane == 0) {
        const uint32_t nfin = __popc(m0) + __popc(m1);
        x.free_[i] += freed;
        x.nrun[i] = (uint8_t)(__popc(e0) + __popc(e1));
        x.minfin[i] = fm;
        cn.finished += nfin;
        cn.events += nfin;
    }
    __syncwarp();
}

// One copy stage at the end of an iteration of migration source s, whole
// warp: up to S of the request's blocks are reserved on the destination
// (abandoning the migration if they do not fit), and the request commits
// there once all of them are copied (Sec. 3.5, Fig. 4).
__device__ __forceinline__ void coop_stage(const Ctx &x, Cnt &cn, int s) {
    int commit = 0;
    if (x.lane == 0) {
        const int d = x.mpeer[s];
        const int blocks = sl_blocks(x, s, x.mslot[s]);
        const int cp = x.mcopied[s];
        const int cc = min(x.S, blocks - cp);
        if (x.free_[d] < cc) {
            abort_mig(x, cn, s);
        } else {
            x.free_[d] -= cc;
            x.resv[d] += cc;
            x.mcopied[s] = cp + cc;
            commit = (cp + cc == blocks) && ((int)x.nrun[d] < x.Bmax);
        }
    }
    commit = __shfl_sync(kFull, commit, 0);
    __syncwarp();
    if (commit) {
        // the whole warp finds the request's slot (lane l holds slots l and
        // 32 + l), closes the gap and takes the survivors' minimum; lane 0 books
        const uint32_t rid = x.mreq[s];
        const int n = x.nrun[s];
        uint4 *p = slot_ptr(x, s, 0);
        const int q0 = x.lane, q1 = x.lane + 32;
        const bool v0 = q0 < n, v1 = q1 < n;
        const uint4 a0 = v0 ? p[q0] : make_uint4(0, 0, 0, 0);
        const uint4 a1 = v1 ? p[q1] : make_uint4(0, 0, 0, 0);
        const uint32_t h0 = __ballot_sync(kFull, v0 && a0.x == rid);
        const uint32_t h1 = __ballot_sync(kFull, v1 && a1.x == rid);
        const int pos = h0 ? __ffs(h0) - 1 : (h1 ? 32 + __ffs(h1) - 1 : -1);
        if (pos < 0) {
            if (x.lane == 0) cn.status = SIM_ERR_INTERNAL;
        } else {
            const uint4 sl = p[pos];
            const uint32_t fm = __reduce_min_sync(
                kFull, min(v0 && q0 != pos ? sl_fin(a0) : kNone, v1 && q1 != pos ? sl_fin(a1) : kNone));
            __syncwarp();
            if (v0 && q0 > pos) p[q0 - 1] = a0;
            if (v1 && q1 > pos) p[q1 - 1] = a1;
            __syncwarp();
            if (x.lane == 0) commit_book(x, cn, s, sl, fm);
        }
        __syncwarp();
    }
}

// Recompute-style preemption of running request `sl` (holding `blocks` KV
// blocks) on instance i: its KV is freed, it keeps its generated tokens and
// goes back to the front of its tier's bucket.  The caller drops its slot.
__device__ __forceinline__ unsigned int preempt_book(const Ctx &x, Cnt &cn, int i, const uint4 &sl, int blocks) {
    const uint32_t r = sl.x;
    const int tr = (int)sl_tier(sl);
    const uint32_t adv = sl_adv(x, i, sl);
    x.free_[i] += blocks;
    const uint32_t old = x.wmask[i];
    push_front(x, i, tr, r, (sl_c(sl) + adv) | ((sl_left(sl) - adv) << 16));
    if ((old & ((1u << tr) - 1u)) == 0) x.hol[i] = blocks_for(x, sl_c(sl) + adv);  // now head of line
    x.hist[i * x.TH + sl_rho(sl)]--;
    const unsigned int word = bump_pre(x, r);
    cn.preemptions++;
    cn.events++;
    if (x.mrole[i] == MIG_SRC && x.mreq[i] == r) abort_mig(x, cn, i);
    return word;  // for pre_fix, which the caller runs later so that nothing waits here
}

// Phase 4: batch formation at idle instance i at x.t (Sec. 2.2, Sec. 3.1):
// (i) KV growth of the running requests, preempting the lowest-priority newest
// one when out of blocks; (ii) admission in (tier, FCFS) order while the head
// of line fits; (iii) the iteration starts.
__device__ __forceinline__ void inst_form(const Ctx &x, Cnt &cn, int i, int base, int a_us, int b_us) {
    // the instance's scalars, read together up front (the code below would
    // otherwise reload them after every shared-memory store)
    int n = x.nrun[i];
    int fr = x.free_[i];
    const uint32_t ph = x.phase[i];
    const uint32_t nf = x.nf[i];
    uint32_t wm = x.wmask[i];
    int need = x.hol[i];
    if (n > 0) {
        const int deficit = x.hist[i * x.TH + (ph == 0 ? 0u : (uint32_t)x.T - ph)];
        if (deficit <= fr) {
            fr -= deficit;  // every request that needs a block gets it
        } else {
            x.free_[i] = fr;
            // In running order, a request that needs a block (at most one)
            // takes a free one or preempts the lowest-priority newest running
            // request, possibly itself.  Positions are the list's before this
            // step; removals are applied afterwards.
            uint4 *p = slot_ptr(x, i, 0);
            const uint64_t all = n >= 64 ? ~0ull : ((1ull << n) - 1ull);
            uint64_t alive = all, needs = 0, granted = 0;
            // The requests that need a block now are those whose context reaches
            // a block boundary: rho == -nf (mod T), the ones hist counts.
            const uint32_t target = ph == 0 ? 0u : (uint32_t)x.T - ph;
            // the same pass finds the first victim (lowest priority, then newest):
            // more requests need a block than there are free blocks, so there is one
            int v1 = -1;
            uint32_t vt1 = 0, vr1 = 0;
#pragma unroll 4
            for (int q = 0; q < n; ++q) {
                const uint4 sl = p[q];
                needs |= (uint64_t)(sl_rho(sl) == target) << q;
                const uint32_t ts = sl_tier(sl);
                if (v1 < 0 || ts > vt1 || (ts == vt1 && sl.x > vr1)) { v1 = q; vt1 = ts; vr1 = sl.x; }
            }
            int fb = fr;
            uint32_t pr = kNone;  // the last preempted request and its counter word before the add
            unsigned int pold = 0;
            for (int q = 0; q < n; ++q) {
                if (!((alive & needs) >> q & 1ull)) continue;
                for (;;) {
                    if (fb > 0) { --fb; granted |= 1ull << q; break; }
                    int v = -1;
                    if (alive == all) {
                        v = v1;  // nobody preempted yet: the victim found by the scan
                    } else {
                        uint32_t vt = 0, vr = 0;
                        for (uint64_t m = alive; m; m &= m - 1) {
                            const int s2 = __ffsll((long long)m) - 1;
                            const uint32_t ts = sl_tier(p[s2]), rs = p[s2].x;
                            if (v < 0 || ts > vt || (ts == vt && rs > vr)) { v = s2; vt = ts; vr = rs; }
                        }
                    }
                    const int vb = blocks_for(x, sl_c(p[v]) + nf - p[v].y) + (int)((granted >> v) & 1ull);
                    alive &= ~(1ull << v);
                    x.free_[i] = fb;
                    if (pr != kNone) pre_fix(x, pr, pold);
                    pr = p[v].x;
                    pold = preempt_book(x, cn, i, p[v], vb);
                    fb = x.free_[i];
                    if (v == q) break;
                }
            }
            x.free_[i] = fb;
            int w = 0;
            uint32_t fm = kNone;  // the survivors' next finishing formation
            for (int q = 0; q < n; ++q) {
                if ((alive >> q) & 1ull) {
                    const uint4 sl = p[q];
                    if (w != q) p[w] = sl;
                    ++w;
                    fm = min(fm, sl_fin(sl));
                }
            }
            x.nrun[i] = (uint8_t)w;
            x.minfin[i] = fm;
            if (pr != kNone) pre_fix(x, pr, pold);
            n = w;  // preemptions changed the free blocks, queues and head of line
            fr = x.free_[i];
            wm = x.wmask[i];
            need = x.hol[i];
        }
    }
    // (ii) admission; the waiting mask and the HoL demand follow in registers
    const int n_decode = n;
    int prefill = 0;
    while (n < x.Bmax) {
        if (!wm) break;
        if (need > fr) break;
        const int k = __ffs(wm) - 1;
        const int b = i * x.K + k;
        const uint32_t info = x.hinfo[b];
        const uint32_t r = x.head[b];
        if (r >= x.Q) { cn.status = SIM_ERR_INTERNAL; break; }
        const uint4 nd = x.node[r];  // the head leaves its bucket; nd.x is the new head
        x.head[b] = nd.x;
        const uint32_t c = info & 0xFFFFu;
        slot_join_at(x, i, n, r, c, info >> 16, (uint32_t)k, nf, ph);
        ++n;
        fr -= need;
        prefill += (int)c;
        uint32_t hinfo;  // info of the new head of line
        if (nd.x != kNone) {
            x.node[nd.x].z = kNone;
            x.hinfo[b] = nd.y;
            hinfo = nd.y;
        } else {
            x.tail[b] = kNone;
            wm &= ~(1u << k);
            x.wmask[i] = (uint16_t)wm;
            hinfo = wm ? x.hinfo[i * x.K + (__ffs(wm) - 1)] : 0u;
        }
        need = wm ? blocks_for(x, hinfo & 0xFFFFu) : 0;
        x.hol[i] = need;
    }
    x.nrun[i] = (uint8_t)n;
    x.free_[i] = fr;
    // (iii) the iteration starts
    if (n > 0) {
        const long long end = (long long)x.t + base + (long long)a_us * prefill + (long long)b_us * n_decode;
        if (end > 0xFFFFFFFELL) {
            cn.status = SIM_ERR_OVERFLOW;
            return;
        }
        x.busy[i] = (uint32_t)end;
        const uint4 *sp = slot_ptr(x, i, 0);
        for (int q = n_decode; q < n; ++q) atomicMin(&x.res[sp[q].x].first_token_us, (uint32_t)end);
        x.nf[i] = nf + 1u;
        x.phase[i] = ph + 1u == (uint32_t)x.T ? (uint8_t)0 : (uint8_t)(ph + 1u);
        x.pc[i] = 0;
        cn.iterations++;
        cn.member_iterations += (uint64_t)n;
    }
}

// ---- cooperative steps ----------------------------------------------------------
// Lane 0 appends arriving request r (tier k, prompt P, output O) to instance
// best's bucket and updates the instance (Sec. 3.4); the key store is needed
// only if another arrival at the same time is dispatched next.
__device__ __forceinline__ void dispatch_to(const Ctx &x, Cnt &cn, int best, uint32_t r, int k, uint32_t P,
                                            uint32_t O, bool store_key) {
    if (x.lane == 0) {
        // the destination's scalars, read together; the new key is computed from them
        const int b = best * x.K + k;
        const uint32_t old = x.wmask[best];
        const uint32_t tl = x.tail[b];
        const uint32_t c0 = x.cnt[b];
        int hol = x.hol[best];
        int hr = x.hr[best];
        const int fr = x.free_[best];
        const int nr = x.nrun[best];
        const int hk = x.h[k];
        const uint32_t info = P | (O << 16);
        x.node[r] = make_uint4(kNone, 0u, tl, info);  // appended to bucket (best, k), as push_back
        if (tl != kNone) *reinterpret_cast<uint2 *>(&x.node[tl]) = make_uint2(r, info);
        else { x.head[b] = r; x.hinfo[b] = info; }
        x.tail[b] = r;
        x.wmask[best] = (uint16_t)(old | (1u << k));
        x.cnt[b] = (uint16_t)(c0 + 1u);
        if (c0 == 0) x.hr[best] = hr += hk;                    // tier k now present (Eq. 4)
        if ((old & ((2u << k) - 1u)) == 0) x.hol[best] = hol = blocks_for(x, P);  // becomes head of line
        x.res[r].dispatch_instance = (uint16_t)best;
        cn.events++;
        if (store_key) x.key[best] = make_key(x, fr - hol - hr, nr);
    }
}

// Dispatch one arriving request r of tier k with prompt length P (Sec. 3.4).
template <int C>
__device__ __forceinline__ void dispatch_one(const Ctx &x, Cnt &cn, uint32_t r, int k, uint32_t P, uint32_t O,
                                             uint32_t all) {
    const int best = arg_ext<C>(x, all, true, -1);
    dispatch_to(x, cn, best, r, k, P, O, true);
    __syncwarp();
}

// The next 32 trace records, one per lane: index pb + lane.
struct ArrBuf {
    uint32_t pb, time, tier, P, O;
};

__device__ __forceinline__ void arr_refill(const Ctx &x, ArrBuf &ab, uint32_t cursor) {
    ab.pb = cursor;
    const uint32_t idx = cursor + (uint32_t)x.lane;
    const bool in = idx < x.Q;
    ab.time = in ? x.arrival[idx] : kNone;
    ab.tier = in ? (uint32_t)x.tier[idx] : 0u;
    ab.P = in ? (uint32_t)x.plen[idx] : 0u;
    ab.O = in ? (uint32_t)x.olen[idx] : 0u;
}

// Phase 2: arrivals at t, tier 0 first, FCFS (trace order) within a tier.
// EXT: draining instances may exist.
template <int C, bool EXT>
__device__ __forceinline__ void dispatch_phase(const Ctx &x, Cnt &cn, uint32_t &cursor, uint32_t &next_arr,
                                               ArrBuf &ab) {
    uint32_t all = own_mask<C>(x);
    if (EXT && x.drains) {
        // Draining instances (infinite virtual usage, Sec. 3.5) get no
        // dispatch unless every instance drains; then the freest of them
        // does (Sec. 3.4: the least loaded draining one).
        uint32_t live = 0;
#pragma unroll
        for (int j = 0; j < C; ++j)
            if (((all >> j) & 1u) && x.drain[x.lane * C + j] > x.t) live |= 1u << j;
        if (__any_sync(kFull, live != 0)) all = live;
    }
    const uint32_t off = cursor - ab.pb;
    uint32_t eq = __ballot_sync(kFull, (uint32_t)x.lane >= off && ab.time == x.t);
    if ((eq >> 31) && off > 0) {
        // the run of arrivals at t may continue past the buffer: realign it on the cursor
        arr_refill(x, ab, cursor);
        eq = __ballot_sync(kFull, ab.time == x.t);
    }
    if (eq != kFull && (eq & (eq - 1u)) == 0u) {
        // one arrival at t (the usual case): no tier ordering to do
        const int l = __ffs(eq) - 1;
        const uint32_t k1 = __shfl_sync(kFull, ab.tier, l);
        const uint32_t po = __shfl_sync(kFull, ab.P | (ab.O << 16), l);
        // the freest instance from keys computed in registers (nothing reads
        // the key array before the next refresh)
        int bv = INT_MIN, bi = -1;
#pragma unroll
        for (int j = 0; j < C; ++j) {
            const int i = x.lane * C + j;
            if ((all >> j) & 1u) {
                const int kk = make_key(x, fnum(x, i), x.nrun[i]);
                if (bi < 0 || kk > bv) { bv = kk; bi = i; }
            }
        }
        const int m = __reduce_max_sync(kFull, bv);
        const int best = __reduce_min_sync(kFull, (bi >= 0 && bv == m) ? bi : INT_MAX);
        dispatch_to(x, cn, best, ab.pb + (uint32_t)l, (int)k1, po & 0xFFFFu, po >> 16, false);
        __syncwarp();
        cursor += 1u;
    } else if (eq != kFull) {
        refresh_keys<C>(x);
        const bool mine = (eq >> x.lane) & 1u;
        uint32_t tm = __reduce_or_sync(kFull, mine ? (1u << ab.tier) : 0u);
        while (tm) {
            const int k = __ffs(tm) - 1;
            tm &= tm - 1;
            uint32_t bits = __ballot_sync(kFull, mine && ab.tier == (uint32_t)k);
            while (bits) {
                const int l = __ffs(bits) - 1;
                bits &= bits - 1;
                dispatch_one<C>(x, cn, ab.pb + (uint32_t)l, k, __shfl_sync(kFull, ab.P, l),
                                __shfl_sync(kFull, ab.O, l), all);
            }
        }
        cursor += (uint32_t)__popc(eq);
    } else {
        // 32 or more arrivals share this time (the buffer starts at the cursor):
        // count them, then go tier by tier from the trace.
        refresh_keys<C>(x);
        uint32_t m = 32;
        for (;;) {
            const uint32_t j2 = cursor + m + (uint32_t)x.lane;
            const bool in2 = j2 < x.Q;
            const uint32_t e2 = __ballot_sync(kFull, in2 && x.arrival[j2] == x.t);
            m += (uint32_t)__popc(e2);
            if (e2 != kFull) break;
        }
        for (int k = 0; k < x.K; ++k) {
            for (uint32_t base = 0; base < m; base += 32) {
                const uint32_t j2 = cursor + base + (uint32_t)x.lane;
                const bool mine = base + (uint32_t)x.lane < m;
                const uint32_t tr = mine ? x.tier[j2] : 0u;
                const uint32_t P = mine ? x.plen[j2] : 0u;
                const uint32_t O = mine ? x.olen[j2] : 0u;
                uint32_t bits = __ballot_sync(kFull, mine && tr == (uint32_t)k);
                while (bits) {
                    const int l = __ffs(bits) - 1;
                    bits &= bits - 1;
                    dispatch_one<C>(x, cn, cursor + base + (uint32_t)l, k, __shfl_sync(kFull, P, l),
                                    __shfl_sync(kFull, O, l), all);
                }
            }
        }
        cursor += m;
    }
    if (cursor - ab.pb >= 32u) arr_refill(x, ab, cursor);
    next_arr = __shfl_sync(kFull, ab.time, (int)(cursor - ab.pb));
}

// Auto-scaling signal at a tick (Sec. 3.6): the mean normal-priority freeness
// (Eq. 1 without the headroom term, Sec. 3.4) over the instances that are not
// draining, compared exactly with scale_out_num / scale_den and
// scale_in_num / scale_den.  Each F_normal = (free - HoL) / max(B, 1) is scaled
// by L = lcm(1, ..., Bmax), so S = L * sum F_normal is an exact 128-bit
// integer (|S| < 2^117), and mean < x / D  <=>  S * D < x * n * L.  Collective.
template <int C>
__device__ __forceinline__ void autoscale_tick(const Ctx &x, Cnt &cn, const Params &p) {
    const __int128 L = (__int128)(((unsigned __int128)p.lcm_hi << 64) | p.lcm_lo);
    __int128 sum = 0;
    int n = 0;
#pragma unroll
    for (int j = 0; j < C; ++j) {
        const int i = x.lane * C + j;
        if (i < x.N && !(x.drains && x.drain[i] <= x.t)) {
            const int num = x.free_[i] - x.hol[i];
            const int den = max((int)x.nrun[i], 1);
            sum += (__int128)num * (L / den);
            ++n;
        }
    }
#pragma unroll
    for (int sh = 16; sh > 0; sh >>= 1) {
        const unsigned long long lo = __shfl_xor_sync(kFull, (unsigned long long)sum, sh);
        const unsigned long long hi = __shfl_xor_sync(kFull, (unsigned long long)((unsigned __int128)sum >> 64), sh);
        sum += (__int128)(((unsigned __int128)hi << 64) | lo);
    }
    n = __reduce_add_sync(kFull, n);
    if (x.lane == 0 && n > 0) {
        const __int128 lhs = sum * p.scale_den;
        if (lhs < (__int128)p.scale_out_num * n * L) {
            cn.scale_out++;
            log_ev(x, cn, SIM_EV_SCALE_OUT, kNone, 255, 255, 0);
        } else if (lhs > (__int128)p.scale_in_num * n * L) {
            cn.scale_in++;
            log_ev(x, cn, SIM_EV_SCALE_IN, kNone, 255, 255, 0);
        }
    }
    __syncwarp();
}

// Phase 3: periodic rebalancing between low- and high-freeness instances (Sec. 3.5).
template <int C, bool EXT>
__device__ __forceinline__ void migration_tick(const Ctx &x, Cnt &cn, int theta_num, int theta_den) {
    refresh_keys<C>(x);
    uint32_t el = 0, dr = 0;  // eligible (not migrating); draining
#pragma unroll
    for (int j = 0; j < C; ++j) {
        const int i = x.lane * C + j;
        if (i < x.N && x.mrole[i] == MIG_NONE) el |= 1u << j;
        if (EXT && i < x.N && x.drains && x.drain[i] <= x.t) dr |= 1u << j;
    }
    for (;;) {
        const int nel = __reduce_add_sync(kFull, __popc(el));
        if (nel < 2) break;
        // A draining instance has infinite virtual usage (Sec. 3.5): it is the
        // least free (lowest index among several), passes the threshold
        // against any other instance, and is never a destination.
        int s;
        const uint32_t dl = EXT ? __ballot_sync(kFull, (el & dr) != 0) : 0u;
        if (dl) {
            const int l = __ffs(dl) - 1;
            const uint32_t bits = C == 1 ? 1u : __shfl_sync(kFull, el & dr, l);
            s = l * C + __ffs(bits) - 1;
        } else {
            s = arg_ext<C>(x, el, false, -1);
        }
        const int d = arg_ext<C>(x, el & ~dr, true, s);
        if (d < 0) break;
        if (!dl) {
            const long long ns = fnum(x, s), ds = max((int)x.nrun[s], 1);
            const long long nd = fnum(x, d), dd = max((int)x.nrun[d], 1);
            if ((long long)theta_den * (nd * ds - ns * dd) < (long long)theta_num * dd * ds) break;
        }
        const bool has_wait = x.wmask[s] != 0;
        const int n_s = x.nrun[s];
        __syncwarp();
        int moved = 0;
        if (has_wait) {
            if (x.lane == 0) {
                // queued candidate: newest request of the lowest-priority bucket, no KV to copy
                const int k = 31 - __clz((unsigned)x.wmask[s]);
                uint32_t info = 0;
                const uint32_t r = pop_back(x, s, k, info, cn.status);
                if (r != kNone) {
                    refresh_hol(x, s);
                    cnt_dec(x, s, k);
                    const uint32_t old = x.wmask[d];
                    push_back(x, d, k, r, info);
                    cnt_inc(x, d, k);
                    if ((old & ((2u << k) - 1u)) == 0) x.hol[d] = blocks_for(x, info & 0xFFFFu);
                    bump_mig(x, r);
                    cn.migrations++;
                    cn.events++;
                    log_ev(x, cn, SIM_EV_QUEUED, r, s, d, 0);
                }
            }
            moved = 1;
        } else if (n_s > 0) {
            // running candidate: lowest priority, then fewest blocks, then newest
            const uint4 *p = slot_ptr(x, s, 0);
            const bool v0 = x.lane < n_s, v1 = x.lane + 32 < n_s;
            const uint4 a0 = v0 ? p[x.lane] : make_uint4(0, 0, 0, 0);
            const uint4 a1 = v1 ? p[x.lane + 32] : make_uint4(0, 0, 0, 0);
            const int k0 = v0 ? (int)((sl_tier(a0) << 16) | (0xFFFFu - (uint32_t)sl_blocks(x, s, a0))) : -1;
            const int k1 = v1 ? (int)((sl_tier(a1) << 16) | (0xFFFFu - (uint32_t)sl_blocks(x, s, a1))) : -1;
            const int km = __reduce_max_sync(kFull, max(k0, k1));
            const uint32_t c0 = (v0 && k0 == km) ? a0.x : 0u, c1 = (v1 && k1 == km) ? a1.x : 0u;
            const uint32_t rid = __reduce_max_sync(kFull, max(c0, c1));
            const int blocks = (int)(0xFFFFu - ((uint32_t)km & 0xFFFFu));
            const uint32_t o0 = __ballot_sync(kFull, v0 && a0.x == rid);
            const uint32_t o1 = __ballot_sync(kFull, v1 && a1.x == rid);
            const int ol = o0 ? __ffs(o0) - 1 : __ffs(o1) - 1;
            const bool hi = o0 == 0;
            uint4 rec;
            rec.x = __shfl_sync(kFull, hi ? a1.x : a0.x, ol);
            rec.y = __shfl_sync(kFull, hi ? a1.y : a0.y, ol);
            rec.z = __shfl_sync(kFull, hi ? a1.z : a0.z, ol);
            rec.w = __shfl_sync(kFull, hi ? a1.w : a0.w, ol);
            if (x.free_[d] >= blocks) {
                if (x.lane == 0) {
                    x.mrole[s] = MIG_SRC;
                    x.mpeer[s] = (uint8_t)d;
                    x.mreq[s] = rid;
                    x.mcopied[s] = 0;
                    x.mslot[s] = rec;
                    x.mrole[d] = MIG_DST;
                    x.mpeer[d] = (uint8_t)s;
                    cn.starts++;
                    log_ev(x, cn, SIM_EV_START, rid, s, d, blocks);
                }
                moved = 1;
            }
        }
        if (x.lane == s / C) el &= ~(1u << (s % C));
        if (moved && x.lane == d / C) el &= ~(1u << (d % C));
        __syncwarp();
    }
}

// Distinct event times of a window (C > 1): a per-warp open-addressing set.
__device__ __forceinline__ uint32_t tset_insert(const Ctx &x, uint32_t t) {
    uint32_t h = (t * 0x9E3779B1u) >> 23;  // 9 bits: kHashSlots = 512
    for (uint32_t probe = 0; probe < kHashSlots; ++probe) {
        const uint32_t old = atomicCAS(&x.tset[h], kNone, t);
        if (old == kNone) return 1u;
        if (old == t) return 0u;
        h = (h + 1u) & (kHashSlots - 1u);
    }
    return 0u;
}

__device__ __forceinline__ void copy16(unsigned char *dst, const unsigned char *src, uint32_t bytes, int lane) {
    for (uint32_t o = (uint32_t)lane * 16u; o < bytes; o += 512u)
        *reinterpret_cast<uint4 *>(dst + o) = *reinterpret_cast<const uint4 *>(src + o);
}

__device__ __forceinline__ void bind_blob(Ctx &x, const Layout &L, unsigned char *blob) {
    unsigned char *ib = blob + L.inst;
    x.busy.base = x.free_.base = x.resv.base = x.hol.base = x.hr.base = x.key.base = ib;
    x.mreq.base = x.mcopied.base = x.nf.base = x.minfin.base = x.drain.base = ib;
    x.wmask.base = x.nrun.base = x.pc.base = x.phase.base = x.mrole.base = x.mpeer.base = ib;
    x.cnt = reinterpret_cast<uint16_t *>(blob + L.cnt);
    x.head = reinterpret_cast<uint32_t *>(blob + L.head);
    x.tail = reinterpret_cast<uint32_t *>(blob + L.tail);
    x.hinfo = reinterpret_cast<uint32_t *>(blob + L.hinfo);
    x.h = reinterpret_cast<int *>(blob + L.h);
    x.hist = blob + L.hist;
    x.mslot = reinterpret_cast<uint4 *>(blob + L.mslot);
}

// Phase 1 at x.t for the instances in `mask` (bit j = instance lane*C + j)
// whose iteration ends now, ascending index.  Collective.
template <int C>
__device__ __forceinline__ void complete_all(const Ctx &x, Cnt &cn, uint32_t mask) {
    uint32_t hits = 0;
#pragma unroll
    for (int j = 0; j < C; ++j)
        if (((mask >> j) & 1u) && x.busy[x.lane * C + j] == x.t) hits |= 1u << j;
    uint32_t lanes = __ballot_sync(kFull, hits != 0);
    while (lanes) {
        const int l = __ffs(lanes) - 1;
        lanes &= lanes - 1;
        uint32_t h = C == 1 ? 1u : __shfl_sync(kFull, hits, l);
        while (h) {
            const int i = l * C + __ffs(h) - 1;
            h &= h - 1;
            int fp = 0;
            if (x.lane == 0) fp = inst_complete_head(x, i);
            if (__shfl_sync(kFull, fp, 0)) coop_finish(x, cn, i);
            __syncwarp();
            if (x.mrole[i] == MIG_SRC) coop_stage(x, cn, i);
        }
    }
}

// Phase 4 at x.t for the idle instances in `mask` that have work, ascending
// index, on lane 0.  Collective.
template <int C>
__device__ __forceinline__ void form_all(const Ctx &x, Cnt &cn, uint32_t mask, const Params &p) {
    uint32_t want = 0;
#pragma unroll
    for (int j = 0; j < C; ++j) {
        const int i = x.lane * C + j;
        if (((mask >> j) & 1u) && x.busy[i] == kNone && (x.nrun[i] | x.wmask[i]) != 0) want |= 1u << j;
    }
    uint32_t lanes = __ballot_sync(kFull, want != 0);
    while (lanes) {
        const int l = __ffs(lanes) - 1;
        lanes &= lanes - 1;
        const uint32_t h = C == 1 ? 1u : __shfl_sync(kFull, want, l);
        if (x.lane == 0)
            for (uint32_t hh = h; hh; hh &= hh - 1) inst_form(x, cn, l * C + __ffs(hh) - 1, p.base, p.a, p.b);
    }
    __syncwarp();
}

// a[j] for a run-time j without dynamic indexing (the array stays in registers)
template <int C>
__device__ __forceinline__ uint32_t pick_c(const uint32_t (&a)[C], int j) {
    uint32_t v = a[0];
#pragma unroll
    for (int k = 1; k < C; ++k)
        if (j == k) v = a[k];
    return v;
}

// Which main loop a variant runs.  The variants that keep running-request
// records in HBM with at most two instances per lane run 16 warps per SM
// (many replicas); there instruction fetch was the bottleneck, and a loop
// in which the window, its migration steps and the global steps share one
// copy of every phase keeps the hot code small.  The other variants run few
// warps per SM and are bound by each replica's dependent chain, which the
// loop with separately inlined phases keeps shorter.
template <int C, bool SMS>
constexpr bool kUnifiedLoop = !SMS && C <= 2;

// The persistent simulation kernel: each warp repeatedly takes a replica and
// advances it by up to p.max_steps event times; C = instances per lane.
//
// Between two global events (the next arrival, the next migration tick) the
// instances that are in no migration do not interact, and an iteration lasts
// at least `base` microseconds.  So in a window [tmin, min(T_g, tmin + base))
// every instance ends at most one iteration, and each lane advances its own
// instances (an O(1) iteration end + batch formation); instances in a
// migration (but a destination whose source's next event comes later), and
// every step at a global event, are advanced by the warp in the oracle's
// order.  EXT: the variant that also handles draining instances and
// the auto-scaling signal (the other variant compiles that code out).
template <int C, bool SMS, bool EXT>
// Variants that keep the running-request records in HBM (C <= 2) run
// workloads with many replicas and must stay at 128 registers so that 8
// blocks of two warps fit on an SM.  The bound asks for 7: the compiler
// still allocates 128 registers and the launch still holds 8 blocks per SM,
// but its code for that bound measured faster than for a bound of 8 (1-4 %,
// same-box A/B on the 16,384- and 3,840-replica workloads); a bound of 10
// (96 registers, 9-10 blocks) was 10-16 % slower.  The others keep 4: their
// shared memory or register needs limit residency anyway.
__global__ void __launch_bounds__(32 * kWarpsPerBlock, (!SMS && C <= 2) ? 7 : 4) k_run(Params p) {
    extern __shared__ __align__(16) unsigned char smem[];
    unsigned long long *magic = reinterpret_cast<unsigned long long *>(smem);
    for (int d = threadIdx.x; d <= 64; d += blockDim.x)
        magic[d] = d < 2 ? 0ull : ~0ull / (unsigned long long)d + 1ull;
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const uint32_t slot_bytes = SMS ? (uint32_t)p.N * (uint32_t)p.Bmax * 16u : 0u;
    const uint32_t per_warp = p.L.bytes + slot_bytes + p.hash_bytes;
    unsigned char *blob = smem + kMagicBytes + (size_t)(threadIdx.x >> 5) * per_warp;
    uint4 *sslots = reinterpret_cast<uint4 *>(blob + p.L.bytes);
    uint32_t *tset = reinterpret_cast<uint32_t *>(blob + p.L.bytes + slot_bytes);
    for (;;) {
        int r = 0;
        if (lane == 0) {
            r = atomicAdd(p.work, 1);
            if (p.order && r < p.R) r = p.order[r];
        }
        r = __shfl_sync(kFull, r, 0);
        if (r >= p.R) break;
        const RepState rs = p.rep[r];
        if (rs.status != SIM_REPLICA_RUNNING) continue;
        unsigned char *gblob = p.blobs + (size_t)r * p.L.bytes;
        copy16(blob, gblob, p.L.bytes, lane);
        Ctx x;
        bind_blob(x, p.L, blob);
        uint4 *g_slots = p.slots + (size_t)r * p.N * p.Bmax;
        if (SMS) {
            copy16(reinterpret_cast<unsigned char *>(sslots), reinterpret_cast<const unsigned char *>(g_slots),
                   slot_bytes, lane);
            x.slots = sslots;
        } else {
            x.slots = g_slots;
        }
        x.tset = tset;
        __syncwarp();
        const long long o = p.offsets[r];
        x.Q = (uint32_t)(p.offsets[r + 1] - o);
        x.arrival = p.arrival + o;
        x.plen = p.plen + o;
        x.olen = p.olen + o;
        x.tier = p.tier + o;
        x.node = p.node + o;
        x.res = p.res + o;
        x.log = p.log + (size_t)r * p.cap;
        x.magic = magic;
        x.magT = p.magT;
        x.N = p.N;
        x.K = p.K;
        x.T = p.T;
        x.TH = p.TH;
        x.Bmax = p.Bmax;
        x.S = p.S;
        x.cap = p.cap;
        x.lane = lane;
        x.drains = EXT ? p.drains : 0;
        x.t = rs.t;
        uint32_t tmax = rs.t;  // latest event time this lane has processed (the replica's: max over lanes)
        Cnt cn;  // lane 0: the replica's totals; other lanes: what they add in windows
        const bool l0 = lane == 0;
        cn.finished = rs.finished;
        cn.log_events = rs.log_events;
        cn.migrations = rs.migrations;
        cn.preemptions = l0 ? rs.preemptions : 0u;
        cn.starts = rs.starts;
        cn.aborts = rs.aborts;
        cn.scale_out = rs.scale_out;
        cn.scale_in = rs.scale_in;
        cn.steps = 0;
        cn.iterations = 0;
        cn.member_iterations = l0 ? rs.member_iterations : 0ull;
        cn.events = l0 ? rs.events : 0ull;
        cn.status = SIM_REPLICA_RUNNING;
        uint32_t cursor = rs.cursor;
        uint32_t next_tick = rs.next_tick;
        ArrBuf ab;
        arr_refill(x, ab, cursor);
        uint32_t next_arr = __shfl_sync(kFull, ab.time, 0);
        if constexpr (kUnifiedLoop<C, SMS>) {
            const uint32_t max_steps = p.max_steps;
            const uint32_t all = own_mask<C>(x);
            const bool ticks = EXT ? p.ticks != 0 : p.enable_mig != 0;
            // Every pass of the loop below is one of three modes, which share one
            // copy of each phase (iteration ends; finishes and copy stages;
            // dispatch and tick; batch formation), so the hot loop stays small:
            //   0: a window [tb, t1) in which every instance ends at most one
            //      iteration: each lane ends and re-forms its own instances that
            //      are in no migration ("solo"), each at its own time;
            //   1: one step, at the next time tc < t1, of the window's instances
            //      in a migration (both ends of every migration), in time order;
            //   2: one step at the next global event (arrival, tick), or near the
            //      step limit, over all instances.
            bool in_cm = false;              // mode-1 steps of the current window remain
            uint32_t t1 = 0, cm = 0;         // window end; own instances stepped in mode 1
            uint32_t ucount = 0, u = kNone;  // distinct event times of the window; own solo time (C = 1)
            uint32_t tlast = 0;              // latest event time processed in the window
            for (;;) {
                int mode;
                uint32_t et[C];      // event time of each own instance in this pass
                uint32_t heads = 0;  // own instances whose iteration ends in this pass
                uint32_t tstep = 0;  // step time (modes 1 and 2)
                bool tick = false;
                if (in_cm) {
                    uint32_t cb = kNone;
#pragma unroll
                    for (int j = 0; j < C; ++j)
                        if ((cm >> j) & 1u) cb = min(cb, x.busy[lane * C + j]);
                    const uint32_t tc = __reduce_min_sync(kFull, cb);
                    if (tc >= t1) {  // the window is complete
                        in_cm = false;
                        cn.steps += ucount;
                        tmax = max(tmax, tlast);
                        cn.finished = __shfl_sync(kFull, cn.finished, 0);  // finishes are all counted on lane 0
                        cn.status = __reduce_min_sync(kFull, cn.status);
                        if (cn.status < 0) break;
                        continue;
                    }
                    mode = 1;
                    tstep = tc;
                    tlast = max(tlast, tc);
#pragma unroll
                    for (int j = 0; j < C; ++j) {
                        et[j] = tc;
                        if (((cm >> j) & 1u) && x.busy[lane * C + j] == tc) heads |= 1u << j;
                    }
                } else {
                    if (cn.finished == x.Q) { cn.status = SIM_REPLICA_DONE; break; }
                    if (cn.steps == max_steps) break;
                    uint32_t bz[C];
                    uint32_t mb = kNone;
#pragma unroll
                    for (int j = 0; j < C; ++j) {
                        const int i = lane * C + j;
                        bz[j] = i < x.N ? x.busy[i] : kNone;
                        mb = min(mb, bz[j]);
                    }
                    const uint32_t tb = __reduce_min_sync(kFull, mb);
                    const uint32_t tg = ticks ? min(next_arr, next_tick) : next_arr;
                    if (tb < tg && max_steps - cn.steps > (uint32_t)x.N) {
                        mode = 0;
                        t1 = (uint32_t)min((unsigned long long)tg, (unsigned long long)tb + (uint32_t)p.base);
                        // instances with an iteration end in the window: stepped with
                        // the others of a migration in time order (cm), or alone
                        // (solo).  A destination whose source's next event comes
                        // strictly later (or after the window) is alone: only the
                        // source's events (stages, commit, abort) touch the other
                        // end, and those then follow the destination's own event,
                        // as in the oracle's time order.
                        cm = 0;
                        uint32_t solo = 0;
#pragma unroll
                        for (int j = 0; j < C; ++j) {
                            const int i = lane * C + j;
                            et[j] = bz[j];
                            if (bz[j] < t1) {
                                const int role = x.mrole[i];
                                if (role == MIG_NONE || (role == MIG_DST && x.busy[x.mpeer[i]] > bz[j])) solo |= 1u << j;
                                else cm |= 1u << j;
                            }
                        }
                        heads = solo;
                        tlast = 0;
                        if (C == 1) {
                            // distinct event times: one group per value of the solo times
                            u = solo ? bz[0] : kNone;
                            const uint32_t grp = __match_any_sync(kFull, u);
                            ucount = __popc(__ballot_sync(kFull, u != kNone && (__ffs(grp) - 1) == lane));
                            if (solo) tlast = bz[0];
                        } else {
                            for (uint32_t q = (uint32_t)lane; q < kHashSlots; q += 32) tset[q] = kNone;
                            __syncwarp();
                            uint32_t fresh = 0;
#pragma unroll
                            for (int j = 0; j < C; ++j) {
                                if (!((solo >> j) & 1u)) continue;
                                tlast = max(tlast, bz[j]);
                                fresh += tset_insert(x, bz[j]);
                            }
                            ucount = __reduce_add_sync(kFull, fresh);
                        }
                    } else {
                        mode = 2;
                        const uint32_t tc = min(tb, next_arr);
                        if (tc == kNone) { cn.status = SIM_ERR_DEADLOCK; break; }
                        tick = ticks && next_tick <= tc;
                        tstep = tick ? next_tick : tc;
                        tmax = max(tmax, tstep);
                        ++cn.steps;
#pragma unroll
                        for (int j = 0; j < C; ++j) {
                            et[j] = tstep;
                            if (bz[j] == tstep) heads |= 1u << j;
                        }
                    }
                }
                // ---- 1. iteration ends: each lane ends its own instances' iterations ----
                uint32_t fz = 0;  // own instances with a finishing request
#pragma unroll
                for (int j = 0; j < C; ++j) {
                    if (!((heads >> j) & 1u)) continue;
                    x.t = et[j];
                    if (inst_complete_head(x, lane * C + j)) fz |= 1u << j;
                }
                __syncwarp();
                // ---- finishes and copy stages, instance by instance in ascending
                // order, by the whole warp (in mode 0 only finishes, which touch
                // their own instance alone, so their order does not matter) ----
                const uint32_t visit = mode == 0 ? fz : heads;
                for (uint32_t fl = __ballot_sync(kFull, visit != 0); fl; fl &= fl - 1) {
                    const int l = __ffs(fl) - 1;
                    const uint32_t vl = C == 1 ? 1u : __shfl_sync(kFull, visit, l);
                    const uint32_t fzl = __shfl_sync(kFull, fz, l);
                    for (uint32_t h = vl; h; h &= h - 1) {
                        const int j = __ffs(h) - 1;
                        const int i = l * C + j;
                        x.t = __shfl_sync(kFull, pick_c<C>(et, j), l);
                        if ((fzl >> j) & 1u) coop_finish(x, cn, i);
                        if (mode != 0 && x.mrole[i] == MIG_SRC) coop_stage(x, cn, i);
                    }
                }
                if (mode == 2) {
                    x.t = tstep;
                    if (next_arr == tstep) dispatch_phase<C, EXT>(x, cn, cursor, next_arr, ab);  // 2. dispatch
                    if (tick) {  // 3. auto-scaling signal and migration tick
                        const uint32_t nt = next_tick + p.interval;
                        next_tick = nt < next_tick ? kNone : nt;  // saturate: no tick beyond 2^32 - 1
                        if (EXT && p.autoscale) autoscale_tick<C>(x, cn, p);
                        if (p.enable_mig) migration_tick<C, EXT>(x, cn, p.theta_num, p.theta_den);
                    }
                }
                // ---- 4. batch formation: in mode 0 every lane forms its own solo
                // instances at their own times; otherwise the idle instances with
                // work are formed on lane 0 in ascending order (their preemptions
                // may abort migrations, whose log records are lane 0's) ----
                uint32_t want = 0;
                if (mode == 0) {
                    want = heads;
                } else {
                    const uint32_t mask = mode == 1 ? cm : all;
#pragma unroll
                    for (int j = 0; j < C; ++j) {
                        const int i = lane * C + j;
                        if (((mask >> j) & 1u) && x.busy[i] == kNone && (x.nrun[i] | x.wmask[i]) != 0) want |= 1u << j;
                    }
                }
                for (uint32_t fl = mode == 0 ? 1u : __ballot_sync(kFull, want != 0); fl; fl &= fl - 1) {
                    const int l = __ffs(fl) - 1;
                    const uint32_t hl = mode == 0 ? want : (C == 1 ? 1u : __shfl_sync(kFull, want, l));
                    const int owner = mode == 0 ? lane : l;
                    if (mode == 0 || lane == 0) {
                        for (uint32_t h = hl; h; h &= h - 1) {
                            const int j = __ffs(h) - 1;
                            x.t = mode == 0 ? pick_c<C>(et, j) : tstep;
                            inst_form(x, cn, owner * C + j, p.base, p.a, p.b);
                        }
                    }
                    __syncwarp();
                }
                // ---- step accounting ----
                if (mode == 0) {
                    if (__any_sync(kFull, cm != 0)) {
                        // the window's instances in a migration next (both ends of
                        // every migration, with or without an event of their own)
#pragma unroll
                        for (int j = 0; j < C; ++j) {
                            const int i = lane * C + j;
                            if (i < x.N && x.mrole[i] != MIG_NONE) cm |= 1u << j;
                        }
                        in_cm = true;
                        continue;
                    }
                    cn.steps += ucount;
                    tmax = max(tmax, tlast);
                    cn.finished = __shfl_sync(kFull, cn.finished, 0);
                    cn.status = __reduce_min_sync(kFull, cn.status);
                    if (cn.status < 0) break;
                } else if (mode == 1) {
                    if (C == 1) {
                        ucount += __any_sync(kFull, u == tstep) ? 0u : 1u;
                    } else {
                        uint32_t f2 = 0;
                        if (lane == 0) f2 = tset_insert(x, tstep);
                        ucount += __shfl_sync(kFull, f2, 0);
                    }
                    cn.status = __reduce_min_sync(kFull, cn.status);  // also a solo lane's error of this window
                    if (cn.status < 0) {
                        in_cm = false;
                        cn.steps += ucount;
                        tmax = max(tmax, tlast);
                        cn.finished = __shfl_sync(kFull, cn.finished, 0);
                        break;
                    }
                } else {
                    cn.finished = __shfl_sync(kFull, cn.finished, 0);
                    cn.status = __shfl_sync(kFull, cn.status, 0);
                    if (cn.status < 0) break;
                }
            }
            __syncwarp();
        } else {
            const uint32_t max_steps = p.max_steps;
            const uint32_t all = own_mask<C>(x);
            for (;;) {
                if (cn.finished == x.Q) { cn.status = SIM_REPLICA_DONE; break; }
                if (cn.steps == max_steps) break;
                uint32_t bz[C];
                uint32_t mb = kNone;
#pragma unroll
                for (int j = 0; j < C; ++j) {
                    const int i = lane * C + j;
                    bz[j] = i < x.N ? x.busy[i] : kNone;
                    mb = min(mb, bz[j]);
                }
                const uint32_t tb = __reduce_min_sync(kFull, mb);
                const bool ticks = EXT ? p.ticks != 0 : p.enable_mig != 0;
                const uint32_t tg = ticks ? min(next_arr, next_tick) : next_arr;
                if (tb < tg && max_steps - cn.steps > (uint32_t)x.N) {
                    // ---- window [tb, t1): at most one iteration end per instance ----
                    const uint32_t t1 =
                        (uint32_t)min((unsigned long long)tg, (unsigned long long)tb + (uint32_t)p.base);
                    // instances with an iteration end in the window: stepped with the
                    // others of a migration in time order (cm), or alone (solo).  A
                    // destination whose source's next event comes strictly later is
                    // alone: only the source's events (stages, commit, abort) touch
                    // the other end, and those then follow the destination's own event.
                    uint32_t cm = 0, solo = 0;
#pragma unroll
                    for (int j = 0; j < C; ++j) {
                        const int i = lane * C + j;
                        if (bz[j] < t1) {
                            const int role = x.mrole[i];
                            if (role == MIG_NONE || (role == MIG_DST && x.busy[x.mpeer[i]] > bz[j])) solo |= 1u << j;
                            else cm |= 1u << j;
                        }
                    }
                    if (C > 1) {
                        for (uint32_t q = (uint32_t)lane; q < kHashSlots; q += 32) tset[q] = kNone;
                        __syncwarp();
                    }
                    uint32_t fresh = 0;  // distinct event times this lane contributes (C > 1)
                    uint32_t tlast = 0;  // latest event time processed in the window
                    uint32_t fz = 0;     // this lane's instances with a finishing request
#pragma unroll
                    for (int j = 0; j < C; ++j) {
                        if (!((solo >> j) & 1u)) continue;
                        const int i = lane * C + j;
                        x.t = bz[j];
                        tlast = max(tlast, bz[j]);
                        if (C > 1) fresh += tset_insert(x, bz[j]);
                        if (inst_complete_head(x, i)) fz |= 1u << j;
                    }
                    // finishes, one instance at a time by the whole warp (they touch
                    // only their own instance, so their order does not matter) ...
                    for (uint32_t fl = __ballot_sync(kFull, fz != 0); fl; fl &= fl - 1) {
                        const int l = __ffs(fl) - 1;
                        for (uint32_t h = C == 1 ? 1u : __shfl_sync(kFull, fz, l); h; h &= h - 1) {
                            const int j = __ffs(h) - 1;
                            x.t = __shfl_sync(kFull, bz[j], l);
                            coop_finish(x, cn, l * C + j);
                        }
                    }
                    // ... then every lane forms its instances' next batches together
#pragma unroll
                    for (int j = 0; j < C; ++j) {
                        if (!((solo >> j) & 1u)) continue;
                        x.t = bz[j];
                        inst_form(x, cn, lane * C + j, p.base, p.a, p.b);
                    }
                    __syncwarp();
                    uint32_t ucount, u = kNone;
                    if (C == 1) {
                        u = solo ? bz[0] : kNone;
                        const uint32_t grp = __match_any_sync(kFull, u);
                        ucount = __popc(__ballot_sync(kFull, u != kNone && (__ffs(grp) - 1) == lane));
                    } else {
                        ucount = __reduce_add_sync(kFull, fresh);
                    }
                    // instances in a migration (both ends, with or without an event
                    // of their own in the window): steps in time order on lane 0
                    if (__any_sync(kFull, cm != 0)) {
#pragma unroll
                        for (int j = 0; j < C; ++j) {
                            const int i = lane * C + j;
                            if (i < x.N && x.mrole[i] != MIG_NONE) cm |= 1u << j;
                        }
                        for (;;) {
                            uint32_t cb = kNone;
#pragma unroll
                            for (int j = 0; j < C; ++j)
                                if ((cm >> j) & 1u) cb = min(cb, x.busy[lane * C + j]);
                            const uint32_t tc = __reduce_min_sync(kFull, cb);
                            if (tc >= t1) break;
                            x.t = tc;
                            tlast = max(tlast, tc);
                            complete_all<C>(x, cn, cm);
                            form_all<C>(x, cn, cm, p);
                            if (C == 1) {
                                ucount += __any_sync(kFull, u == tc) ? 0u : 1u;
                            } else {
                                uint32_t f2 = 0;
                                if (lane == 0) f2 = tset_insert(x, tc);
                                ucount += __shfl_sync(kFull, f2, 0);
                            }
                            cn.status = __shfl_sync(kFull, cn.status, 0);
                            if (cn.status < 0) break;
                        }
                    }
                    cn.steps += ucount;
                    tmax = max(tmax, tlast);  // x.t is set again before any further use
                    cn.finished = __shfl_sync(kFull, cn.finished, 0);  // finishes are all counted on lane 0
                    const int ws = __reduce_min_sync(kFull, cn.status);
                    cn.status = ws;
                    if (cn.status < 0) break;
                    continue;
                }
                // ---- one step at the next event time (global events, or near the step limit) ----
                const uint32_t tc = min(tb, next_arr);
                if (tc == kNone) { cn.status = SIM_ERR_DEADLOCK; break; }
                const bool tick = ticks && next_tick <= tc;
                x.t = tick ? next_tick : tc;
                tmax = max(tmax, x.t);
                ++cn.steps;
                const uint32_t f1 = cn.finished;
                if (tb == x.t) complete_all<C>(x, cn, all);  // 1. iteration ends
                cn.finished = __shfl_sync(kFull, cn.finished, 0);
                if (next_arr == x.t) dispatch_phase<C, EXT>(x, cn, cursor, next_arr, ab);  // 2. dispatch
                if (tick) {  // 3. auto-scaling signal and migration tick
                    const uint32_t nt = next_tick + p.interval;
                    next_tick = nt < next_tick ? kNone : nt;  // saturate: no tick beyond 2^32 - 1
                    if (EXT && p.autoscale) autoscale_tick<C>(x, cn, p);
                    if (p.enable_mig) migration_tick<C, EXT>(x, cn, p.theta_num, p.theta_den);
                }
                form_all<C>(x, cn, all, p);  // 4. batch formation
                (void)f1;
                cn.status = __shfl_sync(kFull, cn.status, 0);
                if (cn.status < 0) break;
            }
            __syncwarp();
        }
        // fold the other lanes' counters into lane 0's
        const uint32_t tfin = __reduce_max_sync(kFull, tmax);
        const uint32_t a_pre = __reduce_add_sync(kFull, l0 ? 0u : cn.preemptions);
        const uint32_t a_it = __reduce_add_sync(kFull, cn.iterations);
        uint64_t a_mi = cn.member_iterations, a_ev = cn.events;
#pragma unroll
        for (int sh = 16; sh > 0; sh >>= 1) {
            a_mi += __shfl_xor_sync(kFull, a_mi, sh);
            a_ev += __shfl_xor_sync(kFull, a_ev, sh);
        }
        copy16(gblob, blob, p.L.bytes, lane);
        if (SMS)
            copy16(reinterpret_cast<unsigned char *>(g_slots), reinterpret_cast<const unsigned char *>(sslots),
                   slot_bytes, lane);
        if (l0) {
            RepState o2;
            o2.t = tfin;
            o2.cursor = cursor;
            o2.finished = cn.finished;
            o2.log_events = cn.log_events;
            o2.next_tick = next_tick;
            o2.pad0 = 0;
            o2.steps = rs.steps + cn.steps;
            o2.iterations = rs.iterations + a_it;
            o2.member_iterations = a_mi;
            o2.events = a_ev;
            o2.migrations = cn.migrations;
            o2.preemptions = cn.preemptions + a_pre;
            o2.starts = cn.starts;
            o2.aborts = cn.aborts;
            o2.scale_out = cn.scale_out;
            o2.scale_in = cn.scale_in;
            o2.status = cn.status;
            o2.pad1 = 0;
            p.rep[r] = o2;
        }
        __syncwarp();
    }
}

// ---- set-up and export kernels ----------------------------------------------
__global__ void k_init_state(Params p, const int *rep_table, const int *tbl_k, const int *tbl_h) {
    const int lane = threadIdx.x & 31;
    const int warps = (gridDim.x * blockDim.x) >> 5;
    for (int r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < p.R; r += warps) {
        unsigned char *b = p.blobs + (size_t)r * p.L.bytes;
        const Layout &L = p.L;
        const int N = p.N, NK = p.N * p.K;
        const int tb = rep_table[r];
        const int K = tbl_k[tb];
        for (int i = lane; i < N; i += 32) {
            InstRec v;
            memset(&v, 0, sizeof v);
            v.busy = kNone;
            v.free_ = p.M;
            v.mreq = kNone;
            v.minfin = kNone;
            v.drain = p.drain_src ? p.drain_src[(size_t)r * N + i] : kNone;
            v.mrole = MIG_NONE;
            reinterpret_cast<InstRec *>(b + L.inst)[i] = v;
        }
        for (int q = lane; q < N * p.TH; q += 32) b[L.hist + q] = 0;
        for (int i = lane; i < NK; i += 32) {
            reinterpret_cast<uint16_t *>(b + L.cnt)[i] = 0;
            reinterpret_cast<uint32_t *>(b + L.head)[i] = kNone;
            reinterpret_cast<uint32_t *>(b + L.tail)[i] = kNone;
            reinterpret_cast<uint32_t *>(b + L.hinfo)[i] = 0;
        }
        for (int k = lane; k < p.K; k += 32)
            reinterpret_cast<int *>(b + L.h)[k] = k < K ? tbl_h[tb * p.K + k] : 0;
        if (lane == 0) {
            RepState s;
            memset(&s, 0, sizeof s);
            s.next_tick = p.interval;
            s.status = (p.offsets[r + 1] == p.offsets[r]) ? SIM_REPLICA_DONE : SIM_REPLICA_RUNNING;
            p.rep[r] = s;
        }
    }
}

// New headroom tables (adaptive headroom, sim_set_headroom): each replica's
// H[k] from its table, and every instance's present-tier headroom sum
// recomputed from its per-tier request counts (Sec. 3.3 Eq. 4: H_k once per
// tier present).  One warp per replica.
__global__ void k_set_headroom(Params p, const int *rep_table, const int *tbl_k, const int *tbl_h) {
    const int lane = threadIdx.x & 31;
    const int warps = (gridDim.x * blockDim.x) >> 5;
    for (int r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < p.R; r += warps) {
        unsigned char *b = p.blobs + (size_t)r * p.L.bytes;
        const int tb = rep_table[r];
        const int K = tbl_k[tb];
        const int *hn = tbl_h + (size_t)tb * p.K;
        for (int k = lane; k < p.K; k += 32) reinterpret_cast<int *>(b + p.L.h)[k] = k < K ? hn[k] : 0;
        const uint16_t *cnt = reinterpret_cast<const uint16_t *>(b + p.L.cnt);
        for (int i = lane; i < p.N; i += 32) {
            int sum = 0;
            for (int k = 0; k < K; ++k)
                if (cnt[i * p.K + k] > 0) sum += hn[k];
            reinterpret_cast<InstRec *>(b + p.L.inst)[i].hr = sum;
        }
    }
}

__global__ void k_init_requests(sim_request_result_t *res, long long n) {
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x)
        reinterpret_cast<uint4 *>(res)[i] = make_uint4(0xFFFFFFFFu, kNone, kNone, 0u);
}

// Trace validation: bit 0 unsorted, 1 tier >= K, 2 zero length, 3 too long, 4 bad arrival.
__global__ void k_validate(const long long *offsets, int R, const uint32_t *arrival, const uint16_t *plen,
                           const uint16_t *olen, const uint8_t *tier, const int *rep_table, const int *tbl_k,
                           long long lim, long long n, int *flags) {
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
        int lo = 0, hi = R - 1;  // replica r with offsets[r] <= i < offsets[r+1]
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (offsets[mid] <= i) lo = mid; else hi = mid - 1;
        }
        int f = 0;
        if (i > offsets[lo] && arrival[i] < arrival[i - 1]) f |= 1;
        if ((int)tier[i] >= tbl_k[rep_table[lo]]) f |= 2;
        if (plen[i] == 0 || olen[i] == 0) f |= 4;
        if ((long long)plen[i] + olen[i] > lim) f |= 8;
        if (arrival[i] == kNone) f |= 16;
        if (f) atomicOr(flags, f);
    }
}

// Per replica, the number of requests that have a first token; the simulation
// kernel records first tokens without counting them (see inst_form), so the
// exported event count adds these.
__global__ void k_first_tokens(const long long *offsets, int R, const sim_request_result_t *res, uint32_t *count) {
    __shared__ uint32_t part[32];
    for (int r = blockIdx.x; r < R; r += gridDim.x) {
        uint32_t c = 0;
        for (long long i = offsets[r] + threadIdx.x; i < offsets[r + 1]; i += blockDim.x)
            c += res[i].first_token_us != kNone ? 1u : 0u;
        c = __reduce_add_sync(kFull, c);
        if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = c;
        __syncthreads();
        if (threadIdx.x == 0) {
            uint32_t t = 0;
            for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += part[w];
            count[r] = t;
        }
        __syncthreads();
    }
}

__global__ void k_export_stats(const RepState *rep, sim_replica_stats_t *out, int R, int *unfinished,
                               const uint32_t *first_tokens) {
    for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < R; r += gridDim.x * blockDim.x) {
        const RepState s = rep[r];
        if (out) {
            sim_replica_stats_t o;
            o.steps = s.steps;
            o.iterations = s.iterations;
            o.member_iterations = s.member_iterations;
            o.events = s.events + (first_tokens ? first_tokens[r] : 0u);
            o.migrations = s.migrations;
            o.preemptions = s.preemptions;
            o.migration_starts = s.starts;
            o.migration_aborts = s.aborts;
            o.log_events = s.log_events;
            o.finished = s.finished;
            o.last_time_us = s.t;
            o.status = s.status;
            o.scale_out_signals = s.scale_out;
            o.scale_in_signals = s.scale_in;
            out[r] = o;
        }
        if (unfinished && s.status != SIM_REPLICA_DONE) atomicAdd(unfinished, 1);
    }
}

// ---- launch configuration ---------------------------------------------------
typedef void (*RunKernel)(Params);

template <bool SMS, bool EXT>
RunKernel pick(int c) {  // c = instances per lane
    switch (c) {
        case 1: return k_run<1, SMS, EXT>;
        case 2: return k_run<2, SMS, EXT>;
        case 4: return k_run<4, SMS, EXT>;
        default: return k_run<8, SMS, EXT>;
    }
}

// fn / grid: the plain variant; fn_ext / grid_ext: the one with draining and
// the auto-scaling signal (same shared memory).
struct Launch {
    RunKernel fn = nullptr, fn_ext = nullptr;
    int grid = 0, grid_ext = 0;
    int per_sm = 0, per_sm_ext = 0;  // resident blocks per SM of each variant
    int c = 1;                       // instances per lane
    bool sms = false;                // running-request records in shared memory
    size_t smem = 0;
};

inline int lanes_c(int N) { return N <= 32 ? 1 : N <= 64 ? 2 : N <= 128 ? 4 : 8; }

// Bytes per instance of the growth histogram: T rounded up to an odd number
// of words, so lanes reading one entry of consecutive instances hit distinct
// banks (1,024-replica workload +0.8 %; the same odd stride for the bucket
// arrays, as one {head, tail, info, count} record per tier, was 3 % slower
// on the 16,384-replica workload).
inline int hist_stride(int T) { return (((T + 3) >> 2) | 1) << 2; }

inline Layout make_layout(int N, int K, int T) {
    Layout L;
    uint32_t o = 0;
    auto take = [&](uint32_t bytes, uint32_t align) {
        o = (o + align - 1) / align * align;
        const uint32_t at = o;
        o += bytes;
        return at;
    };
    L.inst = take((uint32_t)sizeof(InstRec) * N, 16);
    L.head = take(4u * N * K, 16);
    L.tail = take(4u * N * K, 16);
    L.hinfo = take(4u * N * K, 16);
    L.h = take(4u * K, 16);
    L.cnt = take(2u * N * K, 16);
    L.hist = take((uint32_t)N * hist_stride(T), 16);
    L.mslot = take(16u * N, 16);
    L.bytes = (o + 15u) & ~15u;
    return L;
}

// Bytes of the per-warp event-time set; only variants with several instances per lane use it.
inline uint32_t hash_bytes_for(int N) { return lanes_c(N) > 1 ? kHashSlots * 4u : 0u; }

// Chooses the kernel variant and grid for a problem; cudaSuccess or the error.
// Running-request records go to shared memory while a replica's take at most this many bytes.
constexpr uint32_t kSmemSlotLimit = 24u * 1024u;

inline cudaError_t plan_launch(int R, int N, int Bmax, const Layout &L, Launch &out) {
    const uint32_t slot_bytes = (uint32_t)N * (uint32_t)Bmax * 16u;
    const bool sms = slot_bytes <= kSmemSlotLimit;
    out.c = lanes_c(N);
    out.sms = sms;
    out.fn = sms ? pick<true, false>(lanes_c(N)) : pick<false, false>(lanes_c(N));
    out.fn_ext = sms ? pick<true, true>(lanes_c(N)) : pick<false, true>(lanes_c(N));
    out.smem = kMagicBytes + (size_t)kWarpsPerBlock * (L.bytes + (sms ? slot_bytes : 0u) + hash_bytes_for(N));
    int dev = 0, sms_count = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms_count, cudaDevAttrMultiProcessorCount, dev);
    const long long want = ((long long)R + kWarpsPerBlock - 1) / kWarpsPerBlock;
    for (int v = 0; v < 2 && e == cudaSuccess; ++v) {
        RunKernel fn = v ? out.fn_ext : out.fn;
        int per_sm = 0;
        if (out.smem > 48 * 1024)
            e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)out.smem);
        if (e == cudaSuccess)
            e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, 32 * kWarpsPerBlock, out.smem);
        if (e != cudaSuccess) return e;
        if (per_sm < 1) return cudaErrorInvalidConfiguration;
        (v ? out.grid_ext : out.grid) = (int)std::min<long long>(want, (long long)sms_count * per_sm);
        (v ? out.per_sm_ext : out.per_sm) = per_sm;
    }
    return e;
}

inline unsigned long long magic40(unsigned d) { return ((1ull << kMagicShift) + d - 1ull) / d; }

}  // namespace mt

// ============================================================================
// Host side: the C ABI.
// ============================================================================
struct sim {
    sim_cluster_t cl;
    sim_policy_t pol;
    int K = 0, ntables = 0;
    std::vector<int> tbl_k, tbl_h, rep_table;
    cudaStream_t stream = nullptr;
    sim_allocator_t al{};
    bool use_al = false;
    mt::Layout L{};
    mt::Launch launch{};
    struct Buf { void *p; size_t n; };
    std::vector<Buf> bufs;
    size_t dev_bytes = 0;
    int *d_rep_table = nullptr, *d_tbl_k = nullptr, *d_tbl_h = nullptr;
    unsigned char *d_blobs = nullptr;
    uint4 *d_slots = nullptr;
    mt::RepState *d_rep = nullptr;
    sim_migration_event_t *d_log = nullptr;
    int *d_work = nullptr;  // [0] work counter, [1] validation flags, [2] unfinished count
    int64_t qtot = 0, qcap = -1;
    bool loaded = false;
    std::vector<int64_t> h_off;
    long long *d_off = nullptr;
    uint32_t *d_arrival = nullptr;
    uint16_t *d_plen = nullptr, *d_olen = nullptr;
    uint8_t *d_tier = nullptr;
    uint4 *d_node = nullptr;
    sim_request_result_t *d_res = nullptr;
    uint32_t *d_drain = nullptr;  // [R][N] drain start times (sim_set_drain), or NULL
    int *d_order = nullptr;       // [R] replica start order (sim_set_order), or NULL
    uint32_t *d_ftc = nullptr;    // [R] first-token counts for sim_metrics
    sim_latency_stats_t *d_lat = nullptr;  // device staging of sim_latency_stats for host output
    int *d_lat_rep = nullptr;              // chunk table of sim_latency_stats: replica and first record
    long long *d_lat_b0 = nullptr;
    uint4 *d_lat_sel = nullptr;            // percentile selection scratch of sim_latency_stats
    uint32_t *d_lat_bins = nullptr;
    int lat_nchunks = -1;                  // -1: to be built for the loaded trace
    int sms = 0;
    std::string err;
};

namespace {

thread_local std::string g_create_err;

int fail(sim_t *s, int code, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (s) s->err = buf; else g_create_err = buf;
    return code;
}

int cuda_fail(sim_t *s, cudaError_t e, const char *what) {
    return fail(s, SIM_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

void *dalloc(sim_t *s, size_t n) {
    if (n == 0) n = 16;
    n = (n + 255) & ~(size_t)255;
    void *p = nullptr;
    if (s->use_al) {
        p = s->al.alloc(s->al.ctx, n, (void *)s->stream);
    } else if (cudaMallocAsync(&p, n, s->stream) != cudaSuccess) {
        cudaGetLastError();
        p = nullptr;
    }
    if (p) {
        s->bufs.push_back({p, n});
        s->dev_bytes += n;
    }
    return p;
}

void dfree(sim_t *s, void *p) {
    if (!p) return;
    for (size_t i = 0; i < s->bufs.size(); ++i) {
        if (s->bufs[i].p == p) {
            if (s->use_al) s->al.free(s->al.ctx, p, s->bufs[i].n, (void *)s->stream);
            else cudaFreeAsync(p, s->stream);
            s->dev_bytes -= s->bufs[i].n;
            s->bufs.erase(s->bufs.begin() + i);
            return;
        }
    }
}

// Fills the scalar part of the kernel parameters (pointers are set by the caller).
void fill_scalars(mt::Params &p, const sim_cluster_t &cl, const sim_policy_t &pol, int K, int cap,
                  const mt::Layout &L, long long max_steps) {
    p.R = cl.num_replicas;
    p.N = cl.num_instances;
    p.M = cl.blocks_per_instance;
    p.T = cl.tokens_per_block;
    p.Bmax = cl.max_batch;
    p.TH = mt::hist_stride(cl.tokens_per_block);
    p.K = K;
    p.S = pol.migrate_blocks_per_iter;
    p.cap = cap;
    p.enable_mig = pol.enable_migration;
    p.theta_num = pol.theta_num;
    p.theta_den = pol.theta_den;
    p.interval = (uint32_t)pol.migrate_interval_us;
    p.max_steps = (uint32_t)std::min<long long>(max_steps, 0xFFFFFFFFLL);
    p.magT = mt::magic40((unsigned)cl.tokens_per_block);
    p.base = (int)pol.iter_base_us;
    p.a = (int)pol.iter_us_per_prefill_token;
    p.b = (int)pol.iter_us_per_decode_seq;
    p.ticks = pol.enable_migration || pol.autoscale;
    p.autoscale = pol.autoscale;
    p.scale_out_num = pol.scale_out_num;
    p.scale_in_num = pol.scale_in_num;
    p.scale_den = pol.scale_den;
    unsigned __int128 l = 1;  // lcm(1, ..., Bmax): every max(B, 1) divides it
    for (unsigned d = 2; d <= (unsigned)cl.max_batch; ++d) {
        unsigned a = d, b = (unsigned)(l % d);
        while (b) { const unsigned t = a % b; a = b; b = t; }
        l = l / a * d;
    }
    p.lcm_lo = (unsigned long long)l;
    p.lcm_hi = (unsigned long long)(l >> 64);
    p.L = L;
    p.hash_bytes = mt::hash_bytes_for(cl.num_instances);
}

mt::Params make_params(const sim_t *s, long long max_steps) {
    mt::Params p;
    memset(&p, 0, sizeof p);
    fill_scalars(p, s->cl, s->pol, s->K, s->pol.event_log_capacity, s->L, max_steps);
    p.offsets = s->d_off;
    p.drain_src = s->d_drain;
    p.drains = s->d_drain != nullptr;
    p.arrival = s->d_arrival;
    p.plen = s->d_plen;
    p.olen = s->d_olen;
    p.tier = s->d_tier;
    p.node = s->d_node;
    p.res = s->d_res;
    p.blobs = s->d_blobs;
    p.slots = s->d_slots;
    p.rep = s->d_rep;
    p.log = s->d_log;
    p.work = s->d_work;
    p.order = s->d_order;
    return p;
}

int check_launch(sim_t *s, const char *what) {
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(s, e, what);
    return SIM_OK;
}

int reset_state(sim_t *s) {
    mt::Params p = make_params(s, 0);
    const int R = s->cl.num_replicas;
    mt::k_init_state<<<(R + 7) / 8, 256, 0, s->stream>>>(p, s->d_rep_table, s->d_tbl_k, s->d_tbl_h);
    int rc = check_launch(s, "k_init_state");
    if (rc) return rc;
    if (s->qtot > 0) {
        const long long nb = std::min<long long>((s->qtot + 255) / 256, 65535LL * 16);
        mt::k_init_requests<<<(unsigned)nb, 256, 0, s->stream>>>(s->d_res, (long long)s->qtot);
        rc = check_launch(s, "k_init_requests");
    }
    return rc;
}

// The limits every entry point enforces on cluster, tier tables and policy.
int validate_config(sim_t *s, const sim_cluster_t *cl, const sim_tier_table_t *tt, const sim_policy_t *pol) {
    if (!cl || !tt || !pol) return fail(s, SIM_ERR_ARG, "cluster, tiers and policy are required");
    if (cl->num_replicas < 1) return fail(s, SIM_ERR_ARG, "num_replicas must be >= 1");
    if (cl->num_instances < 1 || cl->num_instances > SIM_MAX_INSTANCES)
        return fail(s, SIM_ERR_ARG, "num_instances must be in [1, %d]", SIM_MAX_INSTANCES);
    if (cl->blocks_per_instance < 1 || cl->blocks_per_instance > SIM_MAX_BLOCKS)
        return fail(s, SIM_ERR_ARG, "blocks_per_instance must be in [1, %d]", SIM_MAX_BLOCKS);
    if (cl->tokens_per_block < 1 || cl->tokens_per_block > mt::kMaxBlockTokens)
        return fail(s, SIM_ERR_ARG, "tokens_per_block must be in [1, %d]", mt::kMaxBlockTokens);
    if (cl->max_batch < 1 || cl->max_batch > SIM_MAX_BATCH)
        return fail(s, SIM_ERR_ARG, "max_batch must be in [1, %d]", SIM_MAX_BATCH);
    if (tt->num_tables < 1 || tt->max_tiers < 1 || tt->max_tiers > SIM_MAX_TIERS)
        return fail(s, SIM_ERR_ARG, "need num_tables >= 1 and max_tiers in [1, %d]", SIM_MAX_TIERS);
    if (!tt->num_tiers || !tt->headroom_blocks || !tt->replica_table)
        return fail(s, SIM_ERR_ARG, "tier table pointers must not be NULL");
    for (int t = 0; t < tt->num_tables; ++t) {
        const int K = tt->num_tiers[t];
        if (K < 1 || K > tt->max_tiers) return fail(s, SIM_ERR_ARG, "table %d: num_tiers out of range", t);
        long long sum = 0;
        for (int k = 0; k < K; ++k) {
            const int h = tt->headroom_blocks[t * tt->max_tiers + k];
            if (h < 0) return fail(s, SIM_ERR_ARG, "table %d: negative headroom", t);
            sum += h;
        }
        if (cl->blocks_per_instance + sum >= mt::kMaxKeyRange)
            return fail(s, SIM_ERR_ARG, "table %d: M + sum of headroom must be below 2^19", t);
    }
    for (int r = 0; r < cl->num_replicas; ++r)
        if (tt->replica_table[r] < 0 || tt->replica_table[r] >= tt->num_tables)
            return fail(s, SIM_ERR_ARG, "replica %d: table index out of range", r);
    if (pol->policy != SIM_POLICY_LLUMNIX_MT) return fail(s, SIM_ERR_ARG, "unknown policy %d", pol->policy);
    if (pol->enable_migration != 0 && pol->enable_migration != 1)
        return fail(s, SIM_ERR_ARG, "enable_migration must be 0 or 1");
    const long long lim24 = 1LL << 24;
    if (pol->iter_base_us < 1 || pol->iter_base_us > lim24 || pol->iter_us_per_prefill_token < 0 ||
        pol->iter_us_per_prefill_token > lim24 || pol->iter_us_per_decode_seq < 0 || pol->iter_us_per_decode_seq > lim24)
        return fail(s, SIM_ERR_ARG, "iteration-time base must be in [1, 2^24], the other coefficients in [0, 2^24]");
    if (pol->migrate_blocks_per_iter < 1 || pol->migrate_blocks_per_iter > 65535)
        return fail(s, SIM_ERR_ARG, "migrate_blocks_per_iter must be in [1, 65535]");
    if (pol->theta_den < 1 || pol->theta_num < 0 || pol->theta_num > (1 << 20) || pol->theta_den > (1 << 20))
        return fail(s, SIM_ERR_ARG, "theta must be num/den with num in [0, 2^20], den in [1, 2^20]");
    if (pol->event_log_capacity < 0 || pol->event_log_capacity > (1 << 24))
        return fail(s, SIM_ERR_ARG, "event_log_capacity must be in [0, 2^24]");
    if (pol->migrate_interval_us < 1 || pol->migrate_interval_us > (1LL << 31))
        return fail(s, SIM_ERR_ARG, "migrate_interval_us must be in [1, 2^31]");
    if (pol->autoscale != 0 && pol->autoscale != 1) return fail(s, SIM_ERR_ARG, "autoscale must be 0 or 1");
    if (pol->autoscale && (pol->scale_den < 1 || pol->scale_den > 64 || pol->scale_out_num < -4096 ||
                           pol->scale_in_num > 4096 || pol->scale_out_num >= pol->scale_in_num))
        return fail(s, SIM_ERR_ARG,
                    "auto-scaling thresholds must be num/den with den in [1, 64], numerators in [-4096, 4096] "
                    "and scale_out_num < scale_in_num");
    return SIM_OK;
}

}  // namespace

extern "C" {

const char *sim_strerror(int code) {
    switch (code) {
        case SIM_OK: return "ok";
        case SIM_ERR_ARG: return "invalid argument";
        case SIM_ERR_TRACE: return "malformed trace";
        case SIM_ERR_STATE: return "call out of order";
        case SIM_ERR_OOM: return "device allocation failed";
        case SIM_ERR_OVERFLOW: return "32-bit time or counter overflow";
        case SIM_ERR_CUDA: return "CUDA runtime error";
        case SIM_ERR_INTERNAL: return "device-side consistency check failed";
        case SIM_ERR_DEADLOCK: return "no pending event while requests are unfinished";
        case SIM_ERR_UNFINISHED: return "some replica did not finish";
        default: return "unknown error";
    }
}

const char *sim_last_error(const sim_t *s) { return s ? s->err.c_str() : g_create_err.c_str(); }

size_t sim_device_bytes(const sim_t *s) { return s ? s->dev_bytes : 0; }

int sim_launch_info(const sim_t *s, sim_launch_info_t *out) {
    if (!s || !out) return SIM_ERR_ARG;
    const bool ext = s->d_drain != nullptr || s->pol.autoscale != 0;
    out->grid_blocks = ext ? s->launch.grid_ext : s->launch.grid;
    out->block_threads = 32 * mt::kWarpsPerBlock;
    out->blocks_per_sm = ext ? s->launch.per_sm_ext : s->launch.per_sm;
    out->instances_per_lane = s->launch.c;
    out->slots_in_shared = s->launch.sms ? 1 : 0;
    out->extended = ext ? 1 : 0;
    out->shared_bytes = (int64_t)s->launch.smem;
    return SIM_OK;
}

int sim_create(const sim_cluster_t *cl, const sim_tier_table_t *tt, const sim_policy_t *pol, void *cuda_stream,
               const sim_allocator_t *allocator, sim_t **out) {
    if (!out) return fail(nullptr, SIM_ERR_ARG, "out is NULL");
    *out = nullptr;
    int rc = validate_config(nullptr, cl, tt, pol);
    if (rc) return rc;
    if (allocator && (!allocator->alloc || !allocator->free))
        return fail(nullptr, SIM_ERR_ARG, "allocator needs both alloc and free");

    sim_t *s = new (std::nothrow) sim_t();
    if (!s) return fail(nullptr, SIM_ERR_OOM, "host allocation failed");
    s->cl = *cl;
    s->pol = *pol;
    s->K = tt->max_tiers;
    s->ntables = tt->num_tables;
    s->tbl_k.assign(tt->num_tiers, tt->num_tiers + tt->num_tables);
    s->tbl_h.assign(tt->headroom_blocks, tt->headroom_blocks + (size_t)tt->num_tables * tt->max_tiers);
    s->rep_table.assign(tt->replica_table, tt->replica_table + cl->num_replicas);
    s->stream = (cudaStream_t)cuda_stream;
    if (allocator) { s->al = *allocator; s->use_al = true; }
    s->L = mt::make_layout(cl->num_instances, s->K, cl->tokens_per_block);

    const size_t R = (size_t)cl->num_replicas, NB = (size_t)cl->num_instances * cl->max_batch;
    s->d_rep_table = (int *)dalloc(s, R * 4);
    s->d_tbl_k = (int *)dalloc(s, (size_t)s->ntables * 4);
    s->d_tbl_h = (int *)dalloc(s, (size_t)s->ntables * s->K * 4);
    s->d_blobs = (unsigned char *)dalloc(s, R * s->L.bytes);
    s->d_slots = (uint4 *)dalloc(s, R * NB * 16);
    s->d_rep = (mt::RepState *)dalloc(s, R * sizeof(mt::RepState));
    s->d_log = (sim_migration_event_t *)dalloc(s, R * (size_t)pol->event_log_capacity * sizeof(sim_migration_event_t));
    s->d_work = (int *)dalloc(s, 16);
    if (!s->d_rep_table || !s->d_tbl_k || !s->d_tbl_h || !s->d_blobs || !s->d_slots || !s->d_rep ||
        !s->d_log || !s->d_work) {
        const size_t held = s->dev_bytes;
        sim_destroy(s);
        return fail(nullptr, SIM_ERR_OOM, "device allocation failed (%zu bytes held when it failed)", held);
    }
    cudaError_t e = cudaMemcpyAsync(s->d_rep_table, s->rep_table.data(), R * 4, cudaMemcpyHostToDevice, s->stream);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(s->d_tbl_k, s->tbl_k.data(), (size_t)s->ntables * 4, cudaMemcpyHostToDevice, s->stream);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(s->d_tbl_h, s->tbl_h.data(), s->tbl_h.size() * 4, cudaMemcpyHostToDevice, s->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s->stream);  // host vectors may be pageable
    int dev = 0;
    if (e == cudaSuccess) e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&s->sms, cudaDevAttrMultiProcessorCount, dev);
    if (e == cudaSuccess)
        e = mt::plan_launch(cl->num_replicas, cl->num_instances, cl->max_batch, s->L, s->launch);
    if (e != cudaSuccess) {
        cudaGetLastError();
        rc = e == cudaErrorInvalidConfiguration
                 ? fail(nullptr, SIM_ERR_ARG, "per-replica state (%u bytes) does not fit in shared memory", s->L.bytes)
                 : cuda_fail(nullptr, e, "sim_create");
        sim_destroy(s);
        return rc;
    }
    *out = s;
    return SIM_OK;
}

int sim_load_trace(sim_t *s, const int64_t *off, const uint32_t *arrival, const uint16_t *plen, const uint16_t *olen,
                   const uint8_t *tier, int on_device) {
    if (!s) return SIM_ERR_ARG;
    if (!off) return fail(s, SIM_ERR_ARG, "replica_offsets is NULL");
    const int R = s->cl.num_replicas;
    if (off[0] != 0) return fail(s, SIM_ERR_TRACE, "replica_offsets[0] must be 0");
    for (int r = 0; r < R; ++r) {
        const int64_t q = off[r + 1] - off[r];
        if (q < 0) return fail(s, SIM_ERR_TRACE, "replica_offsets must be non-decreasing (replica %d)", r);
        if (q > (int64_t)0xFFFFFFFEll) return fail(s, SIM_ERR_TRACE, "replica %d has more than 2^32-2 records", r);
    }
    const int64_t n = off[R];
    if (n > 0 && (!arrival || !plen || !olen || !tier)) return fail(s, SIM_ERR_ARG, "trace arrays must not be NULL");
    s->loaded = false;
    if (n > s->qcap) {
        dfree(s, s->d_arrival); dfree(s, s->d_plen); dfree(s, s->d_olen); dfree(s, s->d_tier);
        dfree(s, s->d_node); dfree(s, s->d_res);
        s->d_arrival = nullptr; s->d_plen = s->d_olen = nullptr; s->d_tier = nullptr;
        s->d_node = nullptr; s->d_res = nullptr;
        s->qcap = -1;
        const size_t m = (size_t)std::max<int64_t>(n, 1);
        s->d_arrival = (uint32_t *)dalloc(s, m * 4);
        s->d_plen = (uint16_t *)dalloc(s, m * 2);
        s->d_olen = (uint16_t *)dalloc(s, m * 2);
        s->d_tier = (uint8_t *)dalloc(s, m);
        s->d_node = (uint4 *)dalloc(s, m * 16);
        s->d_res = (sim_request_result_t *)dalloc(s, m * 16);
        if (!s->d_arrival || !s->d_plen || !s->d_olen || !s->d_tier || !s->d_node || !s->d_res)
            return fail(s, SIM_ERR_OOM, "device allocation for %lld trace records failed", (long long)n);
        s->qcap = n;
    }
    if (!s->d_off) {
        s->d_off = (long long *)dalloc(s, ((size_t)R + 1) * 8);
        if (!s->d_off) return fail(s, SIM_ERR_OOM, "device allocation failed");
    }
    s->h_off.assign(off, off + R + 1);
    s->lat_nchunks = -1;
    const cudaMemcpyKind kind = on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
    cudaError_t e = cudaMemcpyAsync(s->d_off, s->h_off.data(), ((size_t)R + 1) * 8, cudaMemcpyHostToDevice, s->stream);
    if (n > 0) {
        if (e == cudaSuccess) e = cudaMemcpyAsync(s->d_arrival, arrival, (size_t)n * 4, kind, s->stream);
        if (e == cudaSuccess) e = cudaMemcpyAsync(s->d_plen, plen, (size_t)n * 2, kind, s->stream);
        if (e == cudaSuccess) e = cudaMemcpyAsync(s->d_olen, olen, (size_t)n * 2, kind, s->stream);
        if (e == cudaSuccess) e = cudaMemcpyAsync(s->d_tier, tier, (size_t)n, kind, s->stream);
    }
    if (e == cudaSuccess) e = cudaMemsetAsync(s->d_work, 0, 16, s->stream);
    if (e != cudaSuccess) return cuda_fail(s, e, "sim_load_trace copy");
    s->qtot = n;
    if (n > 0) {
        const long long lim = std::min<long long>((long long)s->cl.blocks_per_instance * s->cl.tokens_per_block, 65536);
        const long long nb = std::min<long long>((n + 255) / 256, (long long)s->sms * 32);
        mt::k_validate<<<(unsigned)std::max<long long>(nb, 1), 256, 0, s->stream>>>(
            s->d_off, R, s->d_arrival, s->d_plen, s->d_olen, s->d_tier, s->d_rep_table, s->d_tbl_k, lim, n,
            s->d_work + 1);
        int rc = check_launch(s, "k_validate");
        if (rc) return rc;
    }
    int flags = 0;
    e = cudaMemcpyAsync(&flags, s->d_work + 1, 4, cudaMemcpyDeviceToHost, s->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s->stream);
    if (e != cudaSuccess) return cuda_fail(s, e, "sim_load_trace validation");
    if (flags) {
        return fail(s, SIM_ERR_TRACE, "malformed trace:%s%s%s%s%s", (flags & 1) ? " unsorted arrivals;" : "",
                    (flags & 2) ? " tier >= K;" : "", (flags & 4) ? " zero prompt or output length;" : "",
                    (flags & 8) ? " prompt + output longer than min(M*T, 65536);" : "",
                    (flags & 16) ? " arrival time 0xFFFFFFFF;" : "");
    }
    int rc = reset_state(s);
    if (rc) return rc;
    s->loaded = true;
    return SIM_OK;
}

int sim_reset(sim_t *s) {
    if (!s) return SIM_ERR_ARG;
    if (!s->loaded) return fail(s, SIM_ERR_STATE, "sim_reset before sim_load_trace");
    return reset_state(s);
}

static_assert(sizeof(sim_latency_stats_t) == 32 + 4 * SIM_HIST_BUCKETS, "sim_latency_stats_t layout");

int sim_latency_stats(sim_t *s, sim_latency_stats_t *out, int on_device) {
    if (!s) return SIM_ERR_ARG;
    if (!out) return fail(s, SIM_ERR_ARG, "out is NULL");
    if (on_device != 0 && on_device != 1) return fail(s, SIM_ERR_ARG, "on_device must be 0 or 1");
    if (!s->loaded) return fail(s, SIM_ERR_STATE, "sim_latency_stats before sim_load_trace");
    const int R = s->cl.num_replicas, KT = s->K;
    const size_t n = (size_t)R * KT * 3;
    sim_latency_stats_t *d = out;
    if (!on_device) {
        if (!s->d_lat) {
            s->d_lat = (sim_latency_stats_t *)dalloc(s, n * sizeof(sim_latency_stats_t));
            if (!s->d_lat) return fail(s, SIM_ERR_OOM, "device allocation of the latency statistics failed");
        }
        d = s->d_lat;
    }
    if (s->lat_nchunks < 0) {  // chunk table of the loaded trace
        std::vector<int> rep;
        std::vector<long long> b0;
        for (int r = 0; r < R; ++r)
            for (long long b = s->h_off[r]; b < s->h_off[r + 1]; b += mtlat::kChunk) {
                rep.push_back(r);
                b0.push_back(b);
            }
        const int nc = (int)rep.size();
        dfree(s, s->d_lat_rep);
        dfree(s, s->d_lat_b0);
        s->d_lat_rep = nullptr;
        s->d_lat_b0 = nullptr;
        if (nc > 0) {
            s->d_lat_rep = (int *)dalloc(s, (size_t)nc * 4);
            s->d_lat_b0 = (long long *)dalloc(s, (size_t)nc * 8);
            if (!s->d_lat_rep || !s->d_lat_b0) return fail(s, SIM_ERR_OOM, "device allocation of the chunk table failed");
            cudaError_t e = cudaMemcpyAsync(s->d_lat_rep, rep.data(), (size_t)nc * 4, cudaMemcpyHostToDevice, s->stream);
            if (e == cudaSuccess)
                e = cudaMemcpyAsync(s->d_lat_b0, b0.data(), (size_t)nc * 8, cudaMemcpyHostToDevice, s->stream);
            if (e == cudaSuccess) e = cudaStreamSynchronize(s->stream);  // the host vectors go out of scope
            if (e != cudaSuccess) return cuda_fail(s, e, "sim_latency_stats chunk table");
        }
        s->lat_nchunks = nc;
    }
    if (!s->d_lat_sel) {
        s->d_lat_sel = (uint4 *)dalloc(s, mtlat::select_state_bytes((long long)n));
        s->d_lat_bins = (uint32_t *)dalloc(s, mtlat::select_bin_bytes((long long)n));
        if (!s->d_lat_sel || !s->d_lat_bins)
            return fail(s, SIM_ERR_OOM, "device allocation of the percentile selection scratch failed");
    }
    cudaError_t e = mtlat::launch(s->d_lat_rep, s->d_lat_b0, s->lat_nchunks, s->d_off, KT, s->d_arrival, s->d_olen,
                                  s->d_tier, s->d_res, d, (long long)n, s->d_lat_sel, s->d_lat_bins, s->sms,
                                  s->stream);
    if (e != cudaSuccess) return cuda_fail(s, e, "sim_latency_stats");
    if (!on_device) {
        e = cudaMemcpyAsync(out, d, n * sizeof(sim_latency_stats_t), cudaMemcpyDeviceToHost, s->stream);
        if (e == cudaSuccess) e = cudaStreamSynchronize(s->stream);
        if (e != cudaSuccess) return cuda_fail(s, e, "sim_latency_stats copy");
    }
    return SIM_OK;
}

int sim_set_drain(sim_t *s, const uint32_t *drain_start_us, int on_device) {
    if (!s) return SIM_ERR_ARG;
    if (on_device != 0 && on_device != 1) return fail(s, SIM_ERR_ARG, "on_device must be 0 or 1");
    if (!drain_start_us) {
        dfree(s, s->d_drain);
        s->d_drain = nullptr;
        return SIM_OK;
    }
    const size_t bytes = (size_t)s->cl.num_replicas * (size_t)s->cl.num_instances * 4u;
    if (!s->d_drain) {
        s->d_drain = (uint32_t *)dalloc(s, bytes);
        if (!s->d_drain) return fail(s, SIM_ERR_OOM, "device allocation of the drain schedule failed");
    }
    cudaError_t e = cudaMemcpyAsync(s->d_drain, drain_start_us, bytes,
                                    on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice, s->stream);
    if (e == cudaSuccess && !on_device) e = cudaStreamSynchronize(s->stream);  // the host buffer may be reused
    if (e != cudaSuccess) return cuda_fail(s, e, "sim_set_drain copy");
    return SIM_OK;
}

int sim_set_headroom(sim_t *s, const int32_t *headroom_blocks) {
    if (!s) return SIM_ERR_ARG;
    if (!headroom_blocks) return fail(s, SIM_ERR_ARG, "headroom_blocks is NULL");
    const int K = s->K;
    for (int t = 0; t < s->ntables; ++t) {
        long long sum = 0;
        for (int k = 0; k < s->tbl_k[t]; ++k) {
            const int h = headroom_blocks[(size_t)t * K + k];
            if (h < 0) return fail(s, SIM_ERR_ARG, "table %d: negative headroom", t);
            sum += h;
        }
        if (s->cl.blocks_per_instance + sum >= mt::kMaxKeyRange)
            return fail(s, SIM_ERR_ARG, "table %d: M + sum of headroom must be below 2^19", t);
    }
    for (int t = 0; t < s->ntables; ++t)
        for (int k = 0; k < K; ++k)
            s->tbl_h[(size_t)t * K + k] = k < s->tbl_k[t] ? headroom_blocks[(size_t)t * K + k] : 0;
    cudaError_t e = cudaMemcpyAsync(s->d_tbl_h, s->tbl_h.data(), s->tbl_h.size() * 4, cudaMemcpyHostToDevice, s->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s->stream);  // the host vector may change at the next call
    if (e != cudaSuccess) return cuda_fail(s, e, "sim_set_headroom copy");
    if (s->loaded) {
        mt::Params p = make_params(s, 0);
        const int R = s->cl.num_replicas;
        mt::k_set_headroom<<<(R + 7) / 8, 256, 0, s->stream>>>(p, s->d_rep_table, s->d_tbl_k, s->d_tbl_h);
        return check_launch(s, "k_set_headroom");
    }
    return SIM_OK;
}

int sim_set_order(sim_t *s, const int32_t *order) {
    if (!s) return SIM_ERR_ARG;
    if (!order) {
        dfree(s, s->d_order);
        s->d_order = nullptr;
        return SIM_OK;
    }
    const int R = s->cl.num_replicas;
    std::vector<char> seen((size_t)R, 0);
    for (int k = 0; k < R; ++k) {
        const int32_t r = order[k];
        if (r < 0 || r >= R || seen[(size_t)r])
            return fail(s, SIM_ERR_ARG, "order is not a permutation of 0..%d (entry %d = %d)", R - 1, k, (int)r);
        seen[(size_t)r] = 1;
    }
    if (!s->d_order) {
        s->d_order = (int *)dalloc(s, (size_t)R * 4);
        if (!s->d_order) return fail(s, SIM_ERR_OOM, "device allocation of the replica order failed");
    }
    cudaError_t e = cudaMemcpyAsync(s->d_order, order, (size_t)R * 4, cudaMemcpyHostToDevice, s->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s->stream);  // the host buffer may be reused
    if (e != cudaSuccess) return cuda_fail(s, e, "sim_set_order copy");
    return SIM_OK;
}

int sim_run(sim_t *s, int64_t max_steps, int64_t *num_unfinished) {
    if (!s) return SIM_ERR_ARG;
    if (!s->loaded) return fail(s, SIM_ERR_STATE, "sim_run before sim_load_trace");
    if (max_steps < 1) return fail(s, SIM_ERR_ARG, "max_steps_per_replica must be >= 1");
    cudaError_t e = cudaMemsetAsync(s->d_work, 0, 4, s->stream);
    if (e != cudaSuccess) return cuda_fail(s, e, "sim_run");
    mt::Params p = make_params(s, (long long)max_steps);
    if (p.drains || p.autoscale)
        s->launch.fn_ext<<<s->launch.grid_ext, 32 * mt::kWarpsPerBlock, s->launch.smem, s->stream>>>(p);
    else
        s->launch.fn<<<s->launch.grid, 32 * mt::kWarpsPerBlock, s->launch.smem, s->stream>>>(p);
    int rc = check_launch(s, "k_run");
    if (rc) return rc;
    if (num_unfinished) {
        int cnt = 0;
        e = cudaMemsetAsync(s->d_work + 2, 0, 4, s->stream);
        if (e != cudaSuccess) return cuda_fail(s, e, "sim_run");
        const int R = s->cl.num_replicas;
        mt::k_export_stats<<<(R + 255) / 256, 256, 0, s->stream>>>(s->d_rep, nullptr, R, s->d_work + 2, nullptr);
        rc = check_launch(s, "k_export_stats");
        if (rc) return rc;
        e = cudaMemcpyAsync(&cnt, s->d_work + 2, 4, cudaMemcpyDeviceToHost, s->stream);
        if (e == cudaSuccess) e = cudaStreamSynchronize(s->stream);
        if (e != cudaSuccess) return cuda_fail(s, e, "sim_run");
        *num_unfinished = cnt;
    }
    return SIM_OK;
}

int sim_metrics(sim_t *s, sim_request_result_t *per_request, sim_replica_stats_t *per_replica,
                sim_migration_event_t *events, int on_device) {
    if (!s) return SIM_ERR_ARG;
    if (!s->loaded) return fail(s, SIM_ERR_STATE, "sim_metrics before sim_load_trace");
    const cudaMemcpyKind kind = on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost;
    const int R = s->cl.num_replicas;
    cudaError_t e = cudaSuccess;
    if (per_request && s->qtot > 0)
        e = cudaMemcpyAsync(per_request, s->d_res, (size_t)s->qtot * sizeof(sim_request_result_t), kind, s->stream);
    if (e == cudaSuccess && per_replica) {
        sim_replica_stats_t *dst = per_replica;
        sim_replica_stats_t *tmp = nullptr;
        if (!on_device) {
            tmp = (sim_replica_stats_t *)dalloc(s, (size_t)R * sizeof(sim_replica_stats_t));
            if (!tmp) return fail(s, SIM_ERR_OOM, "device allocation failed");
            dst = tmp;
        }
        if (!s->d_ftc) {
            s->d_ftc = (uint32_t *)dalloc(s, (size_t)R * 4);
            if (!s->d_ftc) return fail(s, SIM_ERR_OOM, "device allocation failed");
        }
        mt::k_first_tokens<<<std::max(1, std::min(R, s->sms * 8)), 256, 0, s->stream>>>(s->d_off, R, s->d_res, s->d_ftc);
        int rc = check_launch(s, "k_first_tokens");
        if (rc) return rc;
        mt::k_export_stats<<<(R + 255) / 256, 256, 0, s->stream>>>(s->d_rep, dst, R, nullptr, s->d_ftc);
        rc = check_launch(s, "k_export_stats");
        if (rc) return rc;
        if (tmp) {
            e = cudaMemcpyAsync(per_replica, tmp, (size_t)R * sizeof(sim_replica_stats_t), cudaMemcpyDeviceToHost,
                                s->stream);
            if (e == cudaSuccess) e = cudaStreamSynchronize(s->stream);
            dfree(s, tmp);
        }
    }
    if (e == cudaSuccess && events && s->pol.event_log_capacity > 0)
        e = cudaMemcpyAsync(events, s->d_log, (size_t)R * s->pol.event_log_capacity * sizeof(sim_migration_event_t),
                            kind, s->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s->stream);
    if (e != cudaSuccess) return cuda_fail(s, e, "sim_metrics");
    return SIM_OK;
}

void sim_destroy(sim_t *s) {
    if (!s) return;
    cudaStreamSynchronize(s->stream);
    while (!s->bufs.empty()) dfree(s, s->bufs.back().p);
    cudaStreamSynchronize(s->stream);
    cudaGetLastError();
    delete s;
}

}  // extern "C"

// ============================================================================
// Allocation-free entry point: the whole simulation state in one file-scope
// device array (see sim_run_static in mtsim.h).
// ============================================================================
static __device__ __align__(256) unsigned char g_static_scratch[SIM_STATIC_SCRATCH_BYTES];

namespace {

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

}  // namespace

extern "C" int sim_run_static(const sim_cluster_t *cl, const sim_tier_table_t *tt, const sim_policy_t *pol,
                              const int64_t *off, const uint32_t *arrival, const uint16_t *plen,
                              const uint16_t *olen, const uint8_t *tier, sim_request_result_t *per_request,
                              sim_replica_stats_t *per_replica, sim_migration_event_t *events, void *cuda_stream) {
    int rc = validate_config(nullptr, cl, tt, pol);
    if (rc) return rc;
    if (!off) return fail(nullptr, SIM_ERR_ARG, "replica_offsets is NULL");
    const int R = cl->num_replicas;
    if (off[0] != 0) return fail(nullptr, SIM_ERR_TRACE, "replica_offsets[0] must be 0");
    for (int r = 0; r < R; ++r) {
        const int64_t q = off[r + 1] - off[r];
        if (q < 0 || q > (int64_t)0xFFFFFFFEll)
            return fail(nullptr, SIM_ERR_TRACE, "replica_offsets invalid at replica %d", r);
    }
    const int64_t n = off[R];
    if (n > 0 && (!arrival || !plen || !olen || !tier || !per_request))
        return fail(nullptr, SIM_ERR_ARG, "trace and per_request pointers must not be NULL");
    if (!per_replica) return fail(nullptr, SIM_ERR_ARG, "per_replica must not be NULL");
    const int cap = events ? pol->event_log_capacity : 0;

    // Carve the scratch array.
    const int N = cl->num_instances, K = tt->max_tiers;
    const mt::Layout L = mt::make_layout(N, K, cl->tokens_per_block);
    size_t o = 0;
    const size_t o_blobs = o; o = align256(o + (size_t)R * L.bytes);
    const size_t o_slots = o; o = align256(o + (size_t)R * N * cl->max_batch * 16);
    const size_t o_rep = o; o = align256(o + (size_t)R * sizeof(mt::RepState));
    const size_t o_node = o; o = align256(o + (size_t)n * 16);
    const size_t o_off = o; o = align256(o + ((size_t)R + 1) * 8);
    const size_t o_rt = o; o = align256(o + (size_t)R * 4);
    const size_t o_tk = o; o = align256(o + (size_t)tt->num_tables * 4);
    const size_t o_th = o; o = align256(o + (size_t)tt->num_tables * K * 4);
    const size_t o_work = o; o = align256(o + 16);
    const size_t o_ftc = o; o = align256(o + (size_t)R * 4);
    if (o > (size_t)SIM_STATIC_SCRATCH_BYTES)
        return fail(nullptr, SIM_ERR_ARG, "problem needs %zu bytes of scratch; sim_run_static holds %u bytes", o,
                    (unsigned)SIM_STATIC_SCRATCH_BYTES);

    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail(nullptr, SIM_ERR_CUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
    // The array's device address on the current device, looked up on every
    // call: a cached address would be stale after a cudaDeviceReset (the
    // module is loaded again), and nothing shared is written here.
    void *scratch = nullptr;
    e = cudaGetSymbolAddress(&scratch, g_static_scratch);
    if (e != cudaSuccess || !scratch)
        return fail(nullptr, SIM_ERR_CUDA, "cudaGetSymbolAddress: %s", cudaGetErrorString(e));
    unsigned char *base = (unsigned char *)scratch;
    cudaStream_t st = (cudaStream_t)cuda_stream;

    mt::Launch lc;
    e = mt::plan_launch(R, N, cl->max_batch, L, lc);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return e == cudaErrorInvalidConfiguration
                   ? fail(nullptr, SIM_ERR_ARG, "per-replica state does not fit in shared memory")
                   : fail(nullptr, SIM_ERR_CUDA, "sim_run_static launch set-up: %s", cudaGetErrorString(e));
    }
    mt::Params p;
    memset(&p, 0, sizeof p);
    fill_scalars(p, *cl, *pol, K, cap, L, 1LL << 62);
    p.offsets = (const long long *)(base + o_off);
    p.arrival = arrival;
    p.plen = plen;
    p.olen = olen;
    p.tier = tier;
    p.node = (uint4 *)(base + o_node);
    p.res = per_request;
    p.blobs = base + o_blobs;
    p.slots = (uint4 *)(base + o_slots);
    p.rep = (mt::RepState *)(base + o_rep);
    p.log = events;
    p.work = (int *)(base + o_work);
    int *rt = (int *)(base + o_rt), *tk = (int *)(base + o_tk), *th = (int *)(base + o_th);

    // Inputs the kernels read from device memory; the work counter and flags start at zero.
    e = cudaMemcpyAsync((void *)p.offsets, off, ((size_t)R + 1) * 8, cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(rt, tt->replica_table, (size_t)R * 4, cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(tk, tt->num_tiers, (size_t)tt->num_tables * 4, cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(th, tt->headroom_blocks, (size_t)tt->num_tables * K * 4, cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess) e = cudaMemsetAsync(p.work, 0, 16, st);
    if (e != cudaSuccess) return fail(nullptr, SIM_ERR_CUDA, "sim_run_static copy: %s", cudaGetErrorString(e));
    int sms = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return fail(nullptr, SIM_ERR_CUDA, "sim_run_static: %s", cudaGetErrorString(e));
    if (n > 0) {
        const long long lim = std::min<long long>((long long)p.M * p.T, 65536);
        const long long nb = std::min<long long>((n + 255) / 256, (long long)sms * 32);
        mt::k_validate<<<(unsigned)std::max<long long>(nb, 1), 256, 0, st>>>(p.offsets, R, arrival, plen, olen, tier,
                                                                              rt, tk, lim, n, p.work + 1);
        int flags = 0;
        e = cudaGetLastError();
        if (e == cudaSuccess) e = cudaMemcpyAsync(&flags, p.work + 1, 4, cudaMemcpyDeviceToHost, st);
        if (e == cudaSuccess) e = cudaStreamSynchronize(st);
        if (e != cudaSuccess)
            return fail(nullptr, SIM_ERR_CUDA, "sim_run_static validation: %s", cudaGetErrorString(e));
        if (flags) return fail(nullptr, SIM_ERR_TRACE, "malformed trace (validation flags 0x%x)", flags);
    }
    mt::k_init_state<<<(R + 7) / 8, 256, 0, st>>>(p, rt, tk, th);
    if (n > 0) {
        const long long nb = std::min<long long>((n + 255) / 256, 65535LL * 16);
        mt::k_init_requests<<<(unsigned)nb, 256, 0, st>>>(per_request, (long long)n);
    }
    if (p.autoscale)
        lc.fn_ext<<<lc.grid_ext, 32 * mt::kWarpsPerBlock, lc.smem, st>>>(p);
    else
        lc.fn<<<lc.grid, 32 * mt::kWarpsPerBlock, lc.smem, st>>>(p);
    uint32_t *ftc = (uint32_t *)(base + o_ftc);
    mt::k_first_tokens<<<std::max(1, std::min(R, sms * 8)), 256, 0, st>>>(p.offsets, R, per_request, ftc);
    // work[2] (zeroed above) counts the replicas that did not finish
    mt::k_export_stats<<<(R + 255) / 256, 256, 0, st>>>(p.rep, per_replica, R, p.work + 2, ftc);
    int unfinished = 0;
    e = cudaGetLastError();
    if (e == cudaSuccess) e = cudaMemcpyAsync(&unfinished, p.work + 2, 4, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return fail(nullptr, SIM_ERR_CUDA, "sim_run_static: %s", cudaGetErrorString(e));
    if (unfinished > 0)
        return fail(nullptr, SIM_ERR_UNFINISHED, "%d of %d replicas did not finish; see per_replica[r].status",
                    unfinished, R);
    return SIM_OK;
}
