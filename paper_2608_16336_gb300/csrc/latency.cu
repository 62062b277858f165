// latency.cu -- per-tier latency statistics of simulated requests (the
// measures the paper reports per priority tier, Sec. 5.1 and Sec. 5.3: TTFT,
// time between tokens and end-to-end latency, their means and P50 / P90 /
// P99), computed on the GPU from the simulation's per-request results.
#include "latency.cuh"

#include <algorithm>

namespace mtlat {
namespace {

constexpr uint32_t kNone = 0xFFFFFFFFu;
constexpr uint32_t kFull = 0xFFFFFFFFu;

// Histogram bucket of a 32-bit value: v for v < 8, else eight equal buckets per
// power of two: with e = floor(log2 v), 8 + 8 (e - 3) + (v >> (e - 3)) - 8.
__device__ __forceinline__ uint32_t lat_bucket(uint32_t v) {
    // with e clamped to at least 3 the same expression gives v for v < 8 (clz(0) = 32)
    const uint32_t e = (uint32_t)max(31 - __clz(v), 3);
    return 8u * (e - 3u) + (v >> (e - 3u));
}
// Smallest value of bucket b.
__device__ __forceinline__ uint32_t lat_floor(uint32_t b) {
    if (b < 8u) return b;
    const uint32_t e = (b - 8u) / 8u + 3u;
    return (8u + (b - 8u) % 8u) << (e - 3u);
}

// Per-tier latency histograms, sums and maxima.  The requests are cut into
// chunks of at most kChunk within one replica (chunk_rep / chunk_b0); a
// block streams one chunk (grid-stride over chunks).  Shared memory holds the
// chunk's histogram [G][SIM_HIST_BUCKETS] and, per thread, an exact sum and a
// maximum for every (tier, measure) group, [G][blockDim.x] each, so a request
// updates only its own group: one histogram atomic, one 64-bit add and one
// maximum per measure.  At the end of the chunk each warp folds the threads'
// sums and maxima of some groups and the block merges everything into out[r]
// with global atomics (non-empty buckets only).  out must be zero on entry.
// Measures: TTFT = first - arrival, TBT = floor((finish - first) / (O - 1))
// for O >= 2, E2E = finish - arrival, over finished requests.
__global__ void k_latency_hist(const int *chunk_rep, const long long *chunk_b0, int nchunks,
                               const long long *offsets, int KT, const uint32_t *arrival, const uint16_t *olen,
                               const uint8_t *tier, const sim_request_result_t *res, sim_latency_stats_t *out) {
    extern __shared__ __align__(16) unsigned char lsm[];
    const int G = KT * 3;  // groups (tier, measure)
    const int B = (int)blockDim.x;
    unsigned long long *ssum = reinterpret_cast<unsigned long long *>(lsm);  // [G][B]
    uint32_t *smax = reinterpret_cast<uint32_t *>(ssum + (size_t)G * B);      // [G][B]
    uint32_t *hist = smax + (size_t)G * B;                                    // [G][SIM_HIST_BUCKETS]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = B >> 5;
    for (int c = blockIdx.x; c < nchunks; c += gridDim.x) {
        const int r = chunk_rep[c];
        const long long b0 = chunk_b0[c];
        const uint32_t nrec = (uint32_t)(min(b0 + (long long)kChunk, offsets[r + 1]) - b0);
        for (int q = threadIdx.x; q < G * SIM_HIST_BUCKETS; q += B) hist[q] = 0;
        for (int g = 0; g < G; ++g) {
            ssum[g * B + threadIdx.x] = 0;
            smax[g * B + threadIdx.x] = 0;
        }
        __syncthreads();
        const uint4 *rs = reinterpret_cast<const uint4 *>(res + b0);
        const uint32_t *ar = arrival + b0;
        const uint16_t *ol = olen + b0;
        const uint8_t *tr = tier + b0;
        constexpr int U = 4;  // requests per thread per pass: their loads are issued together
        for (uint32_t q0 = threadIdx.x; q0 < nrec; q0 += (uint32_t)(U * B)) {
            uint4 rv[U];
            uint32_t a[U], o[U], k[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const uint32_t q = q0 + (uint32_t)(u * B);
                const bool in = q < nrec;
                rv[u] = in ? rs[q] : make_uint4(0, 0, kNone, 0);
                a[u] = in ? ar[q] : 0u;
                o[u] = in ? (uint32_t)ol[q] : 0u;
                k[u] = in ? (uint32_t)tr[q] : 0u;
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const uint32_t first = rv[u].y, fin = rv[u].z;
                if (fin == kNone || k[u] >= (uint32_t)KT) continue;
                const bool has_tbt = o[u] >= 2u;
                uint32_t v[3];
                v[0] = first - a[u];
                v[1] = has_tbt ? (fin - first) / (o[u] - 1u) : 0u;
                v[2] = fin - a[u];
#pragma unroll
                for (int m = 0; m < 3; ++m) {
                    if (m == 1 && !has_tbt) continue;  // a one-token request has no TBT
                    const int g = (int)k[u] * 3 + m;
                    atomicAdd(&hist[g * SIM_HIST_BUCKETS + lat_bucket(v[m])], 1u);
                    const int at = g * B + (int)threadIdx.x;
                    ssum[at] += v[m];
                    smax[at] = max(smax[at], v[m]);
                }
            }
        }
        __syncthreads();
        // the threads' sums and maxima: warp w folds groups w, w + nwarps, ...
        sim_latency_stats_t *orow = out + (size_t)r * G;
        for (int g = warp; g < G; g += nwarps) {
            unsigned long long sv = 0;
            uint32_t mv = 0;
            for (int t = lane; t < B; t += 32) {
                sv += ssum[g * B + t];
                mv = max(mv, smax[g * B + t]);
            }
#pragma unroll
            for (int sh = 16; sh > 0; sh >>= 1) sv += __shfl_xor_sync(kFull, sv, sh);
            mv = __reduce_max_sync(kFull, mv);
            if (lane == 0 && sv) atomicAdd(reinterpret_cast<unsigned long long *>(&orow[g].sum_us), sv);
            if (lane == 0 && mv) atomicMax(&orow[g].max_us, mv);
        }
        for (int q = threadIdx.x; q < G * SIM_HIST_BUCKETS; q += B) {
            const uint32_t h = hist[q];
            if (h) atomicAdd(&orow[q / SIM_HIST_BUCKETS].hist[q % SIM_HIST_BUCKETS], h);
        }
        __syncthreads();
    }
}

__device__ __forceinline__ uint32_t *pct_field(sim_latency_stats_t *o, int q) {
    return q == 0 ? &o->p50_us : (q == 1 ? &o->p90_us : &o->p99_us);
}

// Bit width of bucket b: values of bucket b are [lat_floor(b), lat_floor(b) + 2^w).
__device__ __forceinline__ uint32_t lat_width_bits(uint32_t b) { return b < 8u ? 0u : (b - 8u) / 8u; }

// Counts and the start of the nearest-rank P50 / P90 / P99 selection: one warp
// per (replica, tier, measure).  The value of rank ceil(p n / 100) lies in the
// bucket where the merged histogram's running count reaches that rank; the
// selection state of percentile q is {floor of that bucket, its width in
// bits, the rank among the values of the bucket}.  A bucket one value wide
// gives the value at once; the others are narrowed by the selection passes.
__global__ void k_latency_pct(long long ngroups, sim_latency_stats_t *out, uint4 *sel) {
    const int lane = threadIdx.x & 31;
    const long long warps = ((long long)gridDim.x * blockDim.x) >> 5;
    for (long long g = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5; g < ngroups; g += warps) {
        sim_latency_stats_t *o = out + g;
        // lane l holds buckets [8 l, 8 l + 8) (240 = 30 lanes x 8)
        uint32_t c[8], own = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int bj = lane * 8 + j;
            c[j] = bj < SIM_HIST_BUCKETS ? o->hist[bj] : 0u;
            own += c[j];
        }
        uint32_t incl = own;
#pragma unroll
        for (int sh = 1; sh < 32; sh <<= 1) {
            const uint32_t y = __shfl_up_sync(kFull, incl, sh);
            if (lane >= sh) incl += y;
        }
        const uint32_t n = __shfl_sync(kFull, incl, 31);
        const uint32_t excl = incl - own;
        const uint32_t pct[3] = {50u, 90u, 99u};
#pragma unroll
        for (int q = 0; q < 3; ++q) {
            const uint32_t rank = n ? max(1u, (uint32_t)(((unsigned long long)pct[q] * n + 99u) / 100u)) : 0u;
            uint4 st = make_uint4(0u, 0u, 0u, 0u);  // {low end, width bits, rank in the bucket, -}
            const bool mine = n && excl < rank && rank <= incl;
            if (mine) {
                uint32_t cum = excl;
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    if (st.z == 0u && cum + c[j] >= rank) {
                        const uint32_t bj = (uint32_t)(lane * 8 + j);
                        st = make_uint4(lat_floor(bj), lat_width_bits(bj), rank - cum, 0u);
                    }
                    cum += c[j];
                }
            }
            const uint32_t who = __ballot_sync(kFull, mine);
            const int src = who ? __ffs(who) - 1 : 0;
            st.x = __shfl_sync(kFull, st.x, src);
            st.y = __shfl_sync(kFull, st.y, src);
            st.z = __shfl_sync(kFull, st.z, src);
            if (lane == 0) {
                if (!n) st = make_uint4(0u, 0u, 0u, 0u);
                sel[g * 3 + q] = st;
                *pct_field(o, q) = st.x;  // final when the bucket is one value wide
            }
        }
        if (lane == 0) o->count = n;
    }
}

// One selection pass: every finished request of every chunk adds, for each
// percentile whose current range [lo, lo + 2^w) (w > 0) holds its value v,
// one to bin (v - lo) >> max(w - 8, 0) of that (group, percentile).  A
// block loads its replica's selection states into shared memory and skips a
// chunk whose replica has nothing left to narrow.
__global__ void k_latency_refine(const int *chunk_rep, const long long *chunk_b0, int nchunks,
                                 const long long *offsets, int KT, const uint32_t *arrival, const uint16_t *olen,
                                 const uint8_t *tier, const sim_request_result_t *res, const uint4 *sel,
                                 uint32_t *bins) {
    extern __shared__ __align__(16) unsigned char rsm[];
    uint4 *ss = reinterpret_cast<uint4 *>(rsm);  // [KT * 3 measures * 3 percentiles]
    const int G = KT * 3, S = G * 3;
    for (int c = blockIdx.x; c < nchunks; c += gridDim.x) {
        const int r = chunk_rep[c];
        const long long b0 = chunk_b0[c];
        int open = 0;
        for (int t = threadIdx.x; t < S; t += blockDim.x) {
            const uint4 st = sel[(size_t)r * S + t];
            ss[t] = st;
            open |= st.y != 0u;
        }
        if (!__syncthreads_or(open)) continue;  // uniform: every thread took part
        const uint32_t nrec = (uint32_t)(min(b0 + (long long)kChunk, offsets[r + 1]) - b0);
        uint32_t *rbins = bins + (size_t)r * S * kSelBins;
        for (uint32_t q = threadIdx.x; q < nrec; q += blockDim.x) {
            const uint4 rv = reinterpret_cast<const uint4 *>(res + b0)[q];
            const uint32_t first = rv.y, fin = rv.z, k = tier[b0 + q];
            if (fin == kNone || k >= (uint32_t)KT) continue;
            const uint32_t a = arrival[b0 + q], o = olen[b0 + q];
            uint32_t v[3];
            v[0] = first - a;
            v[1] = o >= 2u ? (fin - first) / (o - 1u) : 0u;
            v[2] = fin - a;
#pragma unroll
            for (int m = 0; m < 3; ++m) {
                if (m == 1 && o < 2u) continue;  // a one-token request has no TBT
                const int g = (int)k * 3 + m;
#pragma unroll
                for (int p = 0; p < 3; ++p) {
                    const uint4 st = ss[g * 3 + p];
                    if (st.y == 0u || v[m] - st.x >= (1u << st.y)) continue;
                    const uint32_t sh = st.y > 8u ? st.y - 8u : 0u;
                    atomicAdd(&rbins[(size_t)(g * 3 + p) * kSelBins + ((v[m] - st.x) >> sh)], 1u);
                }
            }
        }
        __syncthreads();
    }
}

// Closes a selection pass: one warp per (group, percentile) still open reads
// its bins, finds the bin where the running count reaches the rank, narrows
// the range to that bin (rank taken relative to it) and clears the bins for
// the next pass.  A range one value wide is the exact percentile.
__global__ void k_latency_step(long long nstates, uint4 *sel, uint32_t *bins, sim_latency_stats_t *out) {
    const int lane = threadIdx.x & 31;
    const long long warps = ((long long)gridDim.x * blockDim.x) >> 5;
    for (long long i = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5; i < nstates; i += warps) {
        const uint4 st = sel[i];
        if (st.y == 0u) continue;
        uint32_t *bn = bins + (size_t)i * kSelBins;
        uint32_t c[8], own = 0;  // lane l holds bins [8 l, 8 l + 8)
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            c[j] = bn[lane * 8 + j];
            own += c[j];
        }
        uint32_t incl = own;
#pragma unroll
        for (int sh = 1; sh < 32; sh <<= 1) {
            const uint32_t y = __shfl_up_sync(kFull, incl, sh);
            if (lane >= sh) incl += y;
        }
        const uint32_t excl = incl - own;
        const bool mine = excl < st.z && st.z <= incl;
        uint32_t dig = 0, below = 0;
        if (mine) {
            uint32_t cum = excl;
            bool got = false;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                if (!got && cum + c[j] >= st.z) { got = true; dig = (uint32_t)(lane * 8 + j); below = cum; }
                cum += c[j];
            }
        }
        const uint32_t who = __ballot_sync(kFull, mine);
#pragma unroll
        for (int j = 0; j < 8; ++j) bn[lane * 8 + j] = 0u;
        if (!who) {  // counts and rank disagree: stop here (the result keeps the range's low end)
            if (lane == 0) sel[i].y = 0u;
            continue;
        }
        dig = __shfl_sync(kFull, dig, __ffs(who) - 1);
        below = __shfl_sync(kFull, below, __ffs(who) - 1);
        if (lane == 0) {
            const uint32_t sh = st.y > 8u ? st.y - 8u : 0u;
            const uint4 nx = make_uint4(st.x + (dig << sh), sh, st.z - below, 0u);
            sel[i] = nx;
            if (sh == 0u) *pct_field(out + i / 3, (int)(i % 3)) = nx.x;
        }
    }
}

}  // namespace

cudaError_t launch(const int *chunk_rep, const long long *chunk_b0, int nchunks, const long long *offsets, int KT,
                   const uint32_t *arrival, const uint16_t *olen, const uint8_t *tier,
                   const sim_request_result_t *res, sim_latency_stats_t *out, long long ngroups, uint4 *sel,
                   uint32_t *bins, int sms, cudaStream_t stream) {
    cudaError_t e = cudaMemsetAsync(out, 0, (size_t)ngroups * sizeof(sim_latency_stats_t), stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(bins, 0, select_bin_bytes(ngroups), stream);
    if (e != cudaSuccess) return e;
    const int grid = std::max(1, std::min(nchunks, sms * 16));
    if (nchunks > 0) {
        // threads per block: 256 up to 4 tiers, else 128 (the per-thread
        // accumulators take 12 bytes per thread and group)
        const int threads = KT <= 4 ? 256 : 128;
        const size_t smem = (size_t)KT * 3 * (12u * (size_t)threads + 4u * SIM_HIST_BUCKETS);  // <= 119,808 bytes
        if (smem > 48 * 1024) {
            e = cudaFuncSetAttribute(k_latency_hist, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return e;
        }
        k_latency_hist<<<grid, threads, smem, stream>>>(chunk_rep, chunk_b0, nchunks, offsets, KT, arrival, olen, tier,
                                                        res, out);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    const long long nb = std::min<long long>((ngroups + 7) / 8, (long long)sms * 32);
    k_latency_pct<<<(unsigned)std::max<long long>(nb, 1), 256, 0, stream>>>(ngroups, out, sel);
    e = cudaGetLastError();
    if (e != cudaSuccess || nchunks == 0) return e;
    // a bucket spans at most 2^28 values (32-bit values, eight buckets per
    // power of two): four passes of 8 bits reach a single value
    const long long nstates = ngroups * 3;
    const long long nbs = std::min<long long>((nstates + 7) / 8, (long long)sms * 32);
    const size_t rsmem = (size_t)KT * 9u * 16u;
    for (int pass = 0; pass < 4; ++pass) {
        k_latency_refine<<<grid, 256, rsmem, stream>>>(chunk_rep, chunk_b0, nchunks, offsets, KT, arrival, olen, tier,
                                                      res, sel, bins);
        k_latency_step<<<(unsigned)std::max<long long>(nbs, 1), 256, 0, stream>>>(nstates, sel, bins, out);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace mtlat
