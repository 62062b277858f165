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
// block streams one chunk (grid-stride over chunks), histograms it in shared
// memory while every lane keeps its own exact sums and maxima per (tier,
// measure) in registers (KM >= the number of tiers, a compile-time bound so
// the accumulators stay in registers), and merges them into out[r] with
// global atomics (non-empty buckets only).  out must be zero on entry.
// Measures: TTFT = first - arrival, TBT = floor((finish - first) / (O - 1))
// for O >= 2, E2E = finish - arrival, over finished requests.
template <int KM>
__global__ void __launch_bounds__(256) k_latency_hist(const int *chunk_rep, const long long *chunk_b0, int nchunks,
                                                      const long long *offsets, int KT, const uint32_t *arrival,
                                                      const uint16_t *olen, const uint8_t *tier,
                                                      const sim_request_result_t *res, sim_latency_stats_t *out) {
    extern __shared__ __align__(16) unsigned char lsm[];
    const int G = KT * 3;                                  // groups (tier, measure)
    uint32_t *hist = reinterpret_cast<uint32_t *>(lsm);    // [G][SIM_HIST_BUCKETS]
    const int lane = threadIdx.x & 31;
    for (int c = blockIdx.x; c < nchunks; c += gridDim.x) {
        const int r = chunk_rep[c];
        const long long b0 = chunk_b0[c], b1 = min(b0 + (long long)kChunk, offsets[r + 1]);
        for (int q = threadIdx.x; q < G * SIM_HIST_BUCKETS; q += blockDim.x) hist[q] = 0;
        unsigned long long acc[KM][3];
        uint32_t amx[KM][3];
#pragma unroll
        for (int kk = 0; kk < KM; ++kk)
#pragma unroll
            for (int m = 0; m < 3; ++m) { acc[kk][m] = 0; amx[kk][m] = 0; }
        __syncthreads();
        constexpr int U = 4;  // requests per thread per pass: their loads are issued together
        for (long long base = b0 + threadIdx.x; base < b1; base += (long long)U * blockDim.x) {
            uint4 rv[U];
            uint32_t a[U], o[U], k[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const long long i = base + (long long)u * blockDim.x;
                const bool in = i < b1;
                rv[u] = in ? reinterpret_cast<const uint4 *>(res)[i] : make_uint4(0, 0, kNone, 0);
                a[u] = in ? arrival[i] : 0u;
                o[u] = in ? (uint32_t)olen[i] : 0u;
                k[u] = in ? (uint32_t)tier[i] : 0u;
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
                for (int m = 0; m < 3; ++m)
                    if (m != 1 || has_tbt) atomicAdd(&hist[(k[u] * 3 + m) * SIM_HIST_BUCKETS + lat_bucket(v[m])], 1u);
                // every accumulator is updated with a select (never indexed by the
                // tier), so all of them stay in registers; a one-token request's
                // TBT is 0: it adds nothing and leaves the maximum
#pragma unroll
                for (int kk = 0; kk < KM; ++kk) {
                    const bool hit = k[u] == (uint32_t)kk;
#pragma unroll
                    for (int m = 0; m < 3; ++m) {
                        acc[kk][m] += hit ? (unsigned long long)v[m] : 0ull;
                        amx[kk][m] = hit ? max(amx[kk][m], v[m]) : amx[kk][m];
                    }
                }
            }
        }
        // the lanes' sums and maxima: warp reduction, one global atomic per warp and group
        sim_latency_stats_t *orow = out + (size_t)r * G;
#pragma unroll
        for (int kk = 0; kk < KM; ++kk) {
#pragma unroll
            for (int m = 0; m < 3; ++m) {
                if (kk >= KT) continue;  // warp-uniform
                unsigned long long sv = acc[kk][m];
#pragma unroll
                for (int sh = 16; sh > 0; sh >>= 1) sv += __shfl_xor_sync(kFull, sv, sh);
                const uint32_t mv = __reduce_max_sync(kFull, amx[kk][m]);
                if (lane == 0 && sv) atomicAdd(reinterpret_cast<unsigned long long *>(&orow[kk * 3 + m].sum_us), sv);
                if (lane == 0 && mv) atomicMax(&orow[kk * 3 + m].max_us, mv);
            }
        }
        __syncthreads();
        for (int q = threadIdx.x; q < G * SIM_HIST_BUCKETS; q += blockDim.x) {
            const uint32_t h = hist[q];
            if (h) atomicAdd(&orow[q / SIM_HIST_BUCKETS].hist[q % SIM_HIST_BUCKETS], h);
        }
        __syncthreads();
    }
}

// Counts and nearest-rank P50 / P90 / P99 of the merged histograms: one warp per
// (replica, tier, measure); the percentile is the floor of the bucket holding
// the value of rank ceil(p n / 100).
__global__ void k_latency_pct(long long ngroups, sim_latency_stats_t *out) {
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
        uint32_t pv[3];
#pragma unroll
        for (int q = 0; q < 3; ++q) {
            const uint32_t rank = n ? max(1u, (uint32_t)(((unsigned long long)pct[q] * n + 99u) / 100u)) : 0u;
            uint32_t found = kNone;
            if (n && excl < rank && rank <= incl) {
                uint32_t cum = excl;
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    cum += c[j];
                    if (found == kNone && cum >= rank) found = lat_floor((uint32_t)(lane * 8 + j));
                }
            }
            pv[q] = __reduce_min_sync(kFull, found);
            if (!n) pv[q] = 0;
        }
        if (lane == 0) {
            o->count = n;
            o->p50_us = pv[0];
            o->p90_us = pv[1];
            o->p99_us = pv[2];
        }
    }
}

}  // namespace

cudaError_t launch(const int *chunk_rep, const long long *chunk_b0, int nchunks, const long long *offsets, int KT,
                   const uint32_t *arrival, const uint16_t *olen, const uint8_t *tier,
                   const sim_request_result_t *res, sim_latency_stats_t *out, long long ngroups, int sms,
                   cudaStream_t stream) {
    cudaError_t e = cudaMemsetAsync(out, 0, (size_t)ngroups * sizeof(sim_latency_stats_t), stream);
    if (e != cudaSuccess) return e;
    if (nchunks > 0) {
        const size_t smem = (size_t)KT * 3 * 4 * SIM_HIST_BUCKETS;  // <= 46,080 bytes for K <= 16
        const int grid = std::max(1, std::min(nchunks, sms * 16));
        auto fn = KT <= 2 ? k_latency_hist<2> : KT <= 4 ? k_latency_hist<4> : KT <= 8 ? k_latency_hist<8>
                                                                                   : k_latency_hist<16>;
        fn<<<grid, 256, smem, stream>>>(chunk_rep, chunk_b0, nchunks, offsets, KT, arrival, olen, tier, res, out);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    const long long nb = std::min<long long>((ngroups + 7) / 8, (long long)sms * 32);
    k_latency_pct<<<(unsigned)std::max<long long>(nb, 1), 256, 0, stream>>>(ngroups, out);
    return cudaGetLastError();
}

}  // namespace mtlat
