// latency.cuh -- internal interface between the C-ABI host layer (mtsim.cu)
// and the per-tier latency-statistics kernels (latency.cu).
#ifndef MTSIM_LATENCY_CUH
#define MTSIM_LATENCY_CUH

#include "mtsim.h"

#include <cuda_runtime.h>

namespace mtlat {

// Requests are cut into chunks of at most kChunk records within one replica;
// chunk c covers [chunk_b0[c], min(chunk_b0[c] + kChunk, offsets[r + 1])) of
// replica chunk_rep[c].
constexpr int kChunk = 4096;

// Bins of one radix-selection step: the next 8 bits of a value.
constexpr int kSelBins = 256;

// Device scratch of one call, per (group, percentile): the selection state
// (16 bytes) and kSelBins 32-bit bins.
inline size_t select_state_bytes(long long ngroups) { return (size_t)ngroups * 3u * 16u; }
inline size_t select_bin_bytes(long long ngroups) { return (size_t)ngroups * 3u * kSelBins * 4u; }

// Queues on `stream`: clear out ([ngroups] records, ngroups = R * KT * 3),
// histogram, sum and maximum of every (replica, tier, measure) group, the
// counts, the bucket of every percentile's rank, then the selection passes
// that narrow each bucket to the exact value.  sel and bins are scratch of
// select_state_bytes / select_bin_bytes (contents need not be set).  All
// pointers are device memory; res, arrival, olen, tier are the trace and
// results of all replicas (may be NULL when nchunks is 0).  Returns the
// first CUDA error.
cudaError_t launch(const int *chunk_rep, const long long *chunk_b0, int nchunks, const long long *offsets, int KT,
                   const uint32_t *arrival, const uint16_t *olen, const uint8_t *tier,
                   const sim_request_result_t *res, sim_latency_stats_t *out, long long ngroups, uint4 *sel,
                   uint32_t *bins, int sms, cudaStream_t stream);

}  // namespace mtlat

#endif
