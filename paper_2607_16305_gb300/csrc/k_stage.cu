// On-demand loading of a partitioned table (Sec. "Level-2: scene-primitive
// retrieval", last sentence; Sec. "Embedding Lookup in VLMs": only the scene
// centroids stay resident, the table lives outside device memory).
//
// K6 stage: after bucketing has produced the list of routed scenes on the
// device, copy each routed scene's key block from pinned host memory (read
// through its device mapping over the host link) into the HBM slot with the
// same index.  The list never goes back to the host.
#include "common.cuh"

namespace lookme {

__global__ void __launch_bounds__(256) k6_stage(const uint4* __restrict__ keys_host, uint4* __restrict__ slots,
                                                int64_t block_vecs, int64_t n_slots,
                                                const int32_t* __restrict__ routed,
                                                const int32_t* __restrict__ counters) {
    pdl_trigger();
    pdl_wait();
    const int64_t n_routed = min((int64_t)counters[1], n_slots);
    const int64_t total = n_routed * block_vecs;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    // Four independent 16-byte loads in flight per thread and iteration.
    for (; i + 3 * stride < total; i += 4 * stride) {
        uint4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int64_t k = i + u * stride;
            const int64_t slot = k / block_vecs;
            v[u] = keys_host[(int64_t)routed[slot] * block_vecs + (k - slot * block_vecs)];
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) slots[i + u * stride] = v[u];
    }
    for (; i < total; i += stride) {
        const int64_t slot = i / block_vecs;
        slots[i] = keys_host[(int64_t)routed[slot] * block_vecs + (i - slot * block_vecs)];
    }
}

cudaError_t launch_stage(const LaunchCtx& c, const void* keys_host_mapped, void* slots, int64_t block_bytes,
                         int64_t n_slots, const int32_t* routed, const int32_t* counters) {
    return launch_pdl(k6_stage, dim3(c.num_sms * 8), dim3(256), 0, c.stream, (const uint4*)keys_host_mapped,
                      (uint4*)slots, block_bytes / 16, n_slots, routed, counters);
}

}  // namespace lookme
