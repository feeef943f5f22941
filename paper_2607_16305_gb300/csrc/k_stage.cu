// On-demand loading of a partitioned table (Sec. "Level-2: scene-primitive
// retrieval", last sentence; Sec. "Embedding Lookup in VLMs": only the scene
// centroids stay resident, the table lives outside device memory).
//
// The same file holds the load-time kernel that lays keys out as tiles.
//
// K6 stage: after bucketing has produced the list of routed scenes on the
// device, copy each routed scene's key block from pinned host memory (read
// through its device mapping over the host link) into the HBM slot with the
// same index.  The list never goes back to the host.
#include <algorithm>

#include "common.cuh"

namespace lookme {

__global__ void __launch_bounds__(256) k6_stage(const uint4* __restrict__ keys_host, uint4* __restrict__ slots,
                                                int64_t block_vecs, int64_t n_slots,
                                                const int32_t* routed, const int32_t* counters) {
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

// Load time: keys of n scenes, row-major [n][P][d_k] bf16, into the tiled
// layout the tcgen05 level-2 kernel copies straight into shared memory: per
// scene, for each N-tile of 256 rows (the last may be 128), for each 64-wide
// k-block, the N-tile's 128-row sub-blocks; each sub-block is 128 rows x 128
// bytes with 16-byte chunk c of row r at position c ^ (r & 7).  One thread per
// 16-byte output chunk, so the writes are coalesced.
__global__ void __launch_bounds__(256) k_tile_keys(const uint4* __restrict__ src, uint4* __restrict__ dst,
                                                   int64_t n, int64_t P, int row_chunks, int ntile, int nkb) {
    const int64_t per_scene = (int64_t)ntile * nkb * 128 * 8;
    const int64_t total = n * per_scene;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
        const int64_t s = i / per_scene;
        const int64_t rem = i - s * per_scene;
        const int sb = (int)(rem >> 10), w = (int)(rem & 1023);
        const int r = w >> 3, pos = w & 7;
        // Sub-block sb: N-tile nt (two 128-row tiles, the last maybe one), then
        // k-block kb, then the tile within the N-tile.
        const int nt = sb / (2 * nkb), in_nt = sb - nt * 2 * nkb;
        const int ns = (2 * nt + 1 < ntile) ? 2 : 1;
        const int kb = in_nt / ns, tile = 2 * nt + (in_nt - kb * ns);
        const int64_t p = (int64_t)tile * 128 + r;
        const int kc = kb * 8 + (pos ^ (r & 7));  // 16-byte chunk of the source row
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (p < P && kc < row_chunks) v = src[(s * P + p) * row_chunks + kc];
        dst[i] = v;
    }
}

cudaError_t launch_tile_keys(const LaunchCtx& c, const void* src, void* dst, int64_t n, int64_t P, int dk) {
    if (n == 0) return cudaSuccess;
    const int ntile = (int)((P + 127) / 128), nkb = (dk + 63) / 64;
    const int64_t total = n * ntile * nkb * 1024;
    const int64_t blocks = std::min<int64_t>((total + 255) / 256, (int64_t)c.num_sms * 16);
    k_tile_keys<<<(unsigned)blocks, 256, 0, c.stream>>>((const uint4*)src, (uint4*)dst, n, P, dk / 8, ntile, nkb);
    return cudaGetLastError();
}

cudaError_t launch_stage(const LaunchCtx& c, const void* keys_host_mapped, void* slots, int64_t block_bytes,
                         int64_t n_slots, const int32_t* routed, const int32_t* counters) {
    return launch_pdl(k6_stage, dim3(c.num_sms * 8), dim3(256), 0, c.stream, (const uint4*)keys_host_mapped,
                      (uint4*)slots, block_bytes / 16, n_slots, routed, counters);
}

}  // namespace lookme
