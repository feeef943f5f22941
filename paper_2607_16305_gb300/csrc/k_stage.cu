// On-demand loading of a partitioned table (Sec. "Level-2: scene-primitive
// retrieval", last sentence; Sec. "Embedding Lookup in VLMs": only the scene
// centroids stay resident, the table lives outside device memory).
//
// The same file holds the load-time kernel that lays keys out as tiles.
//
// K6, in two launches after bucketing has produced the list of routed
// scenes on the device (the list never goes back to the host):
//  a) one CTA looks every routed scene up in the table's persistent HBM slot
//     cache.  Hits keep their slot; each miss takes a slot that no routed
//     scene of this call uses (an empty one, or the one holding the scene
//     reached longest ago by a clock hand), evicting its scene.  The work
//     items are pointed at their slots and the misses listed for copying.
//  b) the listed key blocks are copied from pinned host memory, read through
//     its device mapping over the host link, into their slots.  The library
//     runs (b) on a stream of its own, ordered by events after (a) and before
//     level 2.
#include <algorithm>

#include "common.cuh"

namespace lookme {

namespace {
constexpr int kAssignThreads = 1024;

// Exclusive prefix sum of v over the CTA's 1,024 threads; total gets the sum.
__device__ int cta_excl_scan(int v, int& total, int* buf) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int n = __shfl_up_sync(0xFFFFFFFFu, inc, o);
        if (lane >= o) inc += n;
    }
    if (lane == 31) buf[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        int w = buf[lane];
        int wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int n = __shfl_up_sync(0xFFFFFFFFu, wi, o);
            if (lane >= o) wi += n;
        }
        buf[lane] = wi - w;
        if (lane == 31) buf[32] = wi;
    }
    __syncthreads();
    const int excl = buf[warp] + inc - v;
    total = buf[32];
    __syncthreads();
    return excl;
}
}  // namespace

__global__ void __launch_bounds__(kAssignThreads, 1)
    k6_assign(StageArgs sa, const int32_t* routed, const int32_t* counters, WorkItem* work, uint32_t* status) {
    __shared__ int buf[33];
    __shared__ int s_epoch, s_hand, s_new_hand;
    pdl_trigger();
    pdl_wait();
    const int tid = threadIdx.x;
    const int n_routed = counters[1], n_work = counters[0];
    const int n_slots = (int)sa.n_slots;
    if (tid == 0) {
        s_epoch = sa.hdr->epoch + 1;
        s_hand = sa.hdr->hand;
        s_new_hand = s_hand;
    }
    __syncthreads();
    const int epoch = s_epoch, hand = s_hand;
    // Hits keep their slot (stamped with this call); misses are marked -1.
    int hits = 0;
    for (int i = tid; i < n_routed; i += kAssignThreads) {
        const int sl = sa.slot_of[routed[i]];
        sa.route_slot[i] = sl;
        if (sl >= 0) {
            sa.slot_stamp[sl] = epoch;
            ++hits;
        }
    }
    __syncthreads();
    // Misses ranked in routed-list order: route_slot = -2 - rank.
    int n_miss = 0;
    for (int base = 0; base < n_routed; base += kAssignThreads) {
        const int i = base + tid;
        const bool miss = i < n_routed && sa.route_slot[i] < 0;
        int tot;
        const int r = cta_excl_scan(miss ? 1 : 0, tot, buf);
        if (miss) sa.route_slot[i] = -2 - (n_miss + r);
        n_miss += tot;
    }
    // Victims: slots not stamped by this call, in clock order from the hand;
    // the m-th one found serves the m-th miss.
    int found = 0;
    for (int base = 0; base < n_slots && found < n_miss; base += kAssignThreads) {
        const int k = base + tid;
        const int j = k < n_slots ? (hand + k) % n_slots : 0;
        const bool cand = k < n_slots && sa.slot_stamp[j] != epoch;
        int tot;
        const int r = cta_excl_scan(cand ? 1 : 0, tot, buf);
        const int m = found + r;
        if (cand && m < n_miss) {
            sa.copy_slot[m] = j;
            if (m == n_miss - 1) s_new_hand = (j + 1) % n_slots;
        }
        found += tot;
    }
    __syncthreads();
    const int n_copy = min(n_miss, found);
    // Evict each victim's scene and bind the miss to the slot.  A victim's
    // scene is not routed in this call (every routed scene's slot is stamped),
    // so no scene is both evicted and bound here.
    for (int i = tid; i < n_routed; i += kAssignThreads) {
        const int v = sa.route_slot[i];
        if (v >= 0) continue;
        const int m = -2 - v;
        if (m < n_copy) {
            const int j = sa.copy_slot[m], sc = routed[i];
            const int old = sa.slot_scene[j];
            if (old >= 0) sa.slot_of[old] = -1;
            sa.slot_scene[j] = sc;
            sa.slot_of[sc] = j;
            sa.slot_stamp[j] = epoch;
            sa.copy_scene[m] = sc;
            sa.route_slot[i] = j;
        } else {
            sa.route_slot[i] = 0;  // no slot left: never reached when n_routed <= n_slots
        }
    }
    int tot_hits;
    cta_excl_scan(hits, tot_hits, buf);  // also orders the writes above before the rewrite
    // Work items carry their scene's routed-list index; point them at the slot.
    for (int e = tid; e < n_work; e += kAssignThreads) work[e].slot = sa.route_slot[work[e].slot];
    if (tid == 0) {
        sa.hdr->epoch = epoch;
        sa.hdr->hand = s_new_hand;
        sa.hdr->n_copy = n_copy;
        sa.hdr->n_hit = tot_hits;
        if (n_copy < n_miss) atomicOr(status, STATUS_STAGE_OVERFLOW);
    }
}

// K6b: copies the key blocks listed by K6a, four independent 16-byte loads in
// flight per thread and iteration.
__global__ void __launch_bounds__(256) k6_stage(const uint4* __restrict__ keys_host, uint4* __restrict__ slots,
                                                int64_t block_vecs, StageArgs sa) {
    pdl_trigger();
    pdl_wait();
    const int64_t total = (int64_t)sa.hdr->n_copy * block_vecs;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    auto src = [&](int64_t k) {
        const int64_t m = k / block_vecs;
        return (int64_t)sa.copy_scene[m] * block_vecs + (k - m * block_vecs);
    };
    auto dst = [&](int64_t k) {
        const int64_t m = k / block_vecs;
        return (int64_t)sa.copy_slot[m] * block_vecs + (k - m * block_vecs);
    };
    for (; i + 3 * stride < total; i += 4 * stride) {
        uint4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) v[u] = keys_host[src(i + u * stride)];
#pragma unroll
        for (int u = 0; u < 4; ++u) slots[dst(i + u * stride)] = v[u];
    }
    for (; i < total; i += stride) slots[dst(i)] = keys_host[src(i)];
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

cudaError_t launch_stage_assign(const LaunchCtx& c, const StageArgs& sa, const int32_t* routed,
                                const int32_t* counters, WorkItem* work, uint32_t* status) {
    return launch_pdl(k6_assign, dim3(1), dim3(kAssignThreads), 0, c.stream, sa, routed, counters, work, status);
}

cudaError_t launch_stage(const LaunchCtx& c, const void* keys_host_mapped, void* slots, int64_t block_bytes,
                         const StageArgs& sa) {
    return launch_pdl(k6_stage, dim3(c.num_sms * 8), dim3(256), 0, c.stream, (const uint4*)keys_host_mapped,
                      (uint4*)slots, block_bytes / 16, sa);
}

}  // namespace lookme
