// Bucketing by scene (the per-scene candidate sets of level 2, Sec. "Level-2:
// scene-primitive retrieval"): a counting sort of token ids by their level-1
// scene, done by one CTA with the per-scene counters in shared memory.
//
// Outputs
//   scene_out[t]   the routed scene of every token (decoded argmax key)
//   perm           token ids grouped by scene (scene-major; order inside a
//                  scene is unspecified)
//   work           level-2 work items (scene, begin, count <= 8, slot) in
//                  scene order: every scene's bucket cut into chunks
//   routed         the distinct routed scenes in increasing order; a scene's
//                  position in it is its `slot`
//   counters[0..3] number of work items, of routed scenes, largest bucket;
//                  [3] is reset to 0 for the level-2 kernel's work taking
#include "common.cuh"

namespace lookme {

namespace {
constexpr int kThreads = 1024;

// Exclusive block-wide scan of three counters at once.
__device__ void block_exclusive_scan3(int3 v, int3& excl, int3& total, int3* warp_buf) {
    const int lane = threadIdx.x % 32, warp = threadIdx.x / 32;
    int3 inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int a = __shfl_up_sync(0xFFFFFFFFu, inc.x, o);
        const int b = __shfl_up_sync(0xFFFFFFFFu, inc.y, o);
        const int c = __shfl_up_sync(0xFFFFFFFFu, inc.z, o);
        if (lane >= o) {
            inc.x += a;
            inc.y += b;
            inc.z += c;
        }
    }
    if (lane == 31) warp_buf[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        int3 w = lane < kThreads / 32 ? warp_buf[lane] : make_int3(0, 0, 0);
        int3 wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int a = __shfl_up_sync(0xFFFFFFFFu, wi.x, o);
            const int b = __shfl_up_sync(0xFFFFFFFFu, wi.y, o);
            const int c = __shfl_up_sync(0xFFFFFFFFu, wi.z, o);
            if (lane >= o) {
                wi.x += a;
                wi.y += b;
                wi.z += c;
            }
        }
        if (lane < kThreads / 32) warp_buf[lane] = make_int3(wi.x - w.x, wi.y - w.y, wi.z - w.z);
        if (lane == kThreads / 32 - 1) warp_buf[32] = wi;
    }
    __syncthreads();
    const int3 wb = warp_buf[warp];
    excl = make_int3(wb.x + inc.x - v.x, wb.y + inc.y - v.y, wb.z + inc.z - v.z);
    total = warp_buf[32];
}
}  // namespace

__global__ void __launch_bounds__(kThreads, 1)
    k2_bucket(unsigned long long* __restrict__ best, int64_t N, int S, int32_t* __restrict__ scene_out,
              int32_t* __restrict__ perm, WorkItem* __restrict__ work, int32_t* __restrict__ routed,
              int32_t* __restrict__ counters) {
    extern __shared__ int cnt[];  // [S]: counts, then running token offsets
    __shared__ int3 warp_buf[33];
    __shared__ int max_bucket;
    pdl_trigger();
    pdl_wait();
    const int tid = threadIdx.x;
    for (int s = tid; s < S; s += kThreads) cnt[s] = 0;
    if (tid == 0) max_bucket = 0;
    __syncthreads();
    for (int64_t t = tid; t < N; t += kThreads) {
        const int32_t s = unpack_scene(best[t], S);
        scene_out[t] = s;
        atomicAdd(&cnt[s], 1);
    }
    __syncthreads();

    // Each thread owns a contiguous run of scenes.
    const int per = (S + kThreads - 1) / kThreads;
    const int s0 = min(S, tid * per), s1 = min(S, s0 + per);
    int3 mine = make_int3(0, 0, 0);  // tokens, work items, routed scenes
    int mx = 0;
    for (int s = s0; s < s1; ++s) {
        const int c = cnt[s];
        mine.x += c;
        mine.y += (c + kTokensPerItem - 1) / kTokensPerItem;
        mine.z += c > 0;
        mx = max(mx, c);
    }
    int3 base, total;
    block_exclusive_scan3(mine, base, total, warp_buf);
    if (mx) atomicMax(&max_bucket, mx);

    int tok = base.x, wi = base.y, slot = base.z;
    for (int s = s0; s < s1; ++s) {
        const int c = cnt[s];
        cnt[s] = tok;
        if (c > 0) {
            routed[slot] = s;
            for (int b = 0; b < c; b += kTokensPerItem) {
                WorkItem w;
                w.scene = s;
                w.begin = tok + b;
                w.count = min(kTokensPerItem, c - b);
                w.slot = slot;
                work[wi++] = w;
            }
            ++slot;
        }
        tok += c;
    }
    __syncthreads();
    if (tid == 0) {
        counters[0] = total.y;
        counters[1] = total.z;
        counters[2] = max_bucket;
        counters[3] = 0;  // level-2 work-taking counter
    }
    for (int64_t t = tid; t < N; t += kThreads) {
        const int32_t s = unpack_scene(best[t], S);
        best[t] = 0ull;  // ready for the next call's argmax
        const int pos = atomicAdd(&cnt[s], 1);
        perm[pos] = (int32_t)t;
    }
}

cudaError_t launch_bucket(const LaunchCtx& c, unsigned long long* best, int64_t N, int64_t S,
                          int32_t* scene_out, int32_t* perm, WorkItem* work, int32_t* routed, int32_t* counters) {
    const size_t smem = (size_t)S * sizeof(int);
    return launch_pdl(k2_bucket, dim3(1), dim3(kThreads), smem, c.stream, best, N, (int)S, scene_out, perm, work,
                      routed, counters);
}

cudaError_t configure_bucket_kernel() {
    return cudaFuncSetAttribute(k2_bucket, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)(LOOKME_MAX_SCENES * sizeof(int)));
}

}  // namespace lookme
