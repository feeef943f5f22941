// Bucketing by scene (the per-scene candidate sets of level 2, Sec. "Level-2:
// scene-primitive retrieval"): a counting sort of token ids by their level-1
// scene, done by one CTA with the per-scene counters in shared memory.
//
// Outputs
//   scene_out[t]   the routed scene of every token (decoded argmax key)
//   work           level-2 work items (scene, begin, count <= 8, slot) in
//                  scene order: every scene's bucket cut into chunks
//   item_tok       the items' token ids, item-major: item i's tokens at
//                  [8 i, 8 i + count) (begin = 8 i), so a consumer that knows
//                  an item's index reads its tokens without first reading the
//                  item; order inside a scene is unspecified
//   routed         the distinct routed scenes in increasing order; a scene's
//                  position in it is its `slot`
//   counters[0..3] number of work items, of routed scenes, largest bucket;
//                  [3] is reset to 0 for the level-2 kernel's work taking
//
// With a gate, CTAs 1.. compute the injection gate meanwhile, one token per
// warp and 8 to 32 tokens per CTA (few per CTA when the call is small, so the
// ranks spread over many SMs and finish within the bucketing; up to all 32
// warps when there are many): rank_t = #{ j in segment : pi_j > pi_t, or pi_j == pi_t and
// j < t }, kept iff rank_t < r, the kept ones listed at sel[sel_base + rank_t]
// (and, optionally, that slot recorded per token in selpos, -1 if not kept).
// Each CTA stages the priorities its tokens' segments span in shared memory
// once.  This runs before the level-2 key stream, whose copies would
// otherwise queue every small load behind them.
#include <string.h>

#include <algorithm>

#include "common.cuh"

namespace lookme {

namespace {
constexpr int kThreads = 1024;
constexpr int kGateMaxTokens = kThreads / 32;  // tokens per gate CTA: at most one per warp
constexpr int kGateStage = 32768;  // bytes of priorities a gate CTA stages

__device__ __forceinline__ int segment_index(const GateSpec& gs, int64_t t) {
    int lo = 0, hi = gs.n_seg;  // off[lo] <= t < off[lo + 1]
    while (hi - lo > 1) {
        const int mid = (lo + hi) / 2;
        if (gs.off[mid] <= t) lo = mid;
        else hi = mid;
    }
    return lo;
}

// Gate CTA number `gi` (tokens [gi tpc, (gi + 1) tpc)).
__device__ void gate_block(const GateSpec& gs, float* buf, int cap, int tpc, int64_t gi) {
    const int tid = threadIdx.x, warp = tid / 32, lane = tid % 32;
    const int64_t tb = gi * tpc, te = min(gs.N, tb + tpc);
    if (tb >= te) return;  // uniform for the CTA
    const int64_t rb = gs.off[segment_index(gs, tb)], re = gs.off[segment_index(gs, te - 1) + 1];
    const bool staged = re - rb <= cap;  // uniform for the CTA
    if (staged) {
        for (int64_t i = tid; i < re - rb; i += kThreads) buf[i] = gs.priority[rb + i];
        __syncthreads();
    }
    const int64_t t = tb + warp;
    if (warp >= tpc || t >= te) return;
    const int sg = segment_index(gs, t);
    const int64_t b = gs.off[sg], len = gs.off[sg + 1] - b;
    const int64_t r = (int64_t)floor((double)len * gs.keep_ratio);
    bool keep;
    int64_t rank = t - b;  // the slot when every token of the segment is kept
    if (r <= 0) {
        keep = false;
    } else if (r >= len) {
        keep = true;
    } else {
        const uint32_t kt = orderable(gs.priority[t]);
        const int tl = (int)(t - b);
        const float* src = staged ? buf + (b - rb) : gs.priority + b;
        int cnt = 0;
        const int n = (int)len;
        int i = lane;
        for (; i + 96 < n; i += 128) {
            const float v0 = src[i], v1 = src[i + 32], v2 = src[i + 64], v3 = src[i + 96];
            const uint32_t k0 = orderable(v0), k1 = orderable(v1), k2 = orderable(v2), k3 = orderable(v3);
            cnt += ((k0 > kt) || (k0 == kt && i < tl)) + ((k1 > kt) || (k1 == kt && i + 32 < tl)) +
                   ((k2 > kt) || (k2 == kt && i + 64 < tl)) + ((k3 > kt) || (k3 == kt && i + 96 < tl));
        }
        for (; i < n; i += 32) {
            const uint32_t kj = orderable(src[i]);
            cnt += (kj > kt) || (kj == kt && i < tl);
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) cnt += __shfl_xor_sync(0xFFFFFFFFu, cnt, o);
        rank = cnt;
        keep = rank < r;
    }
    if (lane == 0) {
        gs.mask[t] = (uint8_t)keep;
        if (keep) gs.sel[gs.sel_base[sg] + rank] = (int32_t)t;
        if (gs.selpos) gs.selpos[t] = keep ? (int32_t)(gs.sel_base[sg] + rank) : -1;
    }
}
// Exclusive block-wide scan of two counters at once.
__device__ void block_exclusive_scan2(int2 v, int2& excl, int2& total, int2* warp_buf) {
    const int lane = threadIdx.x % 32, warp = threadIdx.x / 32;
    int2 inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int a = __shfl_up_sync(0xFFFFFFFFu, inc.x, o);
        const int b = __shfl_up_sync(0xFFFFFFFFu, inc.y, o);
        if (lane >= o) {
            inc.x += a;
            inc.y += b;
        }
    }
    if (lane == 31) warp_buf[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        int2 w = lane < kThreads / 32 ? warp_buf[lane] : make_int2(0, 0);
        int2 wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int a = __shfl_up_sync(0xFFFFFFFFu, wi.x, o);
            const int b = __shfl_up_sync(0xFFFFFFFFu, wi.y, o);
            if (lane >= o) {
                wi.x += a;
                wi.y += b;
            }
        }
        if (lane < kThreads / 32) warp_buf[lane] = make_int2(wi.x - w.x, wi.y - w.y);
        if (lane == kThreads / 32 - 1) warp_buf[32] = wi;
    }
    __syncthreads();
    const int2 wb = warp_buf[warp];
    excl = make_int2(wb.x + inc.x - v.x, wb.y + inc.y - v.y);
    total = warp_buf[32];
}
}  // namespace

__global__ void __launch_bounds__(kThreads, 1)
    k2_bucket(unsigned long long* best, int64_t N, int S, int32_t* __restrict__ scene_out,
              int32_t* __restrict__ item_tok, WorkItem* __restrict__ work, int32_t* __restrict__ routed,
              int32_t* __restrict__ counters, const __grid_constant__ GateSpec gate, int smem_bytes, int gate_tpc) {
    extern __shared__ int cnt[];  // CTA 0: [S] counts, then running item_tok positions; gate CTAs: priorities
    __shared__ int2 warp_buf[33];
    __shared__ int max_bucket;
    pdl_trigger();
    pdl_wait();
    if (blockIdx.x > 0) {
        gate_block(gate, reinterpret_cast<float*>(cnt), smem_bytes / 4, gate_tpc, (int64_t)blockIdx.x - 1);
        return;
    }
    const int tid = threadIdx.x;
    // Both sweeps over the tokens issue kB keys per thread before using any
    // (one round trip per batch, not per token); the scenes of a thread's
    // first batch stay in registers for the second sweep.
    // A batch stops at its last valid token, so a call of at most 1,024
    // tokens runs one slot per thread, not eight mostly idle ones.
    constexpr int kB = 8;
    unsigned long long key[kB];
    // The first batch is requested before the counters are cleared.
#pragma unroll
    for (int u = 0; u < kB; ++u) {
        const int64_t t = tid + (int64_t)u * kThreads;
        if (t >= N) break;
        key[u] = best[t];
    }
    for (int s = tid; s < S; s += kThreads) cnt[s] = 0;
    if (tid == 0) max_bucket = 0;
    __syncthreads();
    int32_t sc[kB];
    for (int64_t t0 = tid; t0 < N; t0 += (int64_t)kB * kThreads) {
        if (t0 != tid) {
#pragma unroll
            for (int u = 0; u < kB; ++u) {
                const int64_t t = t0 + (int64_t)u * kThreads;
                if (t >= N) break;
                key[u] = best[t];
            }
        }
#pragma unroll
        for (int u = 0; u < kB; ++u) {
            const int64_t t = t0 + (int64_t)u * kThreads;
            if (t >= N) break;
            const int32_t s = unpack_scene(key[u], S);
            if (t0 == tid) sc[u] = s;
            scene_out[t] = s;
            atomicAdd(&cnt[s], 1);
        }
    }
    __syncthreads();

    // Each thread owns a contiguous run of scenes.
    const int per = (S + kThreads - 1) / kThreads;
    const int s0 = min(S, tid * per), s1 = min(S, s0 + per);
    int2 mine = make_int2(0, 0);  // work items, routed scenes
    int mx = 0;
    for (int s = s0; s < s1; ++s) {
        const int c = cnt[s];
        mine.x += (c + kTokensPerItem - 1) / kTokensPerItem;
        mine.y += c > 0;
        mx = max(mx, c);
    }
    int2 base, total;
    block_exclusive_scan2(mine, base, total, warp_buf);
    // One shared atomic per warp, not one per routed scene on a single word.
    mx = __reduce_max_sync(0xFFFFFFFFu, mx);
    if (tid % 32 == 0 && mx) atomicMax(&max_bucket, mx);

    int wi = base.x, slot = base.y;
    for (int s = s0; s < s1; ++s) {
        const int c = cnt[s];
        cnt[s] = wi * kTokensPerItem;  // the scene's first item_tok position
        if (c > 0) {
            routed[slot] = s;
            for (int b = 0; b < c; b += kTokensPerItem) {
                WorkItem w;
                w.scene = s;
                w.begin = wi * kTokensPerItem;
                w.count = min(kTokensPerItem, c - b);
                w.slot = slot;
                work[wi++] = w;
            }
            ++slot;
        }
    }
    __syncthreads();
    if (tid == 0) {
        counters[0] = total.x;
        counters[1] = total.y;
        counters[2] = max_bucket;
        counters[3] = 0;  // level-2 work-taking counter
    }
    // A scene's k-th token lands in its item k / 8, lane k % 8; the keys are
    // cleared for the next call's argmax.
    for (int64_t t0 = tid; t0 < N; t0 += (int64_t)kB * kThreads) {
        int32_t s[kB];
        if (t0 == tid) {
#pragma unroll
            for (int u = 0; u < kB; ++u) s[u] = sc[u];
        } else {
            unsigned long long key[kB];
#pragma unroll
            for (int u = 0; u < kB; ++u) {
                const int64_t t = t0 + (int64_t)u * kThreads;
                if (t >= N) break;
                key[u] = best[t];
            }
#pragma unroll
            for (int u = 0; u < kB; ++u) {
                if (t0 + (int64_t)u * kThreads >= N) break;
                s[u] = unpack_scene(key[u], S);
            }
        }
#pragma unroll
        for (int u = 0; u < kB; ++u) {
            const int64_t t = t0 + (int64_t)u * kThreads;
            if (t >= N) break;
            best[t] = 0ull;
            const int pos = atomicAdd(&cnt[s[u]], 1);
            item_tok[pos] = (int32_t)t;
        }
    }
}

// ------------------------------------------------ large calls: three launches
// The same work list and item-major token ids as k2_bucket, over all SMs.
// Tokens of one scene in one warp are counted and placed with one atomic
// (warp-aggregated), so a scene holding a sixth of the tokens (Zipf) costs a
// few thousand atomics on its counter, not tens of thousands.

// Per-scene counts.  CTAs [0, n_count) take token ranges of `per`; the CTAs
// after them are gate CTAs (as in k2_bucket).
__global__ void __launch_bounds__(kThreads, 1)
    k2_count(unsigned long long* best, int64_t N, int S, int32_t* __restrict__ scene_out, int32_t* cnt, int64_t per,
             int n_count, const __grid_constant__ GateSpec gate, int smem_bytes, int gate_tpc) {
    extern __shared__ float stage[];
    pdl_trigger();
    pdl_wait();
    if ((int)blockIdx.x >= n_count) {
        gate_block(gate, stage, smem_bytes / 4, gate_tpc, (int64_t)blockIdx.x - n_count);
        return;
    }
    const int lane = threadIdx.x % 32;
    const int64_t t0 = (int64_t)blockIdx.x * per, t1 = min(N, t0 + per);
    for (int64_t tb = t0; tb < t1; tb += kThreads) {
        const int64_t t = tb + threadIdx.x;
        const bool valid = t < t1;
        const int32_t s = valid ? unpack_scene(best[t], S) : -1;
        if (valid) scene_out[t] = s;
        const uint32_t peers = __match_any_sync(0xFFFFFFFFu, s);
        if (valid && lane == __ffs(peers) - 1) atomicAdd(&cnt[s], __popc(peers));
    }
}

// The work list from the counts (one CTA), in rounds of 1,024 consecutive
// scenes (thread i takes scene 1024 r + i, a block-wide scan per round and a
// carry between rounds), so that every load and store of the round is
// coalesced; pos[s] = the scene's first item_tok position; the counts are
// zeroed for the next call.
__global__ void __launch_bounds__(kThreads, 1)
    k2_scan(int S, int32_t* cnt, int32_t* __restrict__ pos, WorkItem* __restrict__ work,
            int32_t* __restrict__ routed, int32_t* __restrict__ counters) {
    __shared__ int2 warp_buf[33];
    __shared__ int max_bucket;
    pdl_trigger();
    pdl_wait();
    const int tid = threadIdx.x;
    if (tid == 0) max_bucket = 0;
    int carry_items = 0, carry_routed = 0, mx = 0;
    for (int r0 = 0; r0 < S; r0 += kThreads) {
        const int s = r0 + tid;
        const int c = s < S ? cnt[s] : 0;
        if (s < S) cnt[s] = 0;
        mx = max(mx, c);
        int2 base, total;
        block_exclusive_scan2(make_int2((c + kTokensPerItem - 1) / kTokensPerItem, c > 0), base, total, warp_buf);
        const int wi = carry_items + base.x, slot = carry_routed + base.y;
        if (s < S) {
            pos[s] = wi * kTokensPerItem;
            if (c > 0) {
                routed[slot] = s;
                for (int b = 0, i = wi; b < c; b += kTokensPerItem, ++i) {
                    WorkItem w;
                    w.scene = s;
                    w.begin = i * kTokensPerItem;
                    w.count = min(kTokensPerItem, c - b);
                    w.slot = slot;
                    work[i] = w;
                }
            }
        }
        carry_items += total.x;
        carry_routed += total.y;
        __syncthreads();  // warp_buf is reused by the next round
    }
    mx = __reduce_max_sync(0xFFFFFFFFu, mx);
    if (tid % 32 == 0 && mx) atomicMax(&max_bucket, mx);
    __syncthreads();
    if (tid == 0) {
        counters[0] = carry_items;
        counters[1] = carry_routed;
        counters[2] = max_bucket;
        counters[3] = 0;  // level-2 work-taking counter
    }
}

// The token ids into their items: a scene's k-th placed token lands in its
// item k / 8, lane k % 8; the keys are cleared for the next call's argmax.
__global__ void __launch_bounds__(kThreads)
    k2_scatter(unsigned long long* best, int64_t N, const int32_t* scene_out, int32_t* pos,
               int32_t* __restrict__ item_tok, int64_t per) {
    pdl_trigger();
    pdl_wait();
    const int lane = threadIdx.x % 32;
    const int64_t t0 = (int64_t)blockIdx.x * per, t1 = min(N, t0 + per);
    for (int64_t tb = t0; tb < t1; tb += kThreads) {
        const int64_t t = tb + threadIdx.x;
        const bool valid = t < t1;
        const int32_t s = valid ? scene_out[t] : -1;
        const uint32_t peers = __match_any_sync(0xFFFFFFFFu, s);
        const int leader = __ffs(peers) - 1;
        int base = 0;
        if (valid && lane == leader) base = atomicAdd(&pos[s], __popc(peers));
        base = __shfl_sync(0xFFFFFFFFu, base, leader);
        if (valid) {
            item_tok[base + __popc(peers & ((1u << lane) - 1u))] = (int32_t)t;
            best[t] = 0ull;
        }
    }
}

namespace {
// Tokens per gate CTA: about two gate CTAs per SM, 8 to 32 tokens each.
int gate_tokens_per_cta(const LaunchCtx& c, int64_t N) {
    const int64_t want = (N + 2 * (int64_t)c.num_sms - 1) / (2 * (int64_t)c.num_sms);
    return (int)std::min<int64_t>(kGateMaxTokens, std::max<int64_t>(8, want));
}
// Token ranges of the count and scatter launches: one range per SM at most.
int64_t big_ranges(const LaunchCtx& c, int64_t N) {
    return std::max<int64_t>(1, std::min<int64_t>(c.num_sms, (N + kThreads - 1) / kThreads));
}
}  // namespace

cudaError_t launch_bucket_count(const LaunchCtx& c, unsigned long long* best, int64_t N, int64_t S,
                                int32_t* scene_out, int32_t* cnt, const GateSpec* gate) {
    GateSpec gs;
    if (gate) {
        gs = *gate;
    } else {
        memset(&gs, 0, sizeof(gs));
    }
    const int64_t nr = big_ranges(c, N);
    const int64_t per = (N + nr - 1) / nr;
    const int n_count = (int)((N + per - 1) / per);
    const int tpc = gate_tokens_per_cta(c, N);
    const int gate_ctas = gate ? (int)((N + tpc - 1) / tpc) : 0;
    const int smem = gate ? kGateStage : 0;
    return launch_pdl(k2_count, dim3(n_count + gate_ctas), dim3(kThreads), (size_t)smem, c.stream, best, N, (int)S,
                      scene_out, cnt, per, n_count, gs, smem, tpc);
}

cudaError_t launch_bucket_scan(const LaunchCtx& c, int64_t S, int32_t* cnt, int32_t* pos, WorkItem* work,
                               int32_t* routed, int32_t* counters) {
    return launch_pdl(k2_scan, dim3(1), dim3(kThreads), 0, c.stream, (int)S, cnt, pos, work, routed, counters);
}

cudaError_t launch_bucket_scatter(const LaunchCtx& c, unsigned long long* best, int64_t N,
                                  const int32_t* scene_out, int32_t* pos, int32_t* item_tok) {
    const int64_t nr = big_ranges(c, N);
    const int64_t per = (N + nr - 1) / nr;
    const int grid = (int)((N + per - 1) / per);
    return launch_pdl(k2_scatter, dim3(grid), dim3(kThreads), 0, c.stream, best, N, scene_out, pos, item_tok, per);
}

cudaError_t launch_bucket(const LaunchCtx& c, unsigned long long* best, int64_t N, int64_t S,
                          int32_t* scene_out, int32_t* item_tok, WorkItem* work, int32_t* routed, int32_t* counters,
                          const GateSpec* gate) {
    GateSpec gs;
    if (gate) {
        gs = *gate;
    } else {
        memset(&gs, 0, sizeof(gs));
    }
    const int tpc = gate_tokens_per_cta(c, N);
    const int gate_ctas = gate ? (int)((N + tpc - 1) / tpc) : 0;
    const int smem = (int)std::max<int64_t>(S * (int64_t)sizeof(int), gate ? kGateStage : 0);
    return launch_pdl(k2_bucket, dim3(1 + gate_ctas), dim3(kThreads), (size_t)smem, c.stream, best, N, (int)S,
                      scene_out, item_tok, work, routed, counters, gs, smem, tpc);
}

cudaError_t configure_bucket_kernel() {
    return cudaFuncSetAttribute(k2_bucket, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)std::max<int64_t>(LOOKME_MAX_SCENES * sizeof(int), kGateStage));
}

}  // namespace lookme
