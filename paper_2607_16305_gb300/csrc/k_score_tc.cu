// Level 2 on the 5th-generation tensor cores (bf16 tables), Sec. "Level-2:
// scene-primitive retrieval" in its key-similarity form:
//   z_tp = q_t . K[j, p] / sqrt(d_k), I_t = top-k of z_t, w_t = softmax(z_t[I_t]).
//
// Each work item (a scene and <= 8 of its tokens) is a small grouped GEMM:
// D[p][j] = K[scene, p, :] . q_j for the scene's N_p key rows and the item's
// tokens.  The keys are the M = 128 operand, the tokens the N = 16 operand (a
// swizzled K-major tile built in shared memory from bulk-copied query rows),
// and the fp32 accumulator lives in TMEM.
//
// The table stores every scene's keys as the exact shared-memory image the
// MMA reads: sub-blocks of 128 rows x 64 columns (16 KiB, 128-byte swizzle),
// k-block-major then row tile, zero-padded past N_p and d_k.  A scene's block is
// therefore contiguous and is streamed with 1-D bulk copies of up to four
// sub-blocks (64 KiB): a copy costs the SM's copy engine about the same time
// whatever its size in this range, so large copies are what lets one CTA per
// SM pull its share of HBM bandwidth.
//
// With N = 16 each MMA is short, and back-to-back MMAs into one accumulator
// wait on each other; so each row tile accumulates into nacc partial sums
// (k-block b goes to partial b % nacc) and a copy's MMAs are issued k-step by
// k-step across its sub-blocks, which keeps several independent
// accumulations in flight.  The epilogue adds the partials.  The tensor core
// removes the CUDA-core work that would otherwise have to keep pace with the
// key stream.  One CTA
// per SM, static share of the work list (items b, b + G, b + 2G, ...):
//   warp 0       producer: reads each item's work entry and streams the
//                scene's key block through the ring (bulk copies only)
//   warp 1       one thread issues tcgen05.mma into one of two TMEM buffers
//   warps 2..9   epilogue: TMEM -> logits in shared memory (scaled), then
//                top-k + softmax, one token per warp (redux.sync argmax)
//   warp 10      token tiles: reads the item's token ids and query rows with
//                plain 16-byte loads and writes them straight into the
//                swizzled K-major tile (small copies would each cost the
//                copy engine as much time as a 64 KiB one)
// Every wait is bounded; on a timeout the kernel drains its copies and MMAs,
// releases TMEM and reports through the status word.
#include <cuda.h>

#include "common.cuh"
#include "sm100.cuh"
#include "topk.cuh"

namespace lookme {

namespace k3tc {
constexpr int BM = 128;                  // key rows per MMA tile
constexpr int BK = 64;                   // bf16 elements per 128-byte swizzled row
constexpr int BN = 16;                   // token columns (an item holds <= 8 tokens)
constexpr int kTok = kTokensPerItem;
constexpr int kSubBytes = BM * 128;      // one 128 x 64 key sub-block: 16 KiB
constexpr int kBKbBytes = BN * 128;      // one 16 x 64 token block: 2 KiB
constexpr int kEpiWarps = 8;
constexpr int kBuildWarp = 2 + kEpiWarps;
constexpr int kThreads = (3 + kEpiWarps) * 32;
constexpr int kQBatch = 8;               // query-row chunks in flight per lane
constexpr int kMaxStages = 14;          // ring slots (barrier arrays)
constexpr int kMaxGroup = 4;             // sub-blocks per bulk copy / ring slot
constexpr int kBSlots = 2;               // token tiles
constexpr int kISlots = 4;               // item metadata (scene, count, token ids)
constexpr uint64_t kTimeoutNs = 1000000000ull;
constexpr int kSmemLimit = 227 * 1024;

struct Geometry {
    int nkb;              // 64-wide k-blocks of d_k
    int ntile;            // 128-row tiles of N_p
    int group;            // sub-blocks per ring slot (one bulk copy)
    int slot_bytes;       // group x 16 KiB
    int n_stages;         // ring slots
    int spi;              // sub-blocks per item (ntile x nkb)
    int chunks;           // bulk copies per item
    int row_bytes;        // d_k * 2
    int b_bytes;          // one token tile (nkb x 2 KiB)
    int nacc;             // partial accumulators per row tile
    int tmem_cols;        // allocated TMEM columns (two buffers of ntile x nacc x 16)
    int off_b, off_z, off_bar, off_meta;
    int smem;             // bytes requested, including 1 KiB of alignment slack
};

inline Geometry geometry(int64_t P, int dk) {
    Geometry g;
    g.nkb = (dk + BK - 1) / BK;
    g.ntile = (int)((P + BM - 1) / BM);
    g.row_bytes = dk * 2;
    g.b_bytes = g.nkb * kBKbBytes;
    g.nacc = min(4, g.nkb);
    while (g.nacc > 1 && 2 * g.ntile * g.nacc * BN > 512) --g.nacc;
    int cols = 32;
    while (cols < 2 * g.ntile * g.nacc * BN) cols <<= 1;
    g.tmem_cols = cols;
    const int zbytes = (kTok * (int)P * 4 + 15) / 16 * 16;
    const int fixed = kBSlots * g.b_bytes + zbytes + 1024 /*bar+meta*/ + 1024 /*align*/;
    g.spi = g.ntile * g.nkb;
    // The largest copies that still leave at least two ring slots.
    g.group = kMaxGroup;
    while (g.group > 1 && (kSmemLimit - fixed) / (g.group * kSubBytes) < 2) g.group >>= 1;
    if (g.group > g.spi) g.group = g.spi;
    g.slot_bytes = g.group * kSubBytes;
    g.chunks = (g.spi + g.group - 1) / g.group;
    g.n_stages = (kSmemLimit - fixed) / g.slot_bytes;
    if (g.n_stages > kMaxStages) g.n_stages = kMaxStages;
    g.off_b = g.n_stages * g.slot_bytes;
    g.off_z = g.off_b + kBSlots * g.b_bytes;
    g.off_bar = g.off_z + zbytes;
    g.off_meta = g.off_bar + (2 * kMaxStages + 2 * kBSlots + 2 * kISlots + 2 * 2 + 1) * 8;
    g.smem = g.off_meta + kISlots * ((int)sizeof(WorkItem) + kTok * 4) + 16 + 1024;
    return g;
}

// Named barrier 1 over the epilogue warps, returning the OR of `v` over them.
__device__ __forceinline__ bool epi_sync_or(bool v) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.or.pred q, 1, %2, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)v), "n"(kEpiWarps * 32)
        : "memory");
    return r != 0;
}
// Position in an item's sub-blocks (k-block-major, then row tile).
struct SubCursor {
    int kb, tile, kbm;  // k-block, row tile, kb % nacc
};

// Issues the MMAs of one ring slot's nsub sub-blocks, k-step by k-step across
// the sub-blocks so that consecutive MMAs go to different accumulators, and
// returns the cursor past them.  live = 0 runs the same instructions with
// every MMA switched off: called once before the grid dependency wait, it
// pulls this code into the instruction cache while memory is quiet (a first
// fetch under the full key stream costs several microseconds).  One copy of
// the code serves both calls.
__device__ __noinline__ SubCursor mma_chunk(uint32_t live, SubCursor cur, int nsub, uint32_t dbase, uint64_t ad,
                                            uint64_t bd, int ntile, int nacc) {
    constexpr uint32_t idesc = ptx::idesc_bf16_f32<BM, BN>();
    constexpr uint32_t kSubUnits = kSubBytes >> 4, kKbUnits = kBKbBytes >> 4, kKUnits = 32 >> 4;
    uint32_t dcol[kMaxGroup], boff[kMaxGroup], acc0[kMaxGroup];
#pragma unroll
    for (int j = 0; j < kMaxGroup; ++j) {
        dcol[j] = dbase + (uint32_t)((cur.tile * nacc + cur.kbm) * BN);
        boff[j] = (uint32_t)cur.kb * kKbUnits;
        acc0[j] = cur.kb >= nacc ? 1u : 0u;  // a partial's first k-block overwrites at its first k-step
        if (j < nsub && ++cur.tile == ntile) {
            cur.tile = 0;
            ++cur.kb;
            if (++cur.kbm == nacc) cur.kbm = 0;
        }
    }
#pragma unroll
    for (int k = 0; k < BK / 16; ++k) {
#pragma unroll
        for (int j = 0; j < kMaxGroup; ++j) {
            if (j < nsub)
                ptx::mma_bf16_if(live, dcol[j], ad + (uint64_t)(j * kSubUnits + k * kKUnits),
                                 bd + (uint64_t)(boff[j] + k * kKUnits), idesc, k != 0 ? 1u : acc0[j]);
        }
    }
    return cur;
}

// Top-k + softmax of one token; a single copy serves the warm-up call
// (prim_out == nullptr: nothing is written) and the real ones.
__device__ __noinline__ void topk_item(const float* z, int64_t P, int top_k, int lane, int64_t t, int32_t* prim_out,
                                       float* weight_out) {
    k3::topk_any(z, P, top_k, lane, t, prim_out, weight_out);
}
}  // namespace k3tc

__global__ void __launch_bounds__(k3tc::kThreads, 1)
    k3_score_tc(const uint8_t* __restrict__ keys_t, int64_t block_bytes, const __nv_bfloat16* __restrict__ q,
                int64_t P, int dk, int top_k, float scale, const WorkItem* __restrict__ work,
                const int32_t* __restrict__ counters, const int32_t* __restrict__ perm, int use_slots,
                int32_t* __restrict__ prim_out, float* __restrict__ weight_out, uint32_t* __restrict__ status,
                const __grid_constant__ k3tc::Geometry g) {
    using namespace k3tc;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* ring = smem;
    uint8_t* btile = smem + g.off_b;
    float* zs = reinterpret_cast<float*>(smem + g.off_z);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + g.off_bar);
    uint64_t* empty = full + kMaxStages;
    uint64_t* bfull = empty + kMaxStages;
    uint64_t* bempty = bfull + kBSlots;
    uint64_t* ifull = bempty + kBSlots;
    uint64_t* iempty = ifull + kISlots;
    uint64_t* dready = iempty + kISlots;
    uint64_t* tempty = dready + 2;
    uint64_t* drain = tempty + 2;
    WorkItem* items = reinterpret_cast<WorkItem*>(smem + g.off_meta);
    int32_t* toks = reinterpret_cast<int32_t*>(items + kISlots);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(toks + kISlots * kTok);
    volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int tid = threadIdx.x, lane = tid % 32, warp = tid / 32;
    pdl_trigger();
    // While the predecessor finishes, run the MMA issuer and the top-k once
    // without effect, so their code is cached before the key stream starts.
    if (warp == 1 && lane == 0) {
        SubCursor cur{0, 0, 0};
        for (int c = 0; c < min(g.chunks, 2); ++c) cur = mma_chunk(0u, cur, min(g.group, g.spi), 0u, 0ull, 0ull,
                                                                 g.ntile, g.nacc);
    } else if (warp >= 2 && warp < kBuildWarp) {
        topk_item(zs, P, top_k, lane, 0, nullptr, nullptr);
    }
    // The work list is the predecessor's output; TMEM is allocated only after
    // this wait, so a CTA that holds TMEM never waits on an earlier kernel.
    pdl_wait();
    const int n_work = counters[0];
    const int G = gridDim.x;
    const int my_items = n_work > (int)blockIdx.x ? (n_work - (int)blockIdx.x + G - 1) / G : 0;
    if (my_items == 0) return;  // uniform for the CTA: nothing allocated yet
    auto item_index = [&](int i) { return (int)blockIdx.x + i * G; };

    if (tid == 0) {
        for (int i = 0; i < g.n_stages; ++i) {
            ptx::mbar_init(&full[i], 1);
            ptx::mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < kBSlots; ++i) {
            ptx::mbar_init(&bfull[i], 1);
            ptx::mbar_init(&bempty[i], 1);
        }
        for (int i = 0; i < kISlots; ++i) {
            ptx::mbar_init(&ifull[i], 1);
            ptx::mbar_init(&iempty[i], kEpiWarps);
        }
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(&dready[i], 1);
            ptx::mbar_init(&tempty[i], kEpiWarps);
        }
        ptx::mbar_init(drain, 1);
        *abort = 0;
        ptx::fence_mbar_init();
    }
    if (warp == 1) ptx::tmem_alloc(tmem_slot, g.tmem_cols);
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        int64_t stage_seq = 0;  // copies issued
        int slot = 0;
        uint32_t phase = 0;
        bool ok = true;
        // Issues bulk copies [from, to) of item w's key block through the ring;
        // copy c holds sub-blocks [c * group, min(spi, (c + 1) * group)).
        auto issue_stages = [&](const WorkItem& w, int from, int to) {
            const uint8_t* blk = keys_t + (use_slots ? (int64_t)w.slot : (int64_t)w.scene) * block_bytes;
            for (int c = from; c < to && ok; ++c, ++stage_seq) {
                const uint32_t bytes = (uint32_t)(min(g.group, g.spi - c * g.group) * kSubBytes);
                if (lane == 0) {
                    ok = ptx::mbar_wait(&empty[slot], phase ^ 1u, abort, kTimeoutNs);
                    if (ok) {
                        ptx::mbar_arrive_expect_tx(&full[slot], bytes);
                        ptx::bulk_g2s(ring + (int64_t)slot * g.slot_bytes, blk + (int64_t)c * g.slot_bytes, bytes,
                                      &full[slot]);
                    }
                }
                ok = __shfl_sync(0xFFFFFFFFu, (int)ok, 0) != 0;
                if (++slot == g.n_stages) {
                    slot = 0;
                    phase ^= 1u;
                }
            }
        };
        // The work entry of the next item is loaded while this one's copies go out.
        WorkItem w = work[item_index(0)];
        for (int i = 0; i < my_items && ok; ++i) {
            WorkItem wn = w;
            if (i + 1 < my_items) wn = work[item_index(i + 1)];
            issue_stages(w, 0, g.chunks);
            w = wn;
        }
        if (!ok && lane == 0) {
            // Let every copy still in flight land before the CTA can exit.
            for (int64_t s = stage_seq - g.n_stages; s < stage_seq; ++s)
                if (s >= 0) ptx::mbar_wait_drain(&full[s % g.n_stages], (uint32_t)((s / g.n_stages) & 1), kTimeoutNs);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------- MMA
        if (lane == 0) {
            // Operand descriptors advance by adding 16-byte units to their start
            // address field (shared addresses stay below 2^18: no carry out of it).
            const uint64_t ad_ring = ptx::sw128_kmajor_desc(ptx::smem_u32(ring));
            const uint64_t bd_tiles = ptx::sw128_kmajor_desc(ptx::smem_u32(btile));
            int slot = 0;
            uint32_t phase = 0;
            bool ok = true;
            for (int i = 0; i < my_items && ok; ++i) {
                const int bs = i % kBSlots, d = i & 1;
                ok = ptx::mbar_wait(&bfull[bs], (i / kBSlots) & 1, abort, kTimeoutNs) &&
                     ptx::mbar_wait(&tempty[d], ((i >> 1) & 1) ^ 1, abort, kTimeoutNs);
                if (!ok) break;
                ptx::tc_fence_after();
                const uint32_t dbase = tmem_base + (uint32_t)(d * g.ntile * g.nacc * BN);
                const uint64_t bd = bd_tiles + (uint64_t)((bs * g.b_bytes) >> 4);
                SubCursor cur{0, 0, 0};
                for (int c = 0, done = 0; c < g.chunks; ++c) {
                    if (!(ok = ptx::mbar_wait(&full[slot], phase, abort, kTimeoutNs))) break;
                    ptx::tc_fence_after();
                    const int nsub = min(g.group, g.spi - done);
                    cur = mma_chunk(1u, cur, nsub, dbase, ad_ring + (uint64_t)((slot * g.slot_bytes) >> 4), bd,
                                    g.ntile, g.nacc);
                    ptx::mma_commit(&empty[slot]);
                    done += nsub;
                    if (++slot == g.n_stages) {
                        slot = 0;
                        phase ^= 1u;
                    }
                }
                if (ok) {
                    ptx::mma_commit(&bempty[bs]);
                    ptx::mma_commit(&dready[d]);
                }
            }
            // All MMAs complete before TMEM is released and the CTA exits.
            ptx::mma_commit(drain);
            ptx::mbar_wait_drain(drain, 0, kTimeoutNs);
        }
    } else if (warp < kBuildWarp) {
        // -------------------------------------------------------- epilogue
        const int e = warp - 2;           // 0..7
        const int quarter = warp & 3;     // TMEM lanes this warp may access
        const int half = e >> 2;          // the two warps of a quarter split the row tiles
        for (int i = 0; i < my_items; ++i) {
            const int ms = i % kISlots, d = i & 1;
            bool ok = ptx::mbar_wait(&ifull[ms], (i / kISlots) & 1, abort, kTimeoutNs) &&
                      ptx::mbar_wait(&dready[d], (i >> 1) & 1, abort, kTimeoutNs);
            ok = __all_sync(0xFFFFFFFFu, ok);
            // Also orders this item's logit writes after every warp's top-k of the previous item.
            if (k3tc::epi_sync_or(!ok || *abort)) break;
            const int nb = min(items[ms].count, kTok);
            ptx::tc_fence_after();
            for (int tile = half; tile < g.ntile; tile += 2) {
                float acc[kTok];
#pragma unroll
                for (int j = 0; j < kTok; ++j) acc[j] = 0.f;
                const uint32_t tbase = tmem_base + ((uint32_t)(quarter * 32) << 16) +
                                       (uint32_t)((d * g.ntile + tile) * g.nacc * BN);
                for (int a = 0; a < g.nacc; ++a) {
                    uint32_t r[16];
                    ptx::tmem_ld_32x32b_x16(tbase + (uint32_t)(a * BN), r);
                    ptx::tmem_wait_ld();
#pragma unroll
                    for (int j = 0; j < kTok; ++j) acc[j] += __uint_as_float(r[j]);
                }
                const int64_t p = (int64_t)tile * BM + quarter * 32 + lane;
                if (p < P) {
#pragma unroll
                    for (int j = 0; j < kTok; ++j)
                        if (j < nb) zs[j * P + p] = acc[j] * scale;
                }
            }
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&tempty[d]);
            if (k3tc::epi_sync_or(*abort)) break;  // all logits of the item are in shared memory
            for (int j = e; j < nb; j += kEpiWarps)
                k3tc::topk_item(zs + j * P, P, top_k, lane, toks[ms * kTok + j], prim_out, weight_out);
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&iempty[ms]);
        }
    } else {
        // ---------------------------------------------------- token tiles
        // Both tiles start zeroed; columns past d_k are never written again.
        for (int idx = lane; idx < kBSlots * g.b_bytes / 16; idx += 32)
            reinterpret_cast<uint4*>(btile)[idx] = make_uint4(0u, 0u, 0u, 0u);
        const int cpr = g.row_bytes / 16;  // 16-byte chunks per query row
        const uint4* qv = reinterpret_cast<const uint4*>(q);
        WorkItem w = work[item_index(0)];
        int32_t tok = lane < w.count ? perm[w.begin + lane] : 0;
        bool ok = true;
        for (int i = 0; i < my_items; ++i) {
            const int ms = i % kISlots, bs = i % kBSlots;
            if (lane == 0)
                ok = ptx::mbar_wait(&iempty[ms], ((i / kISlots) & 1) ^ 1, abort, kTimeoutNs) &&
                     ptx::mbar_wait(&bempty[bs], ((i / kBSlots) & 1) ^ 1, abort, kTimeoutNs);
            if (!__shfl_sync(0xFFFFFFFFu, (int)ok, 0)) break;
            const int nb = min(w.count, kTok);
            const int total = nb * cpr;
            uint8_t* bt = btile + bs * g.b_bytes;
            WorkItem wn = w;
            int32_t tokn = 0;
            for (int base = 0; base < total; base += 32 * kQBatch) {
                uint4 v[kQBatch];
                int jj[kQBatch], cc[kQBatch];
#pragma unroll
                for (int u = 0; u < kQBatch; ++u) {
                    const int idx = base + u * 32 + lane;
                    const bool valid = idx < total;
                    jj[u] = valid ? idx / cpr : 0;
                    cc[u] = valid ? idx - jj[u] * cpr : -1;
                    const int32_t tj = __shfl_sync(0xFFFFFFFFu, tok, jj[u]);
                    if (valid) v[u] = __ldg(qv + (int64_t)tj * cpr + cc[u]);
                }
                // The next work entry is read while the query rows are in flight.
                if (base == 0 && i + 1 < my_items) wn = work[item_index(i + 1)];
#pragma unroll
                for (int u = 0; u < kQBatch; ++u) {
                    if (cc[u] >= 0) {
                        const int j = jj[u], kb = cc[u] >> 3, c = cc[u] & 7;
                        *reinterpret_cast<uint4*>(bt + kb * kBKbBytes + j * 128 + ((c ^ (j & 7)) * 16)) = v[u];
                    }
                }
            }
            if (total == 0 && i + 1 < my_items) wn = work[item_index(i + 1)];
            if (i + 1 < my_items) tokn = lane < wn.count ? perm[wn.begin + lane] : 0;
            ptx::fence_proxy_async_smem();  // the tile is read by the tensor core (async proxy)
            if (lane < nb) toks[ms * kTok + lane] = tok;
            if (lane == 0) items[ms] = w;
            __syncwarp();
            if (lane == 0) {
                ptx::mbar_arrive(&ifull[ms]);
                ptx::mbar_arrive(&bfull[bs]);
            }
            w = wn;
            tok = tokn;
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem_base, g.tmem_cols);
    }
    if (tid == 0 && *abort) atomicOr(status, STATUS_WAIT_TIMEOUT);
}

bool score_tc_shape_supported(int64_t P, int dk) {
    const k3tc::Geometry g = k3tc::geometry(P, dk);
    return g.n_stages >= 2 && g.smem <= k3tc::kSmemLimit && g.tmem_cols <= 512 && (dk % 8) == 0;
}

int64_t score_tc_block_bytes(int64_t P, int dk) {
    const k3tc::Geometry g = k3tc::geometry(P, dk);
    return (int64_t)g.spi * k3tc::kSubBytes;
}

cudaError_t launch_score_tc(const LaunchCtx& c, const void* keys_tiled, const ScoreArgs& a) {
    const k3tc::Geometry g = k3tc::geometry(a.P, a.dk);
    if (!score_tc_shape_supported(a.P, a.dk)) return cudaErrorInvalidConfiguration;
    return launch_pdl(k3_score_tc, dim3(c.num_sms), dim3(k3tc::kThreads), (size_t)g.smem, c.stream,
                      (const uint8_t*)keys_tiled, (int64_t)g.spi * k3tc::kSubBytes, (const __nv_bfloat16*)a.q, a.P,
                      a.dk, a.top_k, a.scale, a.work, (const int32_t*)a.counters, a.perm, a.use_slots, a.prim_out,
                      a.weight_out, a.status, g);
}
cudaError_t configure_score_tc_kernel() {
    return cudaFuncSetAttribute(k3_score_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, k3tc::kSmemLimit);
}

}  // namespace lookme
