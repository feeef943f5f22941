// Level 2 on the 5th-generation tensor cores (bf16 tables), Sec. "Level-2:
// scene-primitive retrieval" in its key-similarity form:
//   z_tp = q_t . K[j, p] / sqrt(d_k), I_t = top-k of z_t, w_t = softmax(z_t[I_t]).
//
// Each work item (a scene and <= 8 of its tokens) is a small grouped GEMM:
// D[p][j] = K[scene, p, :] . q_j for the scene's N_p key rows and the item's
// tokens.  The keys are the M = 128 operand (one TMA box of 128 rows x 64
// columns, 128-byte swizzle, per ring stage), the tokens the N = 16 operand
// (a swizzled K-major tile built in shared memory from bulk-copied query
// rows), and the fp32 accumulator lives in TMEM.  The kernel stays
// HBM-bound: the tensor core removes the CUDA-core work that would otherwise
// have to keep pace with the key stream.  One CTA per SM:
//   warp 0       producer: static share of the work list, prefetches the
//                next item's header and query rows, converts query rows into
//                the token tile, streams key k-blocks through the ring
//   warp 1       one thread issues tcgen05.mma into one of two TMEM buffers
//   warps 2..5   epilogue: TMEM -> logits in shared memory (scaled), then
//                top-k + softmax, one token per warp (redux.sync argmax)
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
constexpr int kStageBytes = BM * 128;    // one 128 x 64 key block: 16 KiB
constexpr int kBKbBytes = BN * 128;      // one 16 x 64 token block: 2 KiB
constexpr int kEpiWarps = 4;
constexpr int kThreads = (2 + kEpiWarps) * 32;
constexpr int kMaxStages = 14;
constexpr int kBSlots = 2;               // token tiles
constexpr int kISlots = 4;               // item metadata (scene, count, token ids)
constexpr int kQSlots = 2;               // raw query rows
constexpr uint64_t kTimeoutNs = 1000000000ull;
constexpr int kSmemLimit = 227 * 1024;

struct Geometry {
    int nkb;              // 64-wide k-blocks of d_k
    int ntile;            // 128-row tiles of N_p
    int n_stages;         // ring depth
    int row_bytes;        // d_k * 2
    int qraw_bytes;       // one slot of raw query rows
    int b_bytes;          // one token tile (nkb x 2 KiB)
    int tmem_cols;        // allocated TMEM columns (two accumulators of ntile x 16)
    int off_b, off_qraw, off_z, off_bar, off_meta;
    int smem;             // bytes requested, including 1 KiB of alignment slack
};

inline Geometry geometry(int64_t P, int dk) {
    Geometry g;
    g.nkb = (dk + BK - 1) / BK;
    g.ntile = (int)((P + BM - 1) / BM);
    g.row_bytes = dk * 2;
    g.qraw_bytes = (kTok * g.row_bytes + 127) / 128 * 128;
    g.b_bytes = g.nkb * kBKbBytes;
    int cols = 32;
    while (cols < 2 * g.ntile * BN) cols <<= 1;
    g.tmem_cols = cols;
    const int zbytes = (kTok * (int)P * 4 + 15) / 16 * 16;
    const int fixed = kBSlots * g.b_bytes + kQSlots * g.qraw_bytes + zbytes + 1024 /*bar+meta*/ + 1024 /*align*/;
    g.n_stages = (kSmemLimit - fixed) / kStageBytes;
    if (g.n_stages > kMaxStages) g.n_stages = kMaxStages;
    g.off_b = g.n_stages * kStageBytes;
    g.off_qraw = g.off_b + kBSlots * g.b_bytes;
    g.off_z = g.off_qraw + kQSlots * g.qraw_bytes;
    g.off_bar = g.off_z + zbytes;
    g.off_meta = g.off_bar + (2 * kMaxStages + 2 * kBSlots + 2 * kISlots + kQSlots + 2 * 2 + 1) * 8;
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
}  // namespace k3tc

__global__ void __launch_bounds__(k3tc::kThreads, 1)
    k3_score_tc(const __grid_constant__ CUtensorMap tmap_keys, const __nv_bfloat16* __restrict__ q, int64_t P,
                int dk, int top_k, float scale, const WorkItem* __restrict__ work,
                const int32_t* __restrict__ counters, const int32_t* __restrict__ perm, int use_slots,
                int32_t* __restrict__ prim_out, float* __restrict__ weight_out, uint32_t* __restrict__ status,
                const __grid_constant__ k3tc::Geometry g) {
    using namespace k3tc;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* ring = smem;
    uint8_t* btile = smem + g.off_b;
    uint8_t* qraw = smem + g.off_qraw;
    float* zs = reinterpret_cast<float*>(smem + g.off_z);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + g.off_bar);
    uint64_t* empty = full + kMaxStages;
    uint64_t* bfull = empty + kMaxStages;
    uint64_t* bempty = bfull + kBSlots;
    uint64_t* ifull = bempty + kBSlots;
    uint64_t* iempty = ifull + kISlots;
    uint64_t* qfull = iempty + kISlots;
    uint64_t* dready = qfull + kQSlots;
    uint64_t* tempty = dready + 2;
    uint64_t* drain = tempty + 2;
    WorkItem* items = reinterpret_cast<WorkItem*>(smem + g.off_meta);
    int32_t* toks = reinterpret_cast<int32_t*>(items + kISlots);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(toks + kISlots * kTok);
    volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int tid = threadIdx.x, lane = tid % 32, warp = tid / 32;
    if (tid == 0) ptx::prefetch_tmap(&tmap_keys);
    pdl_trigger();
    // The work list is the predecessor's output; TMEM is allocated only after
    // this wait, so a CTA that holds TMEM never waits on an earlier kernel.
    pdl_wait();
    const int n_work = counters[0];
    const int G = gridDim.x;
    const int my_items = n_work > (int)blockIdx.x ? (n_work - (int)blockIdx.x + G - 1) / G : 0;
    if (my_items == 0) return;  // uniform for the CTA: nothing allocated yet

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
        for (int i = 0; i < kQSlots; ++i) ptx::mbar_init(&qfull[i], 1);
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
        auto item_index = [&](int i) { return (int)blockIdx.x + i * G; };
        // Query rows of item i -> raw slot i % kQSlots (bulk copies on qfull).
        auto issue_q = [&](int i, const WorkItem& w, int32_t tok) {
            const int s = i % kQSlots;
            if (lane == 0) ptx::mbar_arrive_expect_tx(&qfull[s], (uint32_t)(w.count * g.row_bytes));
            __syncwarp();
            if (lane < w.count)
                ptx::bulk_g2s(qraw + s * g.qraw_bytes + lane * g.row_bytes,
                              reinterpret_cast<const uint8_t*>(q) + (int64_t)tok * g.row_bytes, (uint32_t)g.row_bytes,
                              &qfull[s]);
        };
        // Item headers run two items ahead of the key stream: the work entry and
        // token ids of item i+2 are loaded while item i streams, and the query
        // rows of item i+1 are copied before item i's key blocks are issued.
        auto load_header = [&](int i, WorkItem& w, int32_t& tok) {
            if (i < my_items) {
                w = work[item_index(i)];
                tok = lane < w.count ? perm[w.begin + lane] : 0;
            }
        };
        int64_t stage_seq = 0;
        bool ok = true;
        const int spi = g.ntile * g.nkb;  // key blocks per item, tile-major then k-block
        // Issues key blocks [from, to) of item w through the ring.
        auto issue_stages = [&](const WorkItem& w, int from, int to) {
            const int32_t row_base = (int32_t)((use_slots ? (int64_t)w.slot : (int64_t)w.scene) * P);
            for (int st = from; st < to && ok; ++st, ++stage_seq) {
                const int tile = st / g.nkb, kb = st - tile * g.nkb;
                const int slot = (int)(stage_seq % g.n_stages);
                const uint32_t par = (uint32_t)((stage_seq / g.n_stages) & 1);
                if (lane == 0) {
                    ok = ptx::mbar_wait(&empty[slot], par ^ 1u, abort, kTimeoutNs);
                    if (ok) {
                        ptx::mbar_arrive_expect_tx(&full[slot], (uint32_t)kStageBytes);
                        ptx::tma_load_2d(ring + slot * kStageBytes, &tmap_keys, kb * BK, row_base + tile * BM,
                                         &full[slot]);
                    }
                }
                ok = __shfl_sync(0xFFFFFFFFu, (int)ok, 0) != 0;
            }
        };
        WorkItem w, w1, w2;
        int32_t tok = 0, tok1 = 0, tok2 = 0;
        w.count = w1.count = w2.count = 0;
        load_header(0, w, tok);
        issue_q(0, w, tok);
        // The first item's first key blocks do not wait for its query rows; the
        // rest follow once its token tile is published (each TMA issue of a
        // 16 KiB block occupies the issuing thread for a few hundred ns).
        const int pre_issued = min(spi, 2);
        issue_stages(w, 0, pre_issued);
        int q_issued = 1;
        for (int i = 0; i < my_items && ok; ++i) {
            const int ms = i % kISlots, bs = i % kBSlots, qs = i % kQSlots;
            if (lane == 0)
                ok = ptx::mbar_wait(&iempty[ms], ((i / kISlots) & 1) ^ 1, abort, kTimeoutNs) &&
                     ptx::mbar_wait(&bempty[bs], ((i / kBSlots) & 1) ^ 1, abort, kTimeoutNs);
            ok = __shfl_sync(0xFFFFFFFFu, (int)ok, 0) != 0;
            // Every lane observes the query rows' completion before reading them.
            ok = ok && ptx::mbar_wait(&qfull[qs], (i / kQSlots) & 1, abort, kTimeoutNs);
            if (!__all_sync(0xFFFFFFFFu, ok)) {
                ok = false;
                break;
            }
            // Token tile: row j, 16-byte chunk c of k-block kb goes to chunk c ^ (j & 7)
            // of the row (the 128-byte swizzle the MMA descriptor names); zero past d_k.
            const uint8_t* qr = qraw + qs * g.qraw_bytes;
            uint8_t* bt = btile + bs * g.b_bytes;
            const int chunks = w.count * g.nkb * 8;
            for (int idx = lane; idx < chunks; idx += 32) {
                const int j = idx / (g.nkb * 8), rem = idx - j * g.nkb * 8;
                const int kb = rem / 8, c = rem & 7;
                const int col = kb * 8 + c;  // 16-byte chunk of the row
                uint4 v = make_uint4(0u, 0u, 0u, 0u);
                if (col * 16 < g.row_bytes) v = *reinterpret_cast<const uint4*>(qr + j * g.row_bytes + col * 16);
                *reinterpret_cast<uint4*>(bt + kb * kBKbBytes + j * 128 + ((c ^ (j & 7)) * 16)) = v;
            }
            ptx::fence_proxy_async_smem();
            if (lane < w.count) toks[ms * kTok + lane] = tok;
            if (lane == 0) items[ms] = w;
            __syncwarp();
            if (lane == 0) {
                ptx::mbar_arrive(&ifull[ms]);
                ptx::mbar_arrive(&bfull[bs]);
            }
            // Next item's query rows (its raw slot was converted one item ago).
            if (i == 0) load_header(1, w1, tok1);  // after item 0 is published, off its critical path
            if (i + 1 < my_items) {
                issue_q(i + 1, w1, tok1);
                ++q_issued;
            }
            // Work entry of item i+2; its token ids are read after the key stream.
            if (i + 2 < my_items) w2 = work[item_index(i + 2)];
            // Key blocks of the item (item 0's first blocks went out before the loop).
            issue_stages(w, i == 0 ? pre_issued : 0, spi);
            if (i + 2 < my_items) tok2 = lane < w2.count ? perm[w2.begin + lane] : 0;
            w = w1;
            tok = tok1;
            w1 = w2;
            tok1 = tok2;
        }
        if (!ok && lane == 0) {
            // Let every copy still in flight land before the CTA can exit.
            for (int64_t s = stage_seq - g.n_stages; s < stage_seq; ++s)
                if (s >= 0) ptx::mbar_wait_drain(&full[s % g.n_stages], (uint32_t)((s / g.n_stages) & 1), kTimeoutNs);
            for (int s = q_issued - kQSlots; s < q_issued; ++s)
                if (s >= 0) ptx::mbar_wait_drain(&qfull[s % kQSlots], (s / kQSlots) & 1, kTimeoutNs);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------- MMA
        if (lane == 0) {
            constexpr uint32_t idesc = ptx::idesc_bf16_f32<BM, BN>();
            int64_t stage_seq = 0;
            bool ok = true;
            for (int i = 0; i < my_items && ok; ++i) {
                const int bs = i % kBSlots, d = i & 1;
                ok = ptx::mbar_wait(&bfull[bs], (i / kBSlots) & 1, abort, kTimeoutNs) &&
                     ptx::mbar_wait(&tempty[d], ((i >> 1) & 1) ^ 1, abort, kTimeoutNs);
                if (!ok) break;
                ptx::tc_fence_after();
                const uint32_t dbase = tmem_base + (uint32_t)(d * g.ntile * BN);
                const uint32_t b0 = ptx::smem_u32(btile + bs * g.b_bytes);
                for (int tile = 0; tile < g.ntile && ok; ++tile) {
                    for (int kb = 0; kb < g.nkb; ++kb, ++stage_seq) {
                        const int slot = (int)(stage_seq % g.n_stages);
                        if (!(ok = ptx::mbar_wait(&full[slot], (uint32_t)((stage_seq / g.n_stages) & 1), abort,
                                                  kTimeoutNs)))
                            break;
                        ptx::tc_fence_after();
                        const uint32_t a0 = ptx::smem_u32(ring + slot * kStageBytes);
#pragma unroll
                        for (int k = 0; k < BK / 16; ++k)
                            ptx::mma_bf16(dbase + (uint32_t)(tile * BN), ptx::sw128_kmajor_desc(a0 + k * 32),
                                          ptx::sw128_kmajor_desc(b0 + kb * kBKbBytes + k * 32), idesc,
                                          (kb | k) != 0);
                        ptx::mma_commit(&empty[slot]);
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
    } else {
        // -------------------------------------------------------- epilogue
        const int e = warp - 2;           // 0..3
        const int quarter = warp & 3;     // TMEM lanes this warp may access
        for (int i = 0; i < my_items; ++i) {
            const int ms = i % kISlots, d = i & 1;
            bool ok = ptx::mbar_wait(&ifull[ms], (i / kISlots) & 1, abort, kTimeoutNs) &&
                      ptx::mbar_wait(&dready[d], (i >> 1) & 1, abort, kTimeoutNs);
            ok = __all_sync(0xFFFFFFFFu, ok);
            // Also orders this item's logit writes after every warp's top-k of the previous item.
            if (k3tc::epi_sync_or(!ok || *abort)) break;
            const int nb = min(items[ms].count, kTok);
            ptx::tc_fence_after();
            for (int tile = 0; tile < g.ntile; ++tile) {
                uint32_t r[16];
                ptx::tmem_ld_32x32b_x16(
                    tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(d * g.ntile * BN + tile * BN), r);
                ptx::tmem_wait_ld();
                const int64_t p = (int64_t)tile * BM + quarter * 32 + lane;
                if (p < P) {
#pragma unroll
                    for (int j = 0; j < kTok; ++j)
                        if (j < nb) zs[j * P + p] = __uint_as_float(r[j]) * scale;
                }
            }
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&tempty[d]);
            if (k3tc::epi_sync_or(*abort)) break;  // all logits of the item are in shared memory
            for (int j = e; j < nb; j += kEpiWarps)
                k3::topk_any(zs + j * P, P, top_k, lane, toks[ms * kTok + j], prim_out, weight_out);
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&iempty[ms]);
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
    return g.n_stages >= 4 && g.smem <= k3tc::kSmemLimit && g.tmem_cols <= 512 && (dk % 8) == 0;
}

cudaError_t launch_score_tc(const LaunchCtx& c, const void* tmap_keys, const ScoreArgs& a) {
    const k3tc::Geometry g = k3tc::geometry(a.P, a.dk);
    if (!score_tc_shape_supported(a.P, a.dk)) return cudaErrorInvalidConfiguration;
    CUtensorMap mk;
    memcpy(&mk, tmap_keys, sizeof(CUtensorMap));
    return launch_pdl(k3_score_tc, dim3(c.num_sms), dim3(k3tc::kThreads), (size_t)g.smem, c.stream, mk,
                      (const __nv_bfloat16*)a.q, a.P, a.dk, a.top_k, a.scale, a.work, (const int32_t*)a.counters, a.perm,
                      a.use_slots, a.prim_out, a.weight_out, a.status, g);
}

cudaError_t configure_score_tc_kernel() {
    return cudaFuncSetAttribute(k3_score_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, k3tc::kSmemLimit);
}

}  // namespace lookme
