// Level 2 (Sec. "Level-2: scene-primitive retrieval", key-similarity form):
// for every token t routed to scene j,
//   z_tp = q_t . K[j, p] / sqrt(d_k)         for p < N_p
//   I_t  = top-k of z_t (larger z first, lower p on ties)
//   w_t  = softmax over z_t[I_t]
//
// The path is HBM-bound: a scene's key block (N_p x d_k) is read once per
// work item while a bucket holds only a few tokens, so the kernel keeps many
// bytes in flight and keeps dependent global reads and the top-k off the
// warps that consume the key stream.  One CTA per SM, three warp roles:
//   producer warp    takes work items from a global counter, reads the item's
//                    token ids, bulk-copies (cp.async.bulk) their query rows
//                    into an item slot and streams the scene's key block
//                    through a ring of 32 KiB stages; every copy completes on
//                    an mbarrier
//   8 compute warps  convert the item's queries to fp32, dot each key row
//                    with them (threads own key rows: TPR threads per row, 8 x
//                    16-byte chunks each, read in a lane-rotated order so
//                    eight consecutive lanes hit eight bank groups; the token
//                    loop is specialised on the bucket size), reduce across
//                    the row's threads with shuffles and write the logits
//                    into one of two logit buffers
//   4 top-k warps    one token per warp: top-k by repeated warp argmax
//                    (redux.sync on order-preserving keys, ties to the lower
//                    primitive), softmax, outputs; they run on buffer i while
//                    the compute warps fill buffer i+1
// Compute warps synchronise among themselves with a named barrier whose OR
// reduction makes the abort decision uniform; every wait is bounded.
#include "common.cuh"
#include "sm100.cuh"
#include "topk.cuh"

namespace lookme {

namespace k3 {
constexpr int kComputeWarps = 8;
constexpr int kCompute = kComputeWarps * 32;
constexpr int kTopkWarps = 4;
constexpr int kProducerWarp = kComputeWarps + kTopkWarps;
constexpr int kThreads = (kProducerWarp + 1) * 32;
constexpr int kTok = kTokensPerItem;
constexpr int kMaxItemSlots = 4;
constexpr int kMaxZBufs = 2;
constexpr int kStageBytes = 32768;
constexpr int kMaxStages = 6;
constexpr uint64_t kTimeoutNs = 1000000000ull;
constexpr int kSmemLimit = 227 * 1024;

struct Geometry {
    int row_bytes;        // d_k * element size
    int row_chunks;       // 16-byte chunks per key row
    int tpr;              // threads per key row (power of two)
    int rows_per_stage;   // key rows per ring stage
    int stages_per_item;  // ring stages per work item (covers N_p rows)
    int n_stages;         // ring depth
    int n_items;          // item slots (query rows + token ids)
    int n_z;              // logit buffers
    int qraw_bytes;       // one item slot of raw query rows
    int off_qraw, off_qf, off_z, off_bar, off_items;
    int smem;
};

inline Geometry geometry(int dtype, int64_t P, int dk) {
    Geometry g;
    const int esz = dtype == LOOKME_BF16 ? 2 : 4;
    g.row_bytes = dk * esz;
    g.row_chunks = g.row_bytes / 16;
    const int need = (g.row_chunks + 7) / 8;
    g.tpr = 1;
    while (g.tpr < need) g.tpr <<= 1;
    g.rows_per_stage = kCompute / g.tpr;
    g.stages_per_item = (int)((P + g.rows_per_stage - 1) / g.rows_per_stage);
    g.qraw_bytes = (kTok * g.row_bytes + 127) / 128 * 128;
    const int zbytes = kTok * (int)P * 4;
    // Deepest ring first; give up logit and item buffering only if the ring would be too shallow.
    const int plans[3][2] = {{kMaxItemSlots, kMaxZBufs}, {kMaxItemSlots, 1}, {2, 1}};
    for (int i = 0; i < 3; ++i) {
        g.n_items = plans[i][0];
        g.n_z = plans[i][1];
        const int fixed = g.n_items * g.qraw_bytes + kTok * dk * 4 + g.n_z * zbytes + 1024;
        g.n_stages = (kSmemLimit - fixed) / kStageBytes;
        if (g.n_stages > kMaxStages) g.n_stages = kMaxStages;
        if (g.n_stages >= 3) break;
    }
    g.off_qraw = g.n_stages * kStageBytes;
    g.off_qf = g.off_qraw + g.n_items * g.qraw_bytes;
    g.off_z = g.off_qf + kTok * dk * 4;
    g.off_bar = (g.off_z + g.n_z * zbytes + 7) / 8 * 8;
    g.off_items = g.off_bar + (2 * kMaxStages + 2 * kMaxItemSlots + 2 * kMaxZBufs) * 8;
    g.smem = g.off_items + kMaxItemSlots * ((int)sizeof(WorkItem) + kTok * 4) + 16;
    return g;
}

// Named barrier 1 over the compute warps, returning the OR of `v` over them.
__device__ __forceinline__ bool compute_sync_or(bool v) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.or.pred q, 1, %2, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)v), "n"(kCompute)
        : "memory");
    return r != 0;
}

// One ring stage: the logits of this thread's key row for the item's NB tokens.
template <typename T, int NB>
__device__ __forceinline__ void score_stage(const uint8_t* krow, const float* qf, const Geometry& g, int seg, int lane,
                                            int64_t row, int64_t P, float scale, float* zs) {
    constexpr int EPC = Vec16<T>::N;
    constexpr int H = EPC / 4;
    float a0[NB], a1[NB];
#pragma unroll
    for (int j = 0; j < NB; ++j) a0[j] = a1[j] = 0.f;
#pragma unroll
    for (int c = 0; c < 8; ++c) {
        const int ch = seg * 8 + ((c + lane) & 7);
        if (ch < g.row_chunks) {
            float kf[EPC];
            Vec16<T>::unpack(*reinterpret_cast<const uint4*>(krow + ch * 16), kf);
#pragma unroll
            for (int j = 0; j < NB; ++j) {
#pragma unroll
                for (int h = 0; h < H; ++h) {
                    const float4 qv = *reinterpret_cast<const float4*>(qf + ((j * H + h) * g.row_chunks + ch) * 4);
                    a0[j] = fmaf(kf[h * 4 + 0], qv.x, a0[j]);
                    a1[j] = fmaf(kf[h * 4 + 1], qv.y, a1[j]);
                    a0[j] = fmaf(kf[h * 4 + 2], qv.z, a0[j]);
                    a1[j] = fmaf(kf[h * 4 + 3], qv.w, a1[j]);
                }
            }
        }
    }
#pragma unroll
    for (int j = 0; j < NB; ++j) {
        float acc = a0[j] + a1[j];
        for (int o = g.tpr / 2; o; o >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, o);
        if (seg == 0 && row < P) zs[j * P + row] = acc * scale;
    }
}

}  // namespace k3

template <typename T>
__global__ void __launch_bounds__(k3::kThreads, 1)
    k3_score(const T* q, const T* __restrict__ keys, int64_t P, int dk, int top_k, float scale,
             const WorkItem* work, int32_t* counters, const int32_t* item_tok,
             int use_slots, int32_t* __restrict__ prim_out, float* __restrict__ weight_out,
             uint32_t* __restrict__ status, const __grid_constant__ k3::Geometry g) {
    using namespace k3;
    constexpr int EPC = Vec16<T>::N;
    constexpr int H = EPC / 4;
    extern __shared__ __align__(128) uint8_t smem[];
    uint8_t* ring = smem;
    uint8_t* qraw = smem + g.off_qraw;
    float* qf = reinterpret_cast<float*>(smem + g.off_qf);
    float* zbase = reinterpret_cast<float*>(smem + g.off_z);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + g.off_bar);
    uint64_t* empty = full + kMaxStages;
    uint64_t* ifull = empty + kMaxStages;
    uint64_t* iempty = ifull + kMaxItemSlots;
    uint64_t* zready = iempty + kMaxItemSlots;
    uint64_t* zfree = zready + kMaxZBufs;
    WorkItem* items = reinterpret_cast<WorkItem*>(smem + g.off_items);
    int32_t* toks = reinterpret_cast<int32_t*>(items + kMaxItemSlots);
    volatile int* abort = reinterpret_cast<volatile int*>(toks + kMaxItemSlots * kTok);

    const int tid = threadIdx.x, lane = tid % 32, warp = tid / 32;
    pdl_trigger();
    pdl_wait();
    const int n_work = counters[0];
    const int64_t zstride = (int64_t)kTok * P;

    if (tid == 0) {
        for (int i = 0; i < g.n_stages; ++i) {
            ptx::mbar_init(&full[i], 1);
            ptx::mbar_init(&empty[i], kComputeWarps);
        }
        for (int i = 0; i < g.n_items; ++i) {
            ptx::mbar_init(&ifull[i], 1);
            ptx::mbar_init(&iempty[i], kTopkWarps);
        }
        for (int i = 0; i < g.n_z; ++i) {
            ptx::mbar_init(&zready[i], kComputeWarps);
            ptx::mbar_init(&zfree[i], kTopkWarps);
        }
        *abort = 0;
        ptx::fence_mbar_init();
    }
    __syncthreads();

    if (warp == kProducerWarp) {
        // ------------------------------------------------------------ producer
        uint32_t item_seq = 0;
        int64_t stage_seq = 0;
        bool ok = true;
        for (;;) {
            int wi = 0;
            if (lane == 0) wi = atomicAdd(counters + 3, 1);
            wi = __shfl_sync(0xFFFFFFFFu, wi, 0);
            const int islot = (int)(item_seq % g.n_items);
            const uint32_t ipar = (item_seq / g.n_items) & 1u;
            if (lane == 0) ok = ptx::mbar_wait(&iempty[islot], ipar ^ 1u, abort, kTimeoutNs);
            if (!__shfl_sync(0xFFFFFFFFu, (int)ok, 0)) break;
            if (wi >= n_work) {
                if (lane == 0) {
                    items[islot].count = -1;  // end of work
                    ptx::mbar_arrive(&ifull[islot]);
                }
                break;
            }
            const WorkItem w = work[wi];
            int32_t t = 0;
            if (lane < w.count) {
                t = item_tok[w.begin + lane];
                toks[islot * kTok + lane] = t;
            }
            if (lane == 0) {
                items[islot] = w;
                ptx::mbar_arrive_expect_tx(&ifull[islot], (uint32_t)(w.count * g.row_bytes));
            }
            __syncwarp();
            if (lane < w.count)
                ptx::bulk_g2s(qraw + islot * g.qraw_bytes + lane * g.row_bytes,
                              reinterpret_cast<const uint8_t*>(q) + (int64_t)t * g.row_bytes, (uint32_t)g.row_bytes,
                              &ifull[islot]);
            const int64_t block = use_slots ? w.slot : w.scene;
            const uint8_t* src = reinterpret_cast<const uint8_t*>(keys) + block * P * (int64_t)g.row_bytes;
            for (int st = 0; st < g.stages_per_item; ++st, ++stage_seq) {
                const int slot = (int)(stage_seq % g.n_stages);
                const uint32_t par = (uint32_t)((stage_seq / g.n_stages) & 1);
                if (lane == 0) {
                    ok = ptx::mbar_wait(&empty[slot], par ^ 1u, abort, kTimeoutNs);
                    if (ok) {
                        const int64_t row0 = (int64_t)st * g.rows_per_stage;
                        const int64_t rows = min((int64_t)g.rows_per_stage, P - row0);
                        const uint32_t bytes = (uint32_t)(rows * g.row_bytes);
                        ptx::mbar_arrive_expect_tx(&full[slot], bytes);
                        ptx::bulk_g2s(ring + slot * kStageBytes, src + row0 * g.row_bytes, bytes, &full[slot]);
                    }
                }
                if (!__shfl_sync(0xFFFFFFFFu, (int)ok, 0)) break;
            }
            if (!ok) break;
            ++item_seq;
        }
        if (!ok && lane == 0) {
            // Let the copies still in flight land before the CTA can exit.
            for (int64_t s = stage_seq - g.n_stages; s < stage_seq; ++s)
                if (s >= 0) ptx::mbar_wait_drain(&full[s % g.n_stages], (uint32_t)((s / g.n_stages) & 1), kTimeoutNs);
            for (uint32_t s = item_seq >= (uint32_t)g.n_items ? item_seq - g.n_items + 1 : 0; s <= item_seq; ++s)
                ptx::mbar_wait_drain(&ifull[s % g.n_items], (s / g.n_items) & 1u, kTimeoutNs);
            atomicOr(status, STATUS_WAIT_TIMEOUT | STATUS_IN_SCORE);
        }
        return;
    }

    if (warp >= kComputeWarps) {
        // ------------------------------------------------------- top-k warps
        const int tw = warp - kComputeWarps;
        for (uint32_t item_seq = 0;; ++item_seq) {
            const int islot = (int)(item_seq % g.n_items);
            const int zb = (int)(item_seq % g.n_z);
            if (!ptx::mbar_wait(&ifull[islot], (item_seq / g.n_items) & 1u, abort, kTimeoutNs)) break;
            const int count = items[islot].count;
            if (count < 0) break;
            if (!ptx::mbar_wait(&zready[zb], (item_seq / g.n_z) & 1u, abort, kTimeoutNs)) break;
            const float* zs = zbase + zb * zstride;
            for (int j = tw; j < min(count, kTok); j += kTopkWarps)
                topk_any(zs + j * P, P, top_k, lane, toks[islot * kTok + j], prim_out, weight_out);
            __syncwarp();
            if (lane == 0) {
                ptx::mbar_arrive(&zfree[zb]);
                ptx::mbar_arrive(&iempty[islot]);
            }
        }
        return;
    }

    // ------------------------------------------------------------ compute warps
    const int r_in_stage = tid / g.tpr;
    const int seg = tid % g.tpr;
    int64_t stage_seq = 0;
    for (uint32_t item_seq = 0;; ++item_seq) {
        const int islot = (int)(item_seq % g.n_items);
        const int zb = (int)(item_seq % g.n_z);
        ptx::mbar_wait(&ifull[islot], (item_seq / g.n_items) & 1u, abort, kTimeoutNs);
        if (compute_sync_or(*abort != 0)) break;
        const WorkItem w = items[islot];
        if (w.count < 0) break;
        const int nb = min(w.count, kTok);

        // Queries of the item's tokens -> fp32, layout [token][half][chunk][4].
        const T* qr = reinterpret_cast<const T*>(qraw + islot * g.qraw_bytes);
        for (int i = tid; i < nb * dk; i += kCompute) {
            const int j = i / dk, e = i - j * dk;
            const int ch = e / EPC, h = (e % EPC) / 4;
            qf[((j * H + h) * g.row_chunks + ch) * 4 + (e & 3)] = to_f32(qr[j * dk + e]);
        }
        // The logit buffer must have been released by the top-k warps.
        ptx::mbar_wait(&zfree[zb], ((item_seq / g.n_z) & 1u) ^ 1u, abort, kTimeoutNs);
        compute_sync_or(false);

        float* zs = zbase + zb * zstride;
        for (int st = 0; st < g.stages_per_item; ++st, ++stage_seq) {
            const int slot = (int)(stage_seq % g.n_stages);
            if (ptx::mbar_wait(&full[slot], (uint32_t)((stage_seq / g.n_stages) & 1), abort, kTimeoutNs)) {
                const uint8_t* krow = ring + slot * kStageBytes + r_in_stage * g.row_bytes;
                const int64_t row = (int64_t)st * g.rows_per_stage + r_in_stage;
                switch (nb) {
                    case 1: score_stage<T, 1>(krow, qf, g, seg, lane, row, P, scale, zs); break;
                    case 2: score_stage<T, 2>(krow, qf, g, seg, lane, row, P, scale, zs); break;
                    case 3: score_stage<T, 3>(krow, qf, g, seg, lane, row, P, scale, zs); break;
                    case 4: score_stage<T, 4>(krow, qf, g, seg, lane, row, P, scale, zs); break;
                    case 5: score_stage<T, 5>(krow, qf, g, seg, lane, row, P, scale, zs); break;
                    case 6: score_stage<T, 6>(krow, qf, g, seg, lane, row, P, scale, zs); break;
                    case 7: score_stage<T, 7>(krow, qf, g, seg, lane, row, P, scale, zs); break;
                    default: score_stage<T, 8>(krow, qf, g, seg, lane, row, P, scale, zs); break;
                }
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&empty[slot]);
        }
        // All logits written (and qf free for the next item) before the top-k warps read them.
        if (compute_sync_or(*abort != 0)) break;
        if (lane == 0) ptx::mbar_arrive(&zready[zb]);
    }
}

bool score_shape_supported(int dtype, int64_t P, int dk) {
    const k3::Geometry g = k3::geometry(dtype, P, dk);
    return g.tpr <= 32 && g.n_stages >= 2 && g.smem <= k3::kSmemLimit &&
           g.rows_per_stage * g.row_bytes <= k3::kStageBytes;
}

cudaError_t launch_score(const LaunchCtx& c, const ScoreArgs& a) {
    const k3::Geometry g = k3::geometry(a.dtype, a.P, a.dk);
    if (g.n_stages < 2 || g.smem > k3::kSmemLimit) return cudaErrorInvalidConfiguration;
    if (a.dtype == LOOKME_BF16)
        return launch_pdl(k3_score<__nv_bfloat16>, dim3(c.num_sms), dim3(k3::kThreads), (size_t)g.smem, c.stream,
                          (const __nv_bfloat16*)a.q, (const __nv_bfloat16*)a.keys, a.P, a.dk, a.top_k, a.scale, a.work,
                          a.counters, a.item_tok, a.use_slots, a.prim_out, a.weight_out, a.status, g);
    return launch_pdl(k3_score<float>, dim3(c.num_sms), dim3(k3::kThreads), (size_t)g.smem, c.stream,
                      (const float*)a.q, (const float*)a.keys, a.P, a.dk, a.top_k, a.scale, a.work, a.counters, a.item_tok,
                      a.use_slots, a.prim_out, a.weight_out, a.status, g);
}

cudaError_t configure_score_kernels() {
    cudaError_t e = cudaFuncSetAttribute(k3_score<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         k3::kSmemLimit);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(k3_score<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, k3::kSmemLimit);
}

}  // namespace lookme
