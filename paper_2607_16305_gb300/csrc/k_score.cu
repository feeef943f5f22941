// Level 2 (Sec. "Level-2: scene-primitive retrieval", key-similarity form):
// for every token t routed to scene j,
//   z_tp = q_t . K[j, p] / sqrt(d_k)         for p < N_p
//   I_t  = top-k of z_t (larger z first, lower p on ties)
//   w_t  = softmax over z_t[I_t]
//
// The path is HBM-bound: a scene's key block (N_p x d_k) is read once per
// work item while a bucket holds only a few tokens.  Each CTA walks a static
// share of the work list; one thread streams the key blocks into a ring of
// shared-memory stages with cp.async.bulk (completion on mbarriers) and runs
// ahead across work items, so the next item's keys are in flight while the
// current item finishes its top-k.  Threads own key rows (TPR threads per
// row, 8 x 16-byte chunks each), read their chunks in a lane-rotated order so
// that eight consecutive lanes hit eight different bank groups, dot them with
// the (broadcast) fp32 queries of the item's tokens, and reduce across the
// TPR lanes with shuffles.  Logits land in shared memory; one warp per token
// then extracts the top-k and the softmax weights.
#include "common.cuh"
#include "sm100.cuh"

namespace lookme {

namespace k3 {
constexpr int kThreads = 256;
constexpr int kTok = kTokensPerItem;  // tokens per work item == warps per CTA
constexpr int kStages = 3;
constexpr int kStageBytes = 32768;
constexpr uint64_t kTimeoutNs = 1000000000ull;

struct Geometry {
    int row_bytes;       // d_k * element size
    int row_chunks;      // 16-byte chunks per key row
    int tpr;             // threads per key row (power of two)
    int rows_per_stage;  // key rows per ring stage
    int stages_per_item; // ring stages per work item (covers N_p rows)
    int q_floats;        // floats of the per-item query buffer
    int z_floats;        // floats of the per-item logit buffer
    int smem;            // dynamic shared memory bytes
};

inline Geometry geometry(int dtype, int64_t P, int dk) {
    Geometry g;
    const int esz = dtype == LOOKME_BF16 ? 2 : 4;
    g.row_bytes = dk * esz;
    g.row_chunks = g.row_bytes / 16;
    const int need = (g.row_chunks + 7) / 8;
    g.tpr = 1;
    while (g.tpr < need) g.tpr <<= 1;
    g.rows_per_stage = kThreads / g.tpr;
    g.stages_per_item = (int)((P + g.rows_per_stage - 1) / g.rows_per_stage);
    g.q_floats = kTok * dk;
    g.z_floats = kTok * (int)P;
    g.smem = kStages * kStageBytes + (g.q_floats + g.z_floats) * 4 + kStages * 8 + 16;
    return g;
}
}  // namespace k3

template <typename T>
__global__ void __launch_bounds__(k3::kThreads, 2)
    k3_score(const T* __restrict__ q, const T* __restrict__ keys, int64_t P, int dk, int top_k, float scale,
             const WorkItem* __restrict__ work, const int32_t* __restrict__ n_work_ptr,
             const int32_t* __restrict__ perm, int use_slots, int32_t* __restrict__ prim_out,
             float* __restrict__ weight_out, uint32_t* __restrict__ status, k3::Geometry g) {
    using namespace k3;
    constexpr int EPC = Vec16<T>::N;   // elements per 16-byte chunk
    constexpr int H = EPC / 4;         // 16-byte halves of a chunk's fp32 query values
    extern __shared__ __align__(128) uint8_t smem[];
    uint8_t* ring = smem;
    float* qs = reinterpret_cast<float*>(ring + kStages * kStageBytes);
    float* zs = qs + g.q_floats;
    uint64_t* full = reinterpret_cast<uint64_t*>(zs + g.z_floats);
    volatile int* abort = reinterpret_cast<volatile int*>(full + kStages);

    const int tid = threadIdx.x, lane = tid % 32, warp = tid / 32;
    const int n_work = *n_work_ptr;
    const int G = gridDim.x;
    const int my_items = n_work > (int)blockIdx.x ? (n_work - (int)blockIdx.x + G - 1) / G : 0;
    if (my_items == 0) return;
    const int64_t total_stages = (int64_t)my_items * g.stages_per_item;

    if (tid == 0) {
        for (int i = 0; i < kStages; ++i) ptx::mbar_init(&full[i], 1);
        *abort = 0;
        ptx::fence_mbar_init();
    }
    __syncthreads();

    // Producer: ring stage `gs` (counted over this CTA's whole item sequence).
    auto issue = [&](int64_t gs) {
        const int it = (int)(gs / g.stages_per_item);
        const int st = (int)(gs % g.stages_per_item);
        const WorkItem w = work[blockIdx.x + (int64_t)it * G];
        const int64_t block = use_slots ? w.slot : w.scene;
        const int64_t row0 = (int64_t)st * g.rows_per_stage;
        const int64_t rows = min((int64_t)g.rows_per_stage, P - row0);
        const uint32_t bytes = (uint32_t)(rows * g.row_bytes);
        const int slot = (int)(gs % kStages);
        ptx::mbar_arrive_expect_tx(&full[slot], bytes);
        const uint8_t* src = reinterpret_cast<const uint8_t*>(keys) + (block * P + row0) * (int64_t)g.row_bytes;
        ptx::bulk_g2s(ring + slot * kStageBytes, src, bytes, &full[slot]);
    };
    if (tid == 0)
        for (int64_t gs = 0; gs < total_stages && gs < kStages; ++gs) issue(gs);

    const int r_in_stage = tid / g.tpr;
    const int seg = tid % g.tpr;
    int64_t gs = 0;
    bool ok = true;
    for (int it = 0; it < my_items && ok; ++it) {
        const WorkItem w = work[blockIdx.x + (int64_t)it * G];
        const int nb = w.count;
        // Queries of the item's tokens -> fp32, layout [token][half][chunk][4].
        for (int i = tid; i < nb * dk; i += kThreads) {
            const int j = i / dk, e = i % dk;
            const int32_t t = perm[w.begin + j];
            const int ch = e / EPC, h = (e % EPC) / 4;
            qs[((j * H + h) * g.row_chunks + ch) * 4 + (e & 3)] = to_f32(q[(int64_t)t * dk + e]);
        }
        __syncthreads();

        for (int st = 0; st < g.stages_per_item; ++st, ++gs) {
            const int slot = (int)(gs % kStages);
            if (!ptx::mbar_wait(&full[slot], (uint32_t)((gs / kStages) & 1), abort, kTimeoutNs)) {
                ok = false;
            }
            __syncthreads();
            if (*abort) {
                ok = false;
                break;
            }
            const uint8_t* krow = ring + slot * kStageBytes + r_in_stage * g.row_bytes;
            float acc[kTok];
#pragma unroll
            for (int j = 0; j < kTok; ++j) acc[j] = 0.f;
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                const int ch = seg * 8 + ((c + lane) & 7);
                if (ch < g.row_chunks) {
                    float kf[EPC];
                    Vec16<T>::unpack(*reinterpret_cast<const uint4*>(krow + ch * 16), kf);
#pragma unroll
                    for (int j = 0; j < kTok; ++j) {
                        if (j < nb) {
#pragma unroll
                            for (int h = 0; h < H; ++h) {
                                const float4 qv =
                                    *reinterpret_cast<const float4*>(qs + ((j * H + h) * g.row_chunks + ch) * 4);
                                acc[j] = fmaf(kf[h * 4 + 0], qv.x, acc[j]);
                                acc[j] = fmaf(kf[h * 4 + 1], qv.y, acc[j]);
                                acc[j] = fmaf(kf[h * 4 + 2], qv.z, acc[j]);
                                acc[j] = fmaf(kf[h * 4 + 3], qv.w, acc[j]);
                            }
                        }
                    }
                }
            }
#pragma unroll
            for (int j = 0; j < kTok; ++j) {
                if (j < nb) {
                    for (int o = g.tpr / 2; o; o >>= 1) acc[j] += __shfl_xor_sync(0xFFFFFFFFu, acc[j], o);
                }
            }
            const int64_t row = (int64_t)st * g.rows_per_stage + r_in_stage;
            if (seg == 0 && row < P) {
#pragma unroll
                for (int j = 0; j < kTok; ++j)
                    if (j < nb) zs[j * P + row] = acc[j] * scale;
            }
            __syncthreads();  // the slot is free and the logits are visible
            if (tid == 0 && gs + kStages < total_stages) issue(gs + kStages);
        }
        if (!ok) break;

        // Top-k and softmax: warp j handles token j of the item.
        if (warp < nb) {
            const float* z = zs + warp * P;
            uint64_t taken = 0ull;  // bit i: element lane + 32 i already selected
            float my_z[2] = {0.f, 0.f};  // output slots lane and lane + 32
            int my_p[2] = {0, 0};
            for (int kk = 0; kk < top_k; ++kk) {
                float bz = 0.f;
                int bp = -1;
                int i = 0;
                for (int64_t p = lane; p < P; p += 32, ++i) {
                    if (!((taken >> i) & 1ull)) {
                        const float zz = z[p];
                        if (bp < 0 || zz > bz) {
                            bz = zz;
                            bp = (int)p;
                        }
                    }
                }
#pragma unroll
                for (int o = 16; o; o >>= 1) {
                    const float oz = __shfl_xor_sync(0xFFFFFFFFu, bz, o);
                    const int op = __shfl_xor_sync(0xFFFFFFFFu, bp, o);
                    if (op >= 0 && (bp < 0 || oz > bz || (oz == bz && op < bp))) {
                        bz = oz;
                        bp = op;
                    }
                }
                if (bp >= 0 && (bp & 31) == lane) taken |= 1ull << (bp >> 5);
                if ((kk & 31) == lane) {
                    my_z[kk >> 5] = bz;
                    my_p[kk >> 5] = bp;
                }
            }
            const float zmax = __shfl_sync(0xFFFFFFFFu, my_z[0], 0);
            float e[2];
            float sum = 0.f;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                e[h] = (h * 32 + lane < top_k) ? expf(my_z[h] - zmax) : 0.f;
                sum += e[h];
            }
#pragma unroll
            for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
            const int64_t t = perm[w.begin + warp];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int j = h * 32 + lane;
                if (j < top_k) {
                    prim_out[t * top_k + j] = my_p[h];
                    weight_out[t * top_k + j] = e[h] / sum;
                }
            }
        }
        __syncthreads();  // logits and queries are rewritten by the next item
    }
    if (tid == 0 && *abort) {
        // Let every copy still in flight land before the CTA exits.
        for (int64_t s = gs; s < total_stages && s < gs + kStages; ++s)
            ptx::mbar_wait_drain(&full[s % kStages], (uint32_t)((s / kStages) & 1), kTimeoutNs);
        atomicOr(status, STATUS_WAIT_TIMEOUT);
    }
}

cudaError_t launch_score(const LaunchCtx& c, const ScoreArgs& a) {
    const k3::Geometry g = k3::geometry(a.dtype, a.P, a.dk);
    // Two CTAs per SM when their shared memory allows it.
    const int per_sm = (2 * (g.smem + 1024) <= 228 * 1024) ? 2 : 1;
    const int grid = c.num_sms * per_sm;
    if (a.dtype == LOOKME_BF16) {
        k3_score<__nv_bfloat16><<<grid, k3::kThreads, g.smem, c.stream>>>(
            (const __nv_bfloat16*)a.q, (const __nv_bfloat16*)a.keys, a.P, a.dk, a.top_k, a.scale, a.work, a.n_work,
            a.perm, a.use_slots, a.prim_out, a.weight_out, a.status, g);
    } else {
        k3_score<float><<<grid, k3::kThreads, g.smem, c.stream>>>(
            (const float*)a.q, (const float*)a.keys, a.P, a.dk, a.top_k, a.scale, a.work, a.n_work, a.perm,
            a.use_slots, a.prim_out, a.weight_out, a.status, g);
    }
    return cudaGetLastError();
}

cudaError_t configure_score_kernels() {
    cudaError_t e = cudaFuncSetAttribute(k3_score<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         227 * 1024);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(k3_score<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
}

}  // namespace lookme
