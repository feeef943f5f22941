// Shared declarations of the LookME CUDA library: element helpers, argmax key
// packing, kernel ids and the launch wrappers each kernel file defines.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "lookme.h"

namespace lookme {

// ---------------------------------------------------------------- kernel ids
enum KernelId : int32_t {
    KID_PREP = 0,        // K0: ||q||, argmax reset
    KID_ROUTE_TC = 1,    // K1: level-1 scores on tcgen05 + fused argmax
    KID_ROUTE_SIMT = 2,  // K1: level-1 scores on CUDA cores (fp32 tables, odd shapes)
    KID_BUCKET = 3,      // K2: counting sort of tokens by scene + work list
    KID_SCORE = 4,       // K3: level-2 key scoring + top-k + softmax
    KID_SELECT = 5,      // K5: top-r token selection per segment
    KID_INJECT = 6,      // K4: gather + weighted sum + residual add
    KID_STAGE = 7,       // K6: host -> HBM staging of routed key blocks
    KID_CENTROID = 8,    // load-time: centroid = mean of keys
    KID_CNORM = 9,       // load-time: 1 / ||centroid||
    KID_ROUTE_DECODE = 10,  // argmax key -> scene id (allocation-free routing)
    KID_SELECT_INJECT = 11, // K5 + K4 fused for short segments
    KID_TILE_KEYS = 12,  // load-time: keys into the tcgen05 level-2 tile layout
    KID_BUCKET_COUNT = 13,    // K2 for large calls: per-scene counts (+ gate CTAs)
    KID_BUCKET_SCAN = 14,     // K2 for large calls: work list from the counts
    KID_BUCKET_SCATTER = 15,  // K2 for large calls: token ids into their items
    KID_STEP = 16,            // K1 + K2 + K3 (+ gate and K4): the fused step on tcgen05
    KID_STAGE_ASSIGN = 17,    // K6a: slot cache look-up and the copy list
    KID_GEMM = 18,            // dense bf16 GEMM (ranker MLP, projection, fusion, propagation, router)
    KID_DECODE = 19,          // argmax key -> scene, key reset (paper-exact level 2)
    KID_RANKED_SELECT = 20,   // top-T by relevance, cos + tanh softmax
    KID_SKA_GATE = 21,        // hard SKA gate
    KID_INJECT_GATED = 22,    // injection on a given gate
    KID_TEXT_INJECT = 23,     // text pathway gather + injection
    KID_COMBINE = 24,         // retrieved embeddings of listed tokens
    KID_ROUTER = 25,          // multi-scale softmax router
    KID_COUNT
};

// Device status bits (table status word).
constexpr uint32_t STATUS_WAIT_TIMEOUT = 1u;
constexpr uint32_t STATUS_IN_ROUTE = 2u;  // set with STATUS_WAIT_TIMEOUT by the level-1 kernel
constexpr uint32_t STATUS_IN_SCORE = 4u;  // set with STATUS_WAIT_TIMEOUT by a level-2 kernel
constexpr uint32_t STATUS_IN_STEP = 8u;   // set with STATUS_WAIT_TIMEOUT by the fused step kernel
constexpr uint32_t STATUS_STAGE_OVERFLOW = 16u;  // more routed scenes than HBM slots (keys not staged)
constexpr uint32_t STATUS_BAD_INDEX = 64u;  // a kernel met an index outside its range and skipped the access

// ------------------------------------------------------------ element access
__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

// 16 bytes -> floats: 8 bf16 or 4 fp32.
template <typename T> struct Vec16;
template <> struct Vec16<__nv_bfloat16> {
    static constexpr int N = 8;
    __device__ __forceinline__ static void unpack(const uint4& v, float* f) {
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            f[2 * i] = __uint_as_float(w[i] << 16);
            f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
        }
    }
    __device__ __forceinline__ static uint4 pack(const float* f) {
        uint32_t w[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            __nv_bfloat162 h = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
            w[i] = *reinterpret_cast<uint32_t*>(&h);
        }
        return make_uint4(w[0], w[1], w[2], w[3]);
    }
};
template <> struct Vec16<float> {
    static constexpr int N = 4;
    __device__ __forceinline__ static void unpack(const uint4& v, float* f) {
        f[0] = __uint_as_float(v.x);
        f[1] = __uint_as_float(v.y);
        f[2] = __uint_as_float(v.z);
        f[3] = __uint_as_float(v.w);
    }
    __device__ __forceinline__ static uint4 pack(const float* f) {
        return make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]), __float_as_uint(f[2]),
                          __float_as_uint(f[3]));
    }
};

// -------------------------------------------------------- argmax key packing
// A 64-bit key whose unsigned order is (score ascending, scene descending), so
// that atomicMax keeps the highest score and, among equal scores, the lowest
// scene index.  Key 0 means "no candidate".
__device__ __forceinline__ uint32_t orderable(float f) {
    uint32_t u = __float_as_uint(f == 0.0f ? 0.0f : f);  // -0 and +0 compare equal
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ unsigned long long pack_argmax(float score, uint32_t scene) {
    return ((unsigned long long)orderable(score) << 32) | (unsigned long long)(0xFFFFFFFFu - scene);
}
__device__ __forceinline__ int32_t unpack_scene(unsigned long long key, int64_t n_scenes) {
    uint32_t s = 0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull);
    return (key == 0ull || s >= (uint64_t)n_scenes) ? 0 : (int32_t)s;
}

// Work item i of level 2: tokens item_tok[begin, begin + count) all routed to
// `scene`, begin = kTokensPerItem * i; `slot` is the scene's index in the
// routed-scene list (and its HBM slot when keys are staged).
struct WorkItem {
    int32_t scene, begin, count, slot;
};

// ---------------------------------------------- programmatic dependent launch
// Every per-call kernel is launched with programmatic stream serialisation:
// it may start while its predecessor on the stream is still running, lets its
// own successor start early (pdl_trigger), and waits for the predecessor's
// completion and memory (pdl_wait) before it touches any data a predecessor
// produces or consumes.  Both are no-ops for a normal launch.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                       Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// ------------------------------------------------------------ launch params
struct LaunchCtx {
    cudaStream_t stream;
    int num_sms;
};

// K0
cudaError_t launch_prep(const LaunchCtx& c, int dtype, const void* q, int64_t N, int dk, float* qnorm,
                        float* qnorm_out, unsigned long long* best);
// K1 (tcgen05, bf16, d_k <= 512).  tmap_q is the CUtensorMap of the queries
// (box 64 x 128); tmap_c[i] the centroids' map with box 64 x (64 << i).  Also
// computes ||q|| into qnorm (and qnorm_out if given), so no prep kernel runs;
// every key of best[0, N) must be 0 on entry.
constexpr int kRouteTcMaxDk = 512;
cudaError_t launch_route_tc(const LaunchCtx& c, const void* tmap_q, const void* const tmap_c[3], int64_t N,
                            int64_t S, int dk, const float* inv_cnorm, const float* bias, float* qnorm,
                            float* qnorm_out, unsigned long long* best, uint32_t* status);
// K1 (CUDA cores)
cudaError_t launch_route_simt(const LaunchCtx& c, int dtype, const void* q, const void* cent, int64_t N,
                              int64_t S, int dk, const float* inv_cnorm, const float* bias, const float* qnorm,
                              unsigned long long* best);
// K2 (also resets best[0, N) to 0 for the next call)
constexpr int kTokensPerItem = 8;
// gate (optional, GateSpec declared below) adds CTAs that compute the injection gate.
struct GateSpec;
cudaError_t launch_bucket(const LaunchCtx& c, unsigned long long* best, int64_t N, int64_t S,
                          int32_t* scene_out, int32_t* item_tok, WorkItem* work, int32_t* routed, int32_t* counters,
                          const GateSpec* gate = nullptr);
// The same result for calls of more than kBucketOneCtaTokens tokens, in three
// launches over all SMs: per-scene counts (global, warp-aggregated atomics;
// the gate CTAs ride along), the work list from the counts (one CTA; it also
// zeroes the counts for the next call), and the token ids into their items.
// cnt [S] must be zero on entry; pos [S] is scratch.
constexpr int64_t kBucketOneCtaTokens = 8192;
cudaError_t launch_bucket_count(const LaunchCtx& c, unsigned long long* best, int64_t N, int64_t S,
                                int32_t* scene_out, int32_t* cnt, const GateSpec* gate);
cudaError_t launch_bucket_scan(const LaunchCtx& c, int64_t S, int32_t* cnt, int32_t* pos, WorkItem* work,
                               int32_t* routed, int32_t* counters);
cudaError_t launch_bucket_scatter(const LaunchCtx& c, unsigned long long* best, int64_t N,
                                  const int32_t* scene_out, int32_t* pos, int32_t* item_tok);
// K3
struct ScoreArgs {
    int dtype;
    const void* q;
    const void* keys;     // [S or slots][P][dk]
    int64_t P;
    int dk;
    int top_k;
    float scale;          // 1 / sqrt(d_k)
    const WorkItem* work;
    int64_t work_cap;     // entries of the work array
    int32_t* counters;    // [0] work items (from bucketing), [3] work-taking counter (reset by bucketing)
    const int32_t* item_tok;  // the items' token ids, kTokensPerItem slots per work entry
    int use_slots;        // index key blocks by WorkItem::slot instead of ::scene
    int32_t* prim_out;
    float* weight_out;
    uint32_t* status;
    // Optional (tcgen05 level 2): the injection gate decided beside the
    // bucketing, as each kept token's slot in the kept-id list (-1: not
    // kept); the value rows (and the first layer's hidden row) of kept tokens
    // are prefetched into L2.
    const int32_t* selpos;
    const void* values;   // [S][P][d_v], device memory
    int64_t vrow_bytes;   // d_v * element size
    const void* hidden0;  // the first layer's hidden states (prefetch only), or null
    // Optional: the injection records of kept tokens at their slots: token id,
    // and top_k value rows (scene * N_p + p) and weights (stride top_k).
    int32_t* rec_t;
    int32_t* rec_row;
    float* rec_w;
};
cudaError_t launch_score(const LaunchCtx& c, const ScoreArgs& a);
// Whether the level-2 kernel's shared-memory plan fits this table shape.
bool score_shape_supported(int dtype, int64_t P, int dk);
// The injection gate computed by extra CTAs of the bucketing kernel: token t
// of segment s is kept iff its rank (larger priority first, lower index on
// ties) is below r_s = floor(len_s * keep_ratio); kept tokens go to
// sel[sel_base[s] + rank].
constexpr int kMaxGateSegments = 64;
struct GateSpec {
    int enabled;
    int n_seg;
    int64_t N;
    double keep_ratio;
    const float* priority;
    uint8_t* mask;
    int32_t* sel;
    int32_t* selpos;  // optional: per token its slot sel_base + rank when kept, else -1
    int64_t off[kMaxGateSegments + 1];
    int64_t sel_base[kMaxGateSegments];
};

// Level 2 on tcgen05 (bf16 tables).  keys_tiled holds every scene's (or
// staging slot's) keys in the tiled layout of k_tile_keys, one block of
// score_tc_block_bytes(P, d_k) bytes per scene; ScoreArgs::keys is unused.
cudaError_t launch_score_tc(const LaunchCtx& c, const void* keys_tiled, const ScoreArgs& a);
bool score_tc_shape_supported(int64_t P, int dk);
int64_t score_tc_block_bytes(int64_t P, int dk);
// Load time: rewrites n scenes of row-major keys [n][P][d_k] (bf16, device
// readable) into the tiled layout: per scene, sub-blocks (tile t of 128 rows,
// k-block b of 64 columns) ordered by N-tile (tiles 2m, 2m + 1), then b, then
// t, each 128 rows x 128 bytes with 16-byte chunk c of row r stored at chunk
// position c ^ (r & 7); rows past P and columns past d_k are zero.
cudaError_t launch_tile_keys(const LaunchCtx& c, const void* src, void* dst, int64_t n, int64_t P, int dk);
// K5
cudaError_t launch_select(const LaunchCtx& c, const float* priority, int64_t N, const int64_t* seg_off_host,
                          int n_seg, double keep_ratio, uint8_t* mask, int32_t* sel);
// K4
struct InjectArgs {
    int dtype;
    const void* values;   // [S][P][dv] (device or host-mapped)
    int64_t P;
    int dv;
    int top_k;
    const int32_t* scene;
    const int32_t* prim;
    const float* weight;
    const int32_t* sel;
    int64_t n_sel;
    int64_t N;
    int64_t S;
    int n_layers;
    void* hidden[LOOKME_MAX_LAYERS];
    uint32_t* status;     // STATUS_BAD_INDEX when a record names no token (records form)
};
cudaError_t launch_inject(const LaunchCtx& c, const InjectArgs& a);
// K4 from the records the tcgen05 level-2 kernel wrote (ScoreArgs::rec_*):
// one CTA per kept slot, every load it needs issued in one round trip.
constexpr int kRecMaxTopK = 16;
cudaError_t launch_inject_records(const LaunchCtx& c, const InjectArgs& a, const int32_t* rec_t,
                                  const int32_t* rec_row, const float* rec_w);
// K5 + K4 in one kernel (one CTA per token) for segments of at most
// kFusedMaxSegment tokens when the kept-id list is not requested.
constexpr int64_t kFusedMaxSegment = 8192;
cudaError_t launch_select_inject(const LaunchCtx& c, const InjectArgs& a, const float* priority,
                                 const int64_t* seg_off_host, int n_seg, double keep_ratio, uint8_t* mask);
// K6: the HBM slot cache of a pinned-host table, kept across calls.  Per
// scene its slot or -1 (slot_of), per slot its scene or -1 (slot_scene) and
// the number of the last call that used it (slot_stamp), and this header.
struct StageCache {
    int32_t epoch;     // calls so far (stamps the slots each call uses)
    int32_t hand;      // where the next search for free slots starts
    int32_t n_copy;    // key blocks the last call copied from the host
    int32_t n_hit;     // routed scenes the last call found in HBM
};
struct StageArgs {
    int32_t* slot_of;     // [S]
    int32_t* slot_scene;  // [n_slots]
    int32_t* slot_stamp;  // [n_slots]
    int32_t* route_slot;  // [S] per routed-list index: its slot (scratch)
    int32_t* copy_slot;   // [n_slots] copies of this call: slot and scene
    int32_t* copy_scene;  // [n_slots]
    StageCache* hdr;
    int64_t n_slots;
};
// K6a (one CTA): find each routed scene's slot, give the misses free or
// least-recently-reached slots, list the copies, point the work items at
// their slots.  K6b: copy the listed key blocks over the host mapping.
cudaError_t launch_stage_assign(const LaunchCtx& c, const StageArgs& sa, const int32_t* routed,
                                const int32_t* counters, WorkItem* work, uint32_t* status);
cudaError_t launch_stage(const LaunchCtx& c, const void* keys_host_mapped, void* slots, int64_t block_bytes,
                         const StageArgs& sa);

// ----------------------------------------------- dense bf16 GEMM on tcgen05
// D[M][Nn] = A[M][K] B[Nn][K]^T (bf16 operands, fp32 accumulation in TMEM),
// with one of these epilogues:
enum GemmEpi : int {
    EPI_F32 = 0,          // out f32 = D + colbias
    EPI_BF16 = 1,         // out bf16 = act(D + colbias + rowbias[rowsel[m]])
    EPI_SWIGLU = 2,       // out bf16 [M][Nn/2] = silu(gate) * up, B rows interleaved per 32 features
    EPI_RESID = 3,        // out bf16 = D + colbias + resid (resid may be out itself)
    EPI_SCATTER_ADD = 4,  // out[rowidx[m]] (bf16) += D + colbias
};
struct GemmArgs {
    int64_t M, Nn, K;
    int mode, act;            // act: 0 none, 1 silu (EPI_BF16)
    const float* colbias;     // [Nn] or null
    const float* rowbias;     // [..][ld_rowbias], row rowsel[m] (EPI_BF16) or null
    const int32_t* rowsel;
    int64_t ld_rowbias;
    void* out;
    int64_t ld_out;           // elements
    const void* resid;        // bf16 [M][ld_resid] (EPI_RESID)
    int64_t ld_resid;
    const int32_t* rowidx;    // destination rows (EPI_SCATTER_ADD)
    uint32_t* status;         // bounded waits report here (bit STATUS_IN_GEMM)
};
constexpr uint32_t STATUS_IN_GEMM = 32u;
// Tile width chosen for (M, Nn) on num_sms SMs: 64, 128 or 256 columns.
int gemm_tile_n(int64_t M, int64_t Nn, int num_sms);
// tmap_a: [M][K] bf16, box 64 x 128 rows; tmap_b: [Nn][K] bf16, box 64 x BN rows
// (BN = gemm_tile_n), both with the 128-byte swizzle.
cudaError_t launch_gemm_tc(const LaunchCtx& c, const void* tmap_a, const void* tmap_b, int bn, const GemmArgs& g);
cudaError_t configure_gemm_kernels();

// ------------------------------------------------ SIMT kernels around GEMMs
// scene_out[t] = the routed scene of argmax key best[t]; best[t] reset to 0.
cudaError_t launch_decode_reset(const LaunchCtx& c, unsigned long long* best, int64_t N, int64_t S,
                                int32_t* scene_out);
// Keys of a bf16 table as stored: tiled (the level-2 kernel's layout) or row-major.
struct KeyView {
    const uint8_t* keys;
    int64_t block_bytes;  // bytes per scene
    int P, dk;
    int tiled, ntile, nkb;
};
// Paper-exact level 2 from the relevance r [N][P] (fp32): top-T per token,
// weights softmax(cos(q, K[scene, p]) + tanh r[p]); one warp per token.
cudaError_t launch_ranked_select(const LaunchCtx& c, const float* r, int64_t ld_r, int64_t N, int T, const __nv_bfloat16* q,
                                 const KeyView& kv, const int32_t* scene, int32_t* prim_out, float* weight_out);
// g_t = [Delta_t . w_g > 0]; logit_out optional.
cudaError_t launch_ska_gate(const LaunchCtx& c, int dtype, const void* delta, const void* wg, int64_t N, int64_t dh,
                            uint8_t* gate, float* logit_out);
// h_l[t] += sum_j w_tj V[scene_t, prim_tj] for every t with gate[t].
cudaError_t launch_inject_gated(const LaunchCtx& c, const InjectArgs& a, const uint8_t* gate);
// h_l[t] += E[ids[t]] for gated t with 0 <= ids[t] < V.
cudaError_t launch_text_inject(const LaunchCtx& c, int dtype, const void* E, int64_t V, int64_t d,
                               const int32_t* ids, const uint8_t* gate, int64_t N, void* const* hidden, int n_layers);
// R_out[i] (bf16) = sum_j w_tj V[scene_t, prim_tj], t = rows[i].
cudaError_t launch_combine(const LaunchCtx& c, const InjectArgs& a, const int32_t* rows, int64_t n,
                           __nv_bfloat16* R_out);
// out_t = sum_m softmax_m(q_t . R^m_t / sqrt(de)) R^m_t; q fp32 [N][de], R^m bf16 [N][de].
constexpr int kRouterMaxScales = 16;
cudaError_t launch_scale_router(const LaunchCtx& c, const float* q, const __nv_bfloat16* const* Rs, int M, int64_t N,
                                int64_t de, __nv_bfloat16* out, float* att_out);

// ------------------------------------------------------------- fused step
// Routing, bucketing, level 2, the injection gate and the injection in one
// launch of one CTA per SM (bf16 tables in HBM, N <= kStepMaxTokens,
// top_k <= kRecMaxTopK).  The call-to-call state it keeps in device memory
// (zero when first allocated): the epoch whose parity picks the argmax-key
// buffer and the grid-barrier counter of a call, and the exit ticket.
constexpr int64_t kStepMaxTokens = 8192;
struct StepState {
    uint32_t epoch;
    uint32_t exit_cnt;
    uint32_t bar[2];
    uint32_t pad[60];
    unsigned long long best[2][kStepMaxTokens];
};
struct StepArgs {
    int64_t N, S, P;
    int dk, dv, top_k;
    float scale;
    const void* q;           // [N][d_k] bf16
    const void* keys_tiled;  // the level-2 tile layout, one block per scene
    int64_t block_bytes;
    const void* values;      // [S][P][d_v] bf16
    const float* inv_cnorm;
    const float* bias;       // or null
    int32_t* scene_out;
    int32_t* prim_out;
    float* weight_out;
    float* qnorm;            // [N] scratch: the query norms (default gate priority)
    float* qnorm_out;        // or null
    // gate and injection; gate = 0 is a lookup without injection
    int gate;
    int n_seg;
    const float* priority;   // or null: the query norms
    uint8_t* mask_out;       // or null
    int64_t seg_off[kMaxGateSegments + 1];
    int64_t seg_r[kMaxGateSegments];
    int n_layers;
    void* hidden[LOOKME_MAX_LAYERS];
    // scratch
    StepState* state;
    WorkItem* work;          // >= N + S entries
    int32_t* item_tok;       // kTokensPerItem per work entry
    int32_t* counters;       // [0] work items, [1] routed scenes, [2] largest bucket
    uint32_t* status;
    // kept tokens past a CTA's on-chip queue: their value rows and weights by
    // token id ([N][kRecMaxTopK]) and their ids (kTokensPerItem per work entry)
    int32_t* rec_row;
    float* rec_w;
    int32_t* ovf_tok;
};
// Whether the fused step handles this table shape (shared memory, TMEM).
bool step_shape_supported(int64_t N, int64_t S, int64_t P, int dk, int dv, int num_sms);
cudaError_t launch_step(const LaunchCtx& c, const void* tmap_q, const void* const tmap_c[3], const StepArgs& a);

// Raise the dynamic shared-memory limits of the kernels that need more than
// 48 KB (per device; call with the device current).
cudaError_t configure_route_kernels();
cudaError_t configure_bucket_kernel();
cudaError_t configure_score_kernels();
cudaError_t configure_score_tc_kernel();
cudaError_t configure_step_kernel();
// load-time
cudaError_t launch_centroid_mean(const LaunchCtx& c, int dtype, const void* keys, int64_t n, int64_t P, int dk,
                                 void* cent);
cudaError_t launch_inv_cnorm(const LaunchCtx& c, int dtype, const void* cent, int64_t n, int dk, float* inv_cnorm);

}  // namespace lookme
