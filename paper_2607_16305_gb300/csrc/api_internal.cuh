// Internals of the host runtime shared by its translation units: the table
// object, argument and error helpers, launch bookkeeping and per-call scratch.
#pragma once
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <climits>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "common.cuh"

using namespace lookme;

namespace lookme_host {

inline thread_local std::string g_last_error;

inline lookme_status fail(lookme_status st, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return st;
}

inline const char* kKernelNames[KID_COUNT] = {"prep",         "route_tc", "route_simt",    "bucket",
                                       "score",        "select",   "inject",        "stage",
                                       "centroid_mean", "inv_cnorm", "route_decode", "select_inject",
                                       "tile_keys",    "bucket_count", "bucket_scan", "bucket_scatter",
                                       "step",         "stage_assign", "gemm",          "decode",
                                              "ranked_select", "ska_gate", "inject_gated",  "text_inject",
                                              "combine",       "router"};

// cuTensorMapEncodeTiled through the runtime's driver entry point, so the
// library does not link libcuda directly.
inline PFN_cuTensorMapEncodeTiled_v12000 get_encode_tiled() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        cudaDriverEntryPointQueryResult q;
        void* p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// 2-D bf16 tensor map over a row-major [rows][cols] matrix, 128-byte swizzle,
// box of 64 columns x box_rows rows; out-of-bounds elements read as zero.
inline bool encode_bf16_2d(CUtensorMap* m, const void* base, int64_t rows, int64_t cols, int box_rows) {
    auto fn = get_encode_tiled();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)(cols * 2)};
    cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Restores the caller's current device on scope exit.
struct DeviceGuard {
    int prev = -1;
    bool ok = false;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) return;
        ok = (prev == dev) || cudaSetDevice(dev) == cudaSuccess;
    }
    ~DeviceGuard() {
        int cur;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

struct TraceEntry {
    int32_t kernel;
    cudaEvent_t start, stop;
};

}  // namespace lookme_host

using lookme_host::TraceEntry;

struct lookme_table {
    lookme_table_desc d{};
    size_t esz = 2;
    int num_sms = 0;
    int small_sms = 0;      // SMs the routing and bucketing grids are sized for (0: num_sms)
    int level2_ctas = 0;    // CTAs of the tcgen05 level 2 (0: num_sms)
    bool tc_route = false;  // level 1 on tcgen05
    bool tc_score = false;  // level 2 on tcgen05
    bool use_step = false;  // whole calls as one fused launch where the shape allows
    int64_t kblock = 0;     // bytes of one scene's stored key block (tiled when tc_score)

    // storage
    void* keys = nullptr;       // device, or device-mapped pinned host
    void* values = nullptr;     // device, or device-mapped pinned host
    void* keys_host = nullptr;  // pinned host allocations (HOST_STAGED)
    void* values_host = nullptr;
    void* slots = nullptr;      // HBM slot cache of staged key blocks
    int64_t n_slots = 0;
    StageArgs stage{};          // the slot cache's map (device), kept across calls
    void* stage_mem = nullptr;
    cudaStream_t stage_stream = nullptr;  // the copies run here, ordered by events
    cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
    void* cent = nullptr;
    float* inv_cnorm = nullptr;
    float* bias = nullptr;
    bool has_bias = false;
    CUtensorMap tmap_c[3];
    std::vector<uint8_t> loaded;
    int64_t n_loaded = 0;

    // scratch
    int64_t cap = 0;
    void* scratch = nullptr;
    unsigned long long* best = nullptr;
    float* qnorm = nullptr;
    int32_t* item_tok = nullptr;
    WorkItem* work = nullptr;
    int32_t* routed = nullptr;
    int32_t* counters = nullptr;  // n_work, n_routed, max bucket
    int32_t* sel = nullptr;
    uint8_t* mask = nullptr;
    int32_t* selpos = nullptr;   // per token: its kept-list slot, or -1
    int32_t* rec_t = nullptr;    // injection records by kept slot: token id,
    int32_t* rec_row = nullptr;  // value rows and weights (kRecMaxTopK per slot)
    float* rec_w = nullptr;
    int32_t* scene_cnt = nullptr;  // large calls' bucketing: per-scene counts (zero between calls)
    int32_t* scene_pos = nullptr;  // and running item_tok positions
    StepState* step = nullptr;     // the fused step's call-to-call state (zero at allocation)
    int32_t* step_ovf = nullptr;   // the fused step's kept tokens past a CTA's on-chip queue
    uint32_t* status = nullptr;   // persistent device status word
    int64_t last_tokens = -1;
    int64_t last_staged_bytes = 0;

    // Paper-exact level 2: the scene-shared ranker MLP (lookme_set_ranker).
    int64_t rk_dm = 0;             // hidden width d_m (0: no ranker)
    void* rk_mem = nullptr;        // one allocation for the weights below
    __nv_bfloat16* rk_w1v = nullptr;  // [d_m][d_k]: W1's query half
    __nv_bfloat16* rk_w1c = nullptr;  // [d_m][d_k]: W1's centroid half
    float* rk_b1 = nullptr;        // [d_m]
    __nv_bfloat16* rk_w2 = nullptr;   // [P][d_m]
    float* rk_b2 = nullptr;        // [P]
    float* rk_c1 = nullptr;        // [S][d_m]: W1c e_img[s] + b1, per scene
    bool rk_c1_stale = true;       // centroids or weights changed since c1 was computed
    void* rk_scratch = nullptr;    // per call: hidden H [cap][d_m] bf16, relevance r [cap][ld_r] fp32
    int64_t rk_cap = 0;

    lookme_status sticky = LOOKME_OK;
    uint64_t launches = 0;

    bool trace = false;
    std::vector<TraceEntry> trace_log;
    std::vector<cudaEvent_t> event_pool;
};

namespace lookme_host {

inline lookme_status cuda_fail(lookme_table* t, cudaError_t e, const char* what) {
    if (t) t->sticky = LOOKME_ERR_CUDA;
    return fail(LOOKME_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

inline cudaEvent_t pool_event(lookme_table* t) {
    if (!t->event_pool.empty()) {
        cudaEvent_t e = t->event_pool.back();
        t->event_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
}

inline bool capturing(cudaStream_t s) {
    cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(s, &st) != cudaSuccess) return false;
    return st != cudaStreamCaptureStatusNone;
}

// Runs one kernel launch: counts it, brackets it with trace events if tracing.
template <typename F>
inline lookme_status launch(lookme_table* t, cudaStream_t s, int32_t kid, F&& fn) {
    const bool tr = t->trace && !capturing(s);
    TraceEntry te{kid, nullptr, nullptr};
    if (tr) {
        te.start = pool_event(t);
        te.stop = pool_event(t);
        cudaEventRecord(te.start, s);
    }
    cudaError_t e = fn();
    if (e != cudaSuccess) return cuda_fail(t, e, kKernelNames[kid]);
    ++t->launches;
    if (tr) {
        cudaEventRecord(te.stop, s);
        t->trace_log.push_back(te);
    }
    return LOOKME_OK;
}

inline lookme_status check_table(const lookme_table* t) {
    if (!t) return fail(LOOKME_ERR_INVALID_ARG, "table is NULL");
    if (t->sticky != LOOKME_OK) return fail(t->sticky, "table is unusable after an earlier CUDA error");
    return LOOKME_OK;
}

inline void free_scratch(lookme_table* t) {
    if (t->scratch) cudaFree(t->scratch);
    t->scratch = nullptr;
    t->cap = 0;
}

inline lookme_status ensure_scratch(lookme_table* t, int64_t n, cudaStream_t s) {
    if (n <= t->cap && t->scratch) return LOOKME_OK;
    if (s && capturing(s))
        return fail(LOOKME_ERR_STATE, "scratch must grow to %lld tokens while the stream is captured; call "
                    "lookme_reserve first", (long long)n);
    const int64_t cap = n > 0 ? n : 1;
    const int64_t S = t->d.n_scenes;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        const size_t o = off;
        off = align_up(off + bytes, 256);
        return o;
    };
    const size_t o_best = take(cap * sizeof(unsigned long long));
    const size_t o_qnorm = take(cap * sizeof(float));
    const size_t o_work = take((cap + S) * sizeof(WorkItem));
    const size_t o_itok = take((cap + S) * kTokensPerItem * sizeof(int32_t));
    const size_t o_routed = take(S * sizeof(int32_t));
    const size_t o_counters = take(4 * sizeof(int32_t));
    const size_t o_sel = take(cap * sizeof(int32_t));
    const size_t o_mask = take(cap);
    const size_t o_selpos = take(cap * sizeof(int32_t));
    const size_t o_rec_t = take(cap * sizeof(int32_t));
    const size_t o_rec_row = take(cap * kRecMaxTopK * sizeof(int32_t));
    const size_t o_rec_w = take(cap * kRecMaxTopK * sizeof(float));
    const size_t o_scnt = take(S * sizeof(int32_t));
    const size_t o_spos = take(S * sizeof(int32_t));
    const size_t o_step = take(sizeof(StepState));
    const size_t o_sovf = take((cap + S) * kTokensPerItem * sizeof(int32_t));
    void* buf = nullptr;
    if (cudaDeviceSynchronize() != cudaSuccess || cudaMalloc(&buf, off) != cudaSuccess) {
        cudaGetLastError();
        return fail(LOOKME_ERR_OOM, "scratch allocation of %zu bytes failed", off);
    }
    free_scratch(t);
    char* b = static_cast<char*>(buf);
    t->scratch = buf;
    t->cap = cap;
    t->best = reinterpret_cast<unsigned long long*>(b + o_best);
    t->qnorm = reinterpret_cast<float*>(b + o_qnorm);
    t->work = reinterpret_cast<WorkItem*>(b + o_work);
    t->item_tok = reinterpret_cast<int32_t*>(b + o_itok);
    t->routed = reinterpret_cast<int32_t*>(b + o_routed);
    t->counters = reinterpret_cast<int32_t*>(b + o_counters);
    t->sel = reinterpret_cast<int32_t*>(b + o_sel);
    t->mask = reinterpret_cast<uint8_t*>(b + o_mask);
    t->selpos = reinterpret_cast<int32_t*>(b + o_selpos);
    t->rec_t = reinterpret_cast<int32_t*>(b + o_rec_t);
    t->rec_row = reinterpret_cast<int32_t*>(b + o_rec_row);
    t->rec_w = reinterpret_cast<float*>(b + o_rec_w);
    t->scene_cnt = reinterpret_cast<int32_t*>(b + o_scnt);
    t->scene_pos = reinterpret_cast<int32_t*>(b + o_spos);
    t->step = reinterpret_cast<StepState*>(b + o_step);
    t->step_ovf = reinterpret_cast<int32_t*>(b + o_sovf);
    t->last_tokens = -1;
    if (cudaMemset(buf, 0, off) != cudaSuccess) return cuda_fail(t, cudaGetLastError(), "scratch memset");
    return LOOKME_OK;
}

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

inline void destroy_table(lookme_table* t) {
    if (!t) return;
    for (auto& te : t->trace_log) {
        cudaEventDestroy(te.start);
        cudaEventDestroy(te.stop);
    }
    for (auto e : t->event_pool) cudaEventDestroy(e);
    free_scratch(t);
    if (t->d.residency == LOOKME_RES_DEVICE) {
        if (t->keys) cudaFree(t->keys);
        if (t->values) cudaFree(t->values);
    } else {
        if (t->keys_host) cudaFreeHost(t->keys_host);
        if (t->values_host) cudaFreeHost(t->values_host);
        if (t->slots) cudaFree(t->slots);
        if (t->stage_mem) cudaFree(t->stage_mem);
        if (t->ev_fork) cudaEventDestroy(t->ev_fork);
        if (t->ev_join) cudaEventDestroy(t->ev_join);
        if (t->stage_stream) cudaStreamDestroy(t->stage_stream);
    }
    if (t->rk_mem) cudaFree(t->rk_mem);
    if (t->rk_scratch) cudaFree(t->rk_scratch);
    if (t->cent) cudaFree(t->cent);
    if (t->inv_cnorm) cudaFree(t->inv_cnorm);
    if (t->bias) cudaFree(t->bias);
    if (t->status) cudaFree(t->status);
    delete t;
}

}  // namespace lookme_host
