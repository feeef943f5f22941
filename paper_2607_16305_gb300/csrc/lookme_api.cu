// Host runtime of the LookME library: the C ABI declared in lookme.h.
//
// A table owns its storage (HBM, or pinned host memory plus an HBM slot
// cache), its centroids with their inverse norms, an optional routing bias and
// the per-call scratch.  Every entry point validates its arguments on the host
// before touching the device, switches to the table's device for the duration
// of the call, enqueues kernels on the caller's stream and never synchronises
// it (except the calls documented as synchronous).
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

#include "api_internal.cuh"

using namespace lookme_host;


extern "C" {

const char* lookme_status_string(lookme_status s) {
    switch (s) {
        case LOOKME_OK: return "ok";
        case LOOKME_ERR_INVALID_ARG: return "invalid argument";
        case LOOKME_ERR_CUDA: return "CUDA error";
        case LOOKME_ERR_OOM: return "out of memory";
        case LOOKME_ERR_TIMEOUT: return "device wait timed out";
        case LOOKME_ERR_STATE: return "call out of order";
        case LOOKME_ERR_UNSUPPORTED: return "unsupported";
    }
    return "unknown status";
}

const char* lookme_last_error(void) { return g_last_error.c_str(); }

const char* lookme_kernel_name(int32_t k) { return (k >= 0 && k < KID_COUNT) ? kKernelNames[k] : "?"; }

lookme_status lookme_table_create(const lookme_table_desc* desc, lookme_table** out) {
    if (!out) return fail(LOOKME_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    if (!desc) return fail(LOOKME_ERR_INVALID_ARG, "desc is NULL");
    const lookme_table_desc& d = *desc;
    if (d.dtype != LOOKME_BF16 && d.dtype != LOOKME_FP32) return fail(LOOKME_ERR_INVALID_ARG, "bad dtype %d", d.dtype);
    if (d.residency != LOOKME_RES_DEVICE && d.residency != LOOKME_RES_HOST_STAGED)
        return fail(LOOKME_ERR_INVALID_ARG, "bad residency %d", d.residency);
    if (d.reserved0 != 0) return fail(LOOKME_ERR_INVALID_ARG, "reserved0 must be 0");
    if (d.n_scenes < 1 || d.n_scenes > LOOKME_MAX_SCENES)
        return fail(LOOKME_ERR_INVALID_ARG, "n_scenes %lld outside [1, %d]", (long long)d.n_scenes, LOOKME_MAX_SCENES);
    if (d.n_prims < 1 || d.n_prims > LOOKME_MAX_PRIMS)
        return fail(LOOKME_ERR_INVALID_ARG, "n_prims %lld outside [1, %d]", (long long)d.n_prims, LOOKME_MAX_PRIMS);
    if (d.d_key < 1 || d.d_key > LOOKME_MAX_DKEY)
        return fail(LOOKME_ERR_INVALID_ARG, "d_key %lld outside [1, %d]", (long long)d.d_key, LOOKME_MAX_DKEY);
    if (d.d_value < 1) return fail(LOOKME_ERR_INVALID_ARG, "d_value must be >= 1");
    const int vec = d.dtype == LOOKME_BF16 ? 8 : 4;
    if (d.d_key % vec || d.d_value % vec)
        return fail(LOOKME_ERR_INVALID_ARG, "d_key and d_value must be multiples of %d for this dtype", vec);
    if (d.max_tokens < 0 || d.stage_slots < 0) return fail(LOOKME_ERR_INVALID_ARG, "negative size");
    if (!score_shape_supported(d.dtype, d.n_prims, (int)d.d_key))
        return fail(LOOKME_ERR_UNSUPPORTED, "n_prims %lld with d_key %lld does not fit the level-2 kernel's shared memory",
                    (long long)d.n_prims, (long long)d.d_key);
    if ((int64_t)d.n_scenes * d.n_prims > ((int64_t)1 << 31) - 1)
        return fail(LOOKME_ERR_INVALID_ARG, "n_scenes * n_prims must fit in int32");

    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || d.device < 0 || d.device >= ndev) {
        cudaGetLastError();
        return fail(LOOKME_ERR_INVALID_ARG, "device %d not available (%d devices)", d.device, ndev);
    }
    DeviceGuard guard(d.device);
    if (!guard.ok) return fail(LOOKME_ERR_CUDA, "cannot select device %d", d.device);

    lookme_table* t = new lookme_table();
    t->d = d;
    t->esz = d.dtype == LOOKME_BF16 ? 2 : 4;
    cudaDeviceGetAttribute(&t->num_sms, cudaDevAttrMultiProcessorCount, d.device);
    t->tc_route = d.dtype == LOOKME_BF16 && d.d_key <= kRouteTcMaxDk;
    t->tc_score = d.dtype == LOOKME_BF16 && score_tc_shape_supported(d.n_prims, (int)d.d_key);
    // Validation switches: LOOKME_ROUTE=simt / LOOKME_SCORE=simt run bf16 tables
    // on the CUDA-core level-1 / level-2 kernels too, so each pair of kernels
    // can be checked against each other.
    if (const char* env = getenv("LOOKME_ROUTE")) {
        if (strcmp(env, "simt") == 0) t->tc_route = false;
    }
    if (const char* env = getenv("LOOKME_SCORE")) {
        if (strcmp(env, "simt") == 0) t->tc_score = false;
    }
    // LOOKME_STEP=on runs whole calls as one launch of the fused step kernel
    // where the shape allows (it is correct, but measured slower than the
    // separate kernels on this GB300, so it is not the default).
    t->use_step = false;
    if (const char* env = getenv("LOOKME_STEP")) {
        if (strcmp(env, "on") == 0) t->use_step = t->tc_route && t->tc_score;
    }
    t->loaded.assign(d.n_scenes, 0);

    cudaError_t e;
    if ((e = configure_route_kernels()) != cudaSuccess || (e = configure_bucket_kernel()) != cudaSuccess ||
        (e = configure_score_kernels()) != cudaSuccess || (e = configure_score_tc_kernel()) != cudaSuccess ||
        (e = configure_step_kernel()) != cudaSuccess || (e = configure_gemm_kernels()) != cudaSuccess) {
        destroy_table(t);
        return fail(LOOKME_ERR_CUDA, "kernel configuration: %s", cudaGetErrorString(e));
    }

    const size_t S = d.n_scenes, P = d.n_prims;
    // tcgen05 tables store keys as the level-2 kernel's shared-memory tiles.
    t->kblock = t->tc_score ? score_tc_block_bytes(d.n_prims, (int)d.d_key) : (int64_t)(P * d.d_key * t->esz);
    const size_t kbytes = S * (size_t)t->kblock, vbytes = S * P * d.d_value * t->esz;
    bool ok = true;
    if (d.residency == LOOKME_RES_DEVICE) {
        ok = cudaMalloc(&t->keys, kbytes) == cudaSuccess && cudaMalloc(&t->values, vbytes) == cudaSuccess;
    } else {
        ok = cudaHostAlloc(&t->keys_host, kbytes, cudaHostAllocMapped | cudaHostAllocPortable) == cudaSuccess &&
             cudaHostAlloc(&t->values_host, vbytes, cudaHostAllocMapped | cudaHostAllocPortable) == cudaSuccess &&
             cudaHostGetDevicePointer(&t->keys, t->keys_host, 0) == cudaSuccess &&
             cudaHostGetDevicePointer(&t->values, t->values_host, 0) == cudaSuccess;
        t->n_slots = d.stage_slots > 0 ? std::min<int64_t>(d.stage_slots, d.n_scenes) : d.n_scenes;
        ok = ok && cudaMalloc(&t->slots, (size_t)t->n_slots * t->kblock) == cudaSuccess;
        // The slot cache's map: slot_of and route_slot [S], slot_scene,
        // slot_stamp, copy_slot and copy_scene [n_slots], the header.
        const size_t a = align_up(S * sizeof(int32_t), 256), b = align_up(t->n_slots * sizeof(int32_t), 256);
        ok = ok && cudaMalloc(&t->stage_mem, 2 * a + 4 * b + 256) == cudaSuccess &&
             cudaStreamCreateWithFlags(&t->stage_stream, cudaStreamNonBlocking) == cudaSuccess &&
             cudaEventCreateWithFlags(&t->ev_fork, cudaEventDisableTiming) == cudaSuccess &&
             cudaEventCreateWithFlags(&t->ev_join, cudaEventDisableTiming) == cudaSuccess;
        if (ok) {
            char* m = static_cast<char*>(t->stage_mem);
            t->stage.slot_of = reinterpret_cast<int32_t*>(m);
            t->stage.route_slot = reinterpret_cast<int32_t*>(m + a);
            t->stage.slot_scene = reinterpret_cast<int32_t*>(m + 2 * a);
            t->stage.slot_stamp = reinterpret_cast<int32_t*>(m + 2 * a + b);
            t->stage.copy_slot = reinterpret_cast<int32_t*>(m + 2 * a + 2 * b);
            t->stage.copy_scene = reinterpret_cast<int32_t*>(m + 2 * a + 3 * b);
            t->stage.hdr = reinterpret_cast<StageCache*>(m + 2 * a + 4 * b);
            t->stage.n_slots = t->n_slots;
            ok = cudaMemset(t->stage_mem, 0, 2 * a + 4 * b + 256) == cudaSuccess &&
                 cudaMemset(t->stage.slot_of, 0xFF, S * sizeof(int32_t)) == cudaSuccess &&
                 cudaMemset(t->stage.slot_scene, 0xFF, t->n_slots * sizeof(int32_t)) == cudaSuccess;
        }
    }
    ok = ok && cudaMalloc(&t->cent, align_up(S * d.d_key * t->esz, 256)) == cudaSuccess &&
         cudaMalloc(&t->inv_cnorm, align_up(S * sizeof(float), 256)) == cudaSuccess &&
         cudaMalloc(&t->bias, align_up(S * sizeof(float), 256)) == cudaSuccess &&
         cudaMalloc(&t->status, 256) == cudaSuccess;
    if (!ok) {
        cudaGetLastError();
        destroy_table(t);
        return fail(LOOKME_ERR_OOM, "table allocation failed (%zu key bytes, %zu value bytes)", kbytes, vbytes);
    }
    if (cudaMemset(t->bias, 0, S * sizeof(float)) != cudaSuccess ||
        cudaMemset(t->inv_cnorm, 0, align_up(S * sizeof(float), 256)) != cudaSuccess ||
        cudaMemset(t->status, 0, 256) != cudaSuccess) {
        destroy_table(t);
        return fail(LOOKME_ERR_CUDA, "table initialisation failed");
    }
    if (t->tc_route) {
        for (int i = 0; i < 3; ++i) {
            if (!encode_bf16_2d(&t->tmap_c[i], t->cent, d.n_scenes, d.d_key, 64 << i)) {
                destroy_table(t);
                return fail(LOOKME_ERR_CUDA, "cuTensorMapEncodeTiled failed for the centroids");
            }
        }
    }
    if (d.max_tokens > 0) {
        lookme_status st = ensure_scratch(t, d.max_tokens, nullptr);
        if (st != LOOKME_OK) {
            destroy_table(t);
            return st;
        }
    }
    if (cudaDeviceSynchronize() != cudaSuccess) {
        destroy_table(t);
        return fail(LOOKME_ERR_CUDA, "table creation: %s", cudaGetErrorString(cudaGetLastError()));
    }
    *out = t;
    return LOOKME_OK;
}

lookme_status lookme_table_destroy(lookme_table* t) {
    if (!t) return LOOKME_OK;
    DeviceGuard guard(t->d.device);
    cudaDeviceSynchronize();
    destroy_table(t);
    return LOOKME_OK;
}

lookme_status lookme_reserve(lookme_table* t, int64_t max_tokens) {
    lookme_status st = check_table(t);
    if (st != LOOKME_OK) return st;
    if (max_tokens < 0) return fail(LOOKME_ERR_INVALID_ARG, "max_tokens < 0");
    DeviceGuard guard(t->d.device);
    return ensure_scratch(t, max_tokens, nullptr);
}

// Forgets what the HBM slot cache holds (asynchronous, on stream s).
cudaError_t stage_invalidate(lookme_table* t, cudaStream_t s) {
    const StageArgs& g = t->stage;
    cudaError_t e = cudaMemsetAsync(g.slot_of, 0xFF, t->d.n_scenes * sizeof(int32_t), s);
    if (e == cudaSuccess) e = cudaMemsetAsync(g.slot_scene, 0xFF, t->n_slots * sizeof(int32_t), s);
    if (e == cudaSuccess) e = cudaMemsetAsync(g.slot_stamp, 0, t->n_slots * sizeof(int32_t), s);
    if (e == cudaSuccess) e = cudaMemsetAsync(g.hdr, 0, sizeof(StageCache), s);
    return e;
}

lookme_status lookme_set_grids(lookme_table* t, int32_t route_sms, int32_t level2_ctas) {
    if (!t) return fail(LOOKME_ERR_INVALID_ARG, "table is NULL");
    if (route_sms < 0 || level2_ctas < 0)
        return fail(LOOKME_ERR_INVALID_ARG, "grid sizes must be >= 0 (got %d, %d)", (int)route_sms, (int)level2_ctas);
    t->small_sms = route_sms;
    t->level2_ctas = level2_ctas;
    return LOOKME_OK;
}

lookme_status lookme_stage_invalidate(lookme_table* t, lookme_stream stream) {
    lookme_status st = check_table(t);
    if (st != LOOKME_OK) return st;
    if (t->d.residency != LOOKME_RES_HOST_STAGED) return LOOKME_OK;
    DeviceGuard guard(t->d.device);
    cudaError_t e = stage_invalidate(t, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(t, e, "slot cache reset");
    return LOOKME_OK;
}

lookme_status lookme_load_scenes(lookme_table* t, int64_t scene_begin, int64_t n, const void* centroids,
                                 const void* keys, const void* values, const float* bias, int src_on_device,
                                 lookme_stream stream) {
    lookme_status st = check_table(t);
    if (st != LOOKME_OK) return st;
    const lookme_table_desc& d = t->d;
    if (n < 0 || scene_begin < 0 || scene_begin + n > d.n_scenes)
        return fail(LOOKME_ERR_INVALID_ARG, "scene range [%lld, %lld) outside [0, %lld)", (long long)scene_begin,
                    (long long)(scene_begin + n), (long long)d.n_scenes);
    if (!keys || !values) return fail(LOOKME_ERR_INVALID_ARG, "keys and values are required");
    if (n == 0) return LOOKME_OK;
    (void)src_on_device;  // copies use unified addressing and work for either source
    DeviceGuard guard(d.device);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    LaunchCtx ctx{s, t->num_sms};
    const size_t P = d.n_prims;
    const size_t krow = P * d.d_key * t->esz, vrow = P * d.d_value * t->esz;
    char* kdst = static_cast<char*>(d.residency == LOOKME_RES_DEVICE ? t->keys : t->keys_host);
    char* vdst = static_cast<char*>(d.residency == LOOKME_RES_DEVICE ? t->values : t->values_host);
    cudaError_t e;
    // Row-major keys readable by the device: the stored copy itself, or (tiled
    // tables) a stream-ordered temporary that the tiling kernel reads.
    const char* krows = nullptr;
    void* ktmp = nullptr;
    if (t->tc_score) {
        if ((e = cudaMallocAsync(&ktmp, n * krow, s)) != cudaSuccess) return cuda_fail(t, e, "key staging buffer");
        if ((e = cudaMemcpyAsync(ktmp, keys, n * krow, cudaMemcpyDefault, s)) != cudaSuccess)
            return cuda_fail(t, e, "copy keys");
        krows = static_cast<const char*>(ktmp);
        // The tiled block goes through the device view of the destination.
        char* tdst = static_cast<char*>(t->keys) + scene_begin * t->kblock;
        st = launch(t, s, KID_TILE_KEYS,
                    [&] { return launch_tile_keys(ctx, ktmp, tdst, n, d.n_prims, (int)d.d_key); });
        if (st != LOOKME_OK) return st;
    } else {
        if ((e = cudaMemcpyAsync(kdst + scene_begin * krow, keys, n * krow, cudaMemcpyDefault, s)) != cudaSuccess)
            return cuda_fail(t, e, "copy keys");
        krows = static_cast<const char*>(t->keys) + scene_begin * krow;  // device view of the stored keys
    }
    if ((e = cudaMemcpyAsync(vdst + scene_begin * vrow, values, n * vrow, cudaMemcpyDefault, s)) != cudaSuccess)
        return cuda_fail(t, e, "copy values");
    char* cdst = static_cast<char*>(t->cent) + scene_begin * d.d_key * t->esz;
    if (centroids) {
        if ((e = cudaMemcpyAsync(cdst, centroids, n * d.d_key * t->esz, cudaMemcpyDefault, s)) != cudaSuccess)
            return cuda_fail(t, e, "copy centroids");
    } else {
        st = launch(t, s, KID_CENTROID,
                    [&] { return launch_centroid_mean(ctx, d.dtype, krows, n, d.n_prims, (int)d.d_key, cdst); });
        if (st != LOOKME_OK) return st;
    }
    if (ktmp && (e = cudaFreeAsync(ktmp, s)) != cudaSuccess) return cuda_fail(t, e, "free key staging buffer");
    st = launch(t, s, KID_CNORM, [&] {
        return launch_inv_cnorm(ctx, d.dtype, cdst, n, (int)d.d_key, t->inv_cnorm + scene_begin);
    });
    if (st != LOOKME_OK) return st;
    if (bias) {
        if ((e = cudaMemcpyAsync(t->bias + scene_begin, bias, n * sizeof(float), cudaMemcpyDefault, s)) !=
            cudaSuccess)
            return cuda_fail(t, e, "copy bias");
        t->has_bias = true;
    }
    t->rk_c1_stale = true;  // the ranker's per-scene term depends on the centroids
    // Cached key blocks of reloaded scenes would be stale: start the slot
    // cache afresh.
    if (d.residency == LOOKME_RES_HOST_STAGED && (e = stage_invalidate(t, s)) != cudaSuccess)
        return cuda_fail(t, e, "slot cache reset");
    for (int64_t i = scene_begin; i < scene_begin + n; ++i) {
        if (!t->loaded[i]) {
            t->loaded[i] = 1;
            ++t->n_loaded;
        }
    }
    return LOOKME_OK;
}

}  // extern "C"

namespace {

// Argument checks shared by every lookup entry point.
lookme_status check_lookup(const lookme_table* t, const void* queries, int64_t N, int32_t top_k,
                           const int32_t* scene_out, const int32_t* prim_out, const float* weight_out) {
    const lookme_table_desc& d = t->d;
    if (N < 0 || N > INT32_MAX / 2) return fail(LOOKME_ERR_INVALID_ARG, "n_tokens %lld out of range", (long long)N);
    if (top_k < 1 || top_k > LOOKME_MAX_TOP_K || top_k > d.n_prims)
        return fail(LOOKME_ERR_INVALID_ARG, "top_k %d outside [1, min(n_prims, %d)]", top_k, LOOKME_MAX_TOP_K);
    if (N > 0 && (!queries || !scene_out || !prim_out || !weight_out))
        return fail(LOOKME_ERR_INVALID_ARG, "queries, scene_out, prim_out and weight_out are required");
    if (N > 0 && !aligned16(queries)) return fail(LOOKME_ERR_INVALID_ARG, "queries must be 16-byte aligned");
    if (t->n_loaded != d.n_scenes)
        return fail(LOOKME_ERR_STATE, "%lld of %lld scenes loaded", (long long)t->n_loaded, (long long)d.n_scenes);
    if (d.residency == LOOKME_RES_HOST_STAGED && std::min<int64_t>(N, d.n_scenes) > t->n_slots)
        return fail(LOOKME_ERR_UNSUPPORTED, "up to %lld routed scenes in one call but only %lld staging slots",
                    (long long)std::min<int64_t>(N, d.n_scenes), (long long)t->n_slots);
    return LOOKME_OK;
}

// Whether a call of N tokens (with n_seg gate segments) runs as the fused step.
bool step_eligible(const lookme_table* t, int64_t N, int32_t top_k, int n_seg) {
    const lookme_table_desc& d = t->d;
    return t->use_step && d.residency == LOOKME_RES_DEVICE && N >= 1 && N <= kStepMaxTokens &&
           top_k <= kRecMaxTopK && n_seg <= kMaxGateSegments &&
           step_shape_supported(N, d.n_scenes, d.n_prims, (int)d.d_key, (int)d.d_value, t->num_sms);
}

// The whole call as one launch of the fused step kernel.  With gate_off
// (the gate's segment offsets, n_seg + 1 of them) the call also decides the
// gate and injects; without it, it is a lookup.  Arguments are checked.
lookme_status run_step(lookme_table* t, cudaStream_t s, const void* queries, int64_t N, int32_t top_k,
                       int32_t* scene_out, int32_t* prim_out, float* weight_out, float* qnorm_out,
                       const int64_t* gate_off, int n_seg, double keep_ratio, const float* priority,
                       void* const* hidden, int32_t n_layers, uint8_t* mask_out) {
    const lookme_table_desc& d = t->d;
    lookme_status st;
    if ((st = ensure_scratch(t, N, s)) != LOOKME_OK) return st;
    CUtensorMap mq;
    if (!encode_bf16_2d(&mq, queries, N, d.d_key, 128))
        return fail(LOOKME_ERR_CUDA, "cuTensorMapEncodeTiled failed for the queries");
    const void* mc[3] = {&t->tmap_c[0], &t->tmap_c[1], &t->tmap_c[2]};
    StepArgs a;
    memset(&a, 0, sizeof(a));
    a.N = N;
    a.S = d.n_scenes;
    a.P = d.n_prims;
    a.dk = (int)d.d_key;
    a.dv = (int)d.d_value;
    a.top_k = top_k;
    a.scale = (float)(1.0 / std::sqrt((double)d.d_key));
    a.q = queries;
    a.keys_tiled = t->keys;
    a.block_bytes = t->kblock;
    a.values = t->values;
    a.inv_cnorm = t->inv_cnorm;
    a.bias = t->has_bias ? t->bias : nullptr;
    a.scene_out = scene_out;
    a.prim_out = prim_out;
    a.weight_out = weight_out;
    a.qnorm = t->qnorm;
    a.qnorm_out = qnorm_out;
    a.gate = gate_off ? 1 : 0;
    a.n_seg = gate_off ? n_seg : 1;
    a.priority = priority;
    a.mask_out = mask_out;
    if (gate_off) {
        for (int i = 0; i <= n_seg; ++i) a.seg_off[i] = gate_off[i];
        for (int i = 0; i < n_seg; ++i)
            a.seg_r[i] = (int64_t)std::floor((double)(gate_off[i + 1] - gate_off[i]) * keep_ratio);
        a.n_layers = n_layers;
        for (int l = 0; l < n_layers; ++l) a.hidden[l] = hidden[l];
    } else {
        a.seg_off[1] = N;
    }
    a.state = t->step;
    a.work = t->work;
    a.item_tok = t->item_tok;
    a.counters = t->counters;
    a.status = t->status;
    a.rec_row = t->rec_row;
    a.rec_w = t->rec_w;
    a.ovf_tok = t->step_ovf;
    LaunchCtx ctx{s, t->num_sms};
    st = launch(t, s, KID_STEP, [&] { return launch_step(ctx, &mq, mc, a); });
    if (st != LOOKME_OK) return st;
    t->last_tokens = N;
    return LOOKME_OK;
}

// lookme_lookup; with gate the bucketing kernel also computes the injection gate.
lookme_status lookup_impl(lookme_table* t, const void* queries, int64_t N, int32_t top_k, int32_t* scene_out,
                          int32_t* prim_out, float* weight_out, float* qnorm_out, lookme_stream stream,
                          const GateSpec* gate, const void* hidden0 = nullptr, bool records = false) {
    lookme_status st = check_table(t);
    if (st != LOOKME_OK) return st;
    const lookme_table_desc& d = t->d;
    if ((st = check_lookup(t, queries, N, top_k, scene_out, prim_out, weight_out)) != LOOKME_OK) return st;
    if (N == 0) return LOOKME_OK;
    DeviceGuard guard(d.device);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (!gate && step_eligible(t, N, top_k, 1))
        return run_step(t, s, queries, N, top_k, scene_out, prim_out, weight_out, qnorm_out, nullptr, 1, 0.0, nullptr,
                        nullptr, 0, nullptr);
    if ((st = ensure_scratch(t, N, s)) != LOOKME_OK) return st;
    LaunchCtx ctx{s, t->num_sms};
    // Routing and bucketing grids: sized for small_sms SMs when it is set.
    const LaunchCtx rctx{s, t->small_sms > 0 ? std::min(t->small_sms, t->num_sms) : t->num_sms};
    const int dk = (int)d.d_key;
    const float* bias = t->has_bias ? t->bias : nullptr;

    if (t->tc_route) {
        // The tcgen05 routing kernel computes the query norms itself; the
        // argmax keys were reset by the previous call's bucketing (or are
        // fresh zeroed scratch).
        CUtensorMap mq;
        if (!encode_bf16_2d(&mq, queries, N, dk, 128))
            return fail(LOOKME_ERR_CUDA, "cuTensorMapEncodeTiled failed for the queries");
        const void* mc[3] = {&t->tmap_c[0], &t->tmap_c[1], &t->tmap_c[2]};
        st = launch(t, s, KID_ROUTE_TC, [&] {
            return launch_route_tc(rctx, &mq, mc, N, d.n_scenes, dk, t->inv_cnorm, bias, t->qnorm, qnorm_out, t->best,
                                   t->status);
        });
    } else {
        st = launch(t, s, KID_PREP,
                    [&] { return launch_prep(rctx, d.dtype, queries, N, dk, t->qnorm, qnorm_out, t->best); });
        if (st != LOOKME_OK) return st;
        st = launch(t, s, KID_ROUTE_SIMT, [&] {
            return launch_route_simt(rctx, d.dtype, queries, t->cent, N, d.n_scenes, dk, t->inv_cnorm, bias, t->qnorm,
                                     t->best);
        });
    }
    if (st != LOOKME_OK) return st;
    // Large calls without the gate: the bucketing over all SMs in three
    // launches.  With the gate, its CTAs dominate and run beside the
    // single-CTA sort, which is then the faster choice.
    if (N <= kBucketOneCtaTokens || gate) {
        st = launch(t, s, KID_BUCKET, [&] {
            return launch_bucket(rctx, t->best, N, d.n_scenes, scene_out, t->item_tok, t->work, t->routed,
                                 t->counters, gate);
        });
    } else {
        st = launch(t, s, KID_BUCKET_COUNT, [&] {
            return launch_bucket_count(rctx, t->best, N, d.n_scenes, scene_out, t->scene_cnt, gate);
        });
        if (st == LOOKME_OK)
            st = launch(t, s, KID_BUCKET_SCAN, [&] {
                return launch_bucket_scan(rctx, d.n_scenes, t->scene_cnt, t->scene_pos, t->work, t->routed,
                                          t->counters);
            });
        if (st == LOOKME_OK)
            st = launch(t, s, KID_BUCKET_SCATTER, [&] {
                return launch_bucket_scatter(rctx, t->best, N, scene_out, t->scene_pos, t->item_tok);
            });
    }
    if (st != LOOKME_OK) return st;
    const bool staged = d.residency == LOOKME_RES_HOST_STAGED;
    if (staged) {
        // Slot look-up on the caller's stream; the copies of the misses on the
        // table's staging stream, forked after the look-up and joined before
        // level 2 (the next call's copies therefore start only after this
        // call's level 2, which reads the slots, is done).
        st = launch(t, s, KID_STAGE_ASSIGN, [&] {
            return launch_stage_assign(ctx, t->stage, t->routed, t->counters, t->work, t->status);
        });
        if (st != LOOKME_OK) return st;
        cudaError_t e = cudaEventRecord(t->ev_fork, s);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(t->stage_stream, t->ev_fork, 0);
        if (e != cudaSuccess) return cuda_fail(t, e, "staging fork");
        LaunchCtx sctx{t->stage_stream, t->num_sms};
        st = launch(t, t->stage_stream, KID_STAGE,
                    [&] { return launch_stage(sctx, t->keys, t->slots, t->kblock, t->stage); });
        if (st != LOOKME_OK) return st;
        e = cudaEventRecord(t->ev_join, t->stage_stream);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(s, t->ev_join, 0);
        if (e != cudaSuccess) return cuda_fail(t, e, "staging join");
    }
    ScoreArgs a;
    a.dtype = d.dtype;
    a.q = queries;
    a.keys = staged ? t->slots : t->keys;
    a.P = d.n_prims;
    a.dk = dk;
    a.top_k = top_k;
    a.scale = (float)(1.0 / std::sqrt((double)dk));
    a.work = t->work;
    a.work_cap = t->cap + d.n_scenes;
    a.counters = t->counters;
    a.item_tok = t->item_tok;
    a.use_slots = staged ? 1 : 0;
    a.prim_out = prim_out;
    a.weight_out = weight_out;
    a.status = t->status;
    // With the gate decided beside the bucketing, level 2 prefetches the kept
    // tokens' value rows (HBM-resident tables) and, with records, writes each
    // kept token's injection record at its slot.
    const bool gated = gate && gate->selpos && d.residency == LOOKME_RES_DEVICE;
    a.selpos = gated ? gate->selpos : nullptr;
    a.values = t->values;
    a.vrow_bytes = d.d_value * (int64_t)t->esz;
    a.hidden0 = gated ? hidden0 : nullptr;
    a.rec_t = gated && records ? t->rec_t : nullptr;
    a.rec_row = gated && records ? t->rec_row : nullptr;
    a.rec_w = gated && records ? t->rec_w : nullptr;
    st = launch(t, s, KID_SCORE,
                [&] {
                    if (!t->tc_score) return launch_score(ctx, a);
                    // The level-2 grid: level2_ctas CTAs when it is set.
                    const LaunchCtx lctx{s, t->level2_ctas > 0 ? std::min(t->level2_ctas, t->num_sms) : t->num_sms};
                    return launch_score_tc(lctx, a.keys, a);
                });
    if (st != LOOKME_OK) return st;
    t->last_tokens = N;
    return LOOKME_OK;
}

// Validated injection arguments: segment offsets (host), kept count, longest segment.
struct InjectPlan {
    std::vector<int64_t> off;
    int n_seg = 1;
    int64_t n_sel = 0, max_seg = 0;
};

lookme_status plan_inject(const lookme_table* t, int64_t N, int32_t top_k, const int64_t* seg_offsets, int32_t n_seg,
                          double keep_ratio, void* const* hidden, int32_t n_layers, InjectPlan& plan) {
    const lookme_table_desc& d = t->d;
    if (N < 0 || N > INT32_MAX / 2) return fail(LOOKME_ERR_INVALID_ARG, "n_tokens %lld out of range", (long long)N);
    if (top_k < 1 || top_k > LOOKME_MAX_TOP_K || top_k > d.n_prims)
        return fail(LOOKME_ERR_INVALID_ARG, "top_k %d outside [1, min(n_prims, %d)]", top_k, LOOKME_MAX_TOP_K);
    if (!(keep_ratio >= 0.0 && keep_ratio <= 1.0)) return fail(LOOKME_ERR_INVALID_ARG, "keep_ratio outside [0, 1]");
    if (n_layers < 1 || n_layers > LOOKME_MAX_LAYERS)
        return fail(LOOKME_ERR_INVALID_ARG, "n_layers %d outside [1, %d]", n_layers, LOOKME_MAX_LAYERS);
    if (!hidden) return fail(LOOKME_ERR_INVALID_ARG, "hidden is NULL");
    for (int l = 0; l < n_layers; ++l) {
        if (N > 0 && (!hidden[l] || !aligned16(hidden[l])))
            return fail(LOOKME_ERR_INVALID_ARG, "hidden[%d] is NULL or not 16-byte aligned", l);
    }
    if (seg_offsets) {
        if (n_seg < 1 || n_seg > LOOKME_MAX_SEGMENTS)
            return fail(LOOKME_ERR_INVALID_ARG, "n_seg %d outside [1, %d]", n_seg, LOOKME_MAX_SEGMENTS);
        plan.off.assign(seg_offsets, seg_offsets + n_seg + 1);
        if (plan.off[0] != 0 || plan.off[n_seg] != N)
            return fail(LOOKME_ERR_INVALID_ARG, "seg_offsets must start at 0 and end at n_tokens");
        for (int i = 0; i < n_seg; ++i)
            if (plan.off[i + 1] < plan.off[i]) return fail(LOOKME_ERR_INVALID_ARG, "seg_offsets must be non-decreasing");
        plan.n_seg = n_seg;
    } else {
        plan.n_seg = 1;
        plan.off = {0, N};
    }
    plan.n_sel = 0;
    plan.max_seg = 0;
    for (int i = 0; i < plan.n_seg; ++i) {
        const int64_t len = plan.off[i + 1] - plan.off[i];
        plan.n_sel += (int64_t)std::floor((double)len * keep_ratio);
        plan.max_seg = std::max(plan.max_seg, len);
    }
    return LOOKME_OK;
}

InjectArgs inject_args(const lookme_table* t, const int32_t* scene, const int32_t* prim, const float* weight,
                       int64_t N, int32_t top_k, void* const* hidden, int32_t n_layers, int32_t* sel, int64_t n_sel) {
    const lookme_table_desc& d = t->d;
    InjectArgs a;
    a.dtype = d.dtype;
    a.values = t->values;
    a.P = d.n_prims;
    a.dv = (int)d.d_value;
    a.top_k = top_k;
    a.scene = scene;
    a.prim = prim;
    a.weight = weight;
    a.sel = sel;
    a.n_sel = n_sel;
    a.N = N;
    a.S = d.n_scenes;
    a.n_layers = n_layers;
    for (int l = 0; l < n_layers; ++l) a.hidden[l] = hidden[l];
    a.status = t->status;
    return a;
}

}  // namespace

extern "C" {

lookme_status lookme_lookup(lookme_table* t, const void* queries, int64_t N, int32_t top_k, int32_t* scene_out,
                            int32_t* prim_out, float* weight_out, float* qnorm_out, lookme_stream stream) {
    return lookup_impl(t, queries, N, top_k, scene_out, prim_out, weight_out, qnorm_out, stream, nullptr);
}

lookme_status lookme_inject(lookme_table* t, const int32_t* scene, const int32_t* prim, const float* weight,
                            int64_t N, int32_t top_k, const float* priority, const int64_t* seg_offsets,
                            int32_t n_seg, double keep_ratio, void* const* hidden, int32_t n_layers,
                            uint8_t* mask_out, int32_t* sel_out, lookme_stream stream) {
    lookme_status st = check_table(t);
    if (st != LOOKME_OK) return st;
    InjectPlan plan;
    if ((st = plan_inject(t, N, top_k, seg_offsets, n_seg, keep_ratio, hidden, n_layers, plan)) != LOOKME_OK) return st;
    if (N == 0) return LOOKME_OK;
    if (!scene || !prim || !weight) return fail(LOOKME_ERR_INVALID_ARG, "scene, prim and weight are required");
    if (!priority && t->last_tokens != N)
        return fail(LOOKME_ERR_STATE, "default priority needs a lookup of %lld tokens first", (long long)N);

    DeviceGuard guard(t->d.device);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if ((st = ensure_scratch(t, N, s)) != LOOKME_OK) return st;
    LaunchCtx ctx{s, t->num_sms};
    uint8_t* mask = mask_out ? mask_out : t->mask;
    int32_t* sel = sel_out ? sel_out : t->sel;
    const float* pr = priority ? priority : t->qnorm;
    const InjectArgs a = inject_args(t, scene, prim, weight, N, top_k, hidden, n_layers, sel, plan.n_sel);
    // Short segments and no kept-id list: selection fused into the injection.
    if (!sel_out && plan.max_seg <= kFusedMaxSegment)
        return launch(t, s, KID_SELECT_INJECT, [&] {
            return launch_select_inject(ctx, a, pr, plan.off.data(), plan.n_seg, keep_ratio, mask);
        });
    st = launch(t, s, KID_SELECT,
                [&] { return launch_select(ctx, pr, N, plan.off.data(), plan.n_seg, keep_ratio, mask, sel); });
    if (st != LOOKME_OK) return st;
    if (plan.n_sel == 0) return LOOKME_OK;
    return launch(t, s, KID_INJECT, [&] { return launch_inject(ctx, a); });
}

lookme_status lookme_lookup_inject(lookme_table* t, const void* queries, int64_t N, int32_t top_k,
                                   const float* priority, const int64_t* seg_offsets, int32_t n_seg,
                                   double keep_ratio, void* const* hidden, int32_t n_layers, int32_t* scene_out,
                                   int32_t* prim_out, float* weight_out, uint8_t* mask_out, lookme_stream stream) {
    lookme_status st = check_table(t);
    if (st != LOOKME_OK) return st;
    InjectPlan plan;
    if ((st = plan_inject(t, N, top_k, seg_offsets, n_seg, keep_ratio, hidden, n_layers, plan)) != LOOKME_OK) return st;
    if (step_eligible(t, N, top_k, plan.n_seg)) {
        // Everything in one launch of the fused step kernel.
        if ((st = check_lookup(t, queries, N, top_k, scene_out, prim_out, weight_out)) != LOOKME_OK) return st;
        DeviceGuard guard(t->d.device);
        return run_step(t, static_cast<cudaStream_t>(stream), queries, N, top_k, scene_out, prim_out, weight_out,
                        nullptr, plan.off.data(), plan.n_seg, keep_ratio, priority, hidden, n_layers, mask_out);
    }
    const bool gate_in_lookup = N > 0 && plan.n_seg <= kMaxGateSegments && plan.max_seg <= kFusedMaxSegment;
    if (!gate_in_lookup) {
        // The two calls in sequence; with PDL the injection kernel's launch
        // overlaps the tail of the level-2 kernel.
        st = lookme_lookup(t, queries, N, top_k, scene_out, prim_out, weight_out, nullptr, stream);
        if (st != LOOKME_OK) return st;
        return lookme_inject(t, scene_out, prim_out, weight_out, N, top_k, priority, seg_offsets, n_seg, keep_ratio,
                             hidden, n_layers, mask_out, nullptr, stream);
    }
    // The bucketing kernel's extra CTAs decide the gate and list the kept
    // tokens while it sorts; the injection then runs on the kept tokens only.
    DeviceGuard guard(t->d.device);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if ((st = ensure_scratch(t, N, s)) != LOOKME_OK) return st;
    GateSpec gs;
    memset(&gs, 0, sizeof(gs));
    gs.enabled = 1;
    gs.n_seg = plan.n_seg;
    gs.N = N;
    gs.keep_ratio = keep_ratio;
    gs.priority = priority ? priority : t->qnorm;
    gs.mask = mask_out ? mask_out : t->mask;
    gs.sel = t->sel;
    gs.selpos = t->selpos;
    int64_t base = 0;
    for (int i = 0; i < plan.n_seg; ++i) {
        gs.off[i] = plan.off[i];
        gs.sel_base[i] = base;
        base += (int64_t)std::floor((double)(plan.off[i + 1] - plan.off[i]) * keep_ratio);
    }
    gs.off[plan.n_seg] = plan.off[plan.n_seg];
    // The tcgen05 level-2 kernel writes each kept token's injection record
    // (token, value rows, weights) at its slot, and the injection reads them
    // in one round trip.
    const lookme_table_desc& d = t->d;
    const bool records = t->tc_score && d.residency == LOOKME_RES_DEVICE && top_k <= kRecMaxTopK &&
                         d.n_scenes * d.n_prims < (int64_t)INT32_MAX;
    st = lookup_impl(t, queries, N, top_k, scene_out, prim_out, weight_out, nullptr, stream, &gs, hidden[0],
                     records);
    if (st != LOOKME_OK) return st;
    if (plan.n_sel == 0) return LOOKME_OK;
    LaunchCtx ctx{s, t->num_sms};
    const InjectArgs a =
        inject_args(t, scene_out, prim_out, weight_out, N, top_k, hidden, n_layers, t->sel, plan.n_sel);
    if (records)
        return launch(t, s, KID_INJECT,
                      [&] { return launch_inject_records(ctx, a, t->rec_t, t->rec_row, t->rec_w); });
    return launch(t, s, KID_INJECT, [&] { return launch_inject(ctx, a); });
}

lookme_status lookme_last_lookup_stats(lookme_table* t, lookme_lookup_stats* out, lookme_stream stream) {
    lookme_status st = check_table(t);
    if (st != LOOKME_OK) return st;
    if (!out) return fail(LOOKME_ERR_INVALID_ARG, "out is NULL");
    memset(out, 0, sizeof(*out));
    if (t->last_tokens < 0 || !t->counters) return LOOKME_OK;
    DeviceGuard guard(t->d.device);
    int32_t c[4];
    StageCache hc{};
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaMemcpyAsync(c, t->counters, sizeof(c), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess && t->d.residency == LOOKME_RES_HOST_STAGED)
        e = cudaMemcpyAsync(&hc, t->stage.hdr, sizeof(hc), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(t, e, "read lookup stats");
    out->n_tokens = t->last_tokens;
    out->n_work_items = c[0];
    out->n_routed_scenes = c[1];
    out->staged_bytes = (int64_t)hc.n_copy * t->kblock;
    out->staged_hits = hc.n_hit;
    return LOOKME_OK;
}

lookme_status lookme_device_status(lookme_table* t, uint32_t* status, int reset, lookme_stream stream) {
    if (!t || !status) return fail(LOOKME_ERR_INVALID_ARG, "NULL argument");
    DeviceGuard guard(t->d.device);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaMemcpyAsync(status, t->status, sizeof(uint32_t), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e == cudaSuccess && reset) e = cudaMemsetAsync(t->status, 0, sizeof(uint32_t), s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(t, e, "read device status");
    return LOOKME_OK;
}

uint64_t lookme_launch_count(const lookme_table* t) { return t ? t->launches : 0; }

lookme_status lookme_trace_enable(lookme_table* t, int enable) {
    if (!t) return fail(LOOKME_ERR_INVALID_ARG, "table is NULL");
    t->trace = enable != 0;
    return LOOKME_OK;
}

lookme_status lookme_trace_read(lookme_table* t, lookme_trace_record* out, int32_t max, int32_t* n_out) {
    if (!t || !n_out || (max > 0 && !out)) return fail(LOOKME_ERR_INVALID_ARG, "NULL argument");
    DeviceGuard guard(t->d.device);
    int32_t n = 0;
    lookme_status st = LOOKME_OK;
    for (auto& te : t->trace_log) {
        float ms = 0.f;
        cudaError_t e = cudaEventSynchronize(te.stop);
        if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, te.start, te.stop);
        if (e != cudaSuccess && st == LOOKME_OK) st = cuda_fail(t, e, "trace event");
        if (n < max) out[n++] = lookme_trace_record{te.kernel, ms};
        t->event_pool.push_back(te.start);
        t->event_pool.push_back(te.stop);
    }
    t->trace_log.clear();
    *n_out = n;
    return st;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Level-1 routing that allocates nothing.
//
// Some callers cannot allocate device memory at the point where they route
// tokens: a serving loop whose device memory is owned by another allocator
// (for example a framework's caching allocator holding the whole card), code
// that must not pay the implicit device-wide synchronisation cudaMalloc and
// cudaFree can cause, or a real-time path with a fixed memory budget.
// lookme_route_scenes_static serves them: its per-token scratch (the packed
// argmax keys and the query norms) lives in the two fixed arrays below, which
// every GPU that loads this library holds until the process exits
// (LOOKME_ROUTE_STATIC_MAX_TOKENS x 12 bytes = 768 KiB per device).  Host code
// must not use the array names as device addresses: it asks the runtime for
// them once per device with cudaGetSymbolAddress.
static __device__ __align__(256) unsigned long long g_static_best[LOOKME_ROUTE_STATIC_MAX_TOKENS];
static __device__ __align__(256) float g_static_qnorm[LOOKME_ROUTE_STATIC_MAX_TOKENS];

namespace {

constexpr int kMaxDevices = 64;

struct StaticScratch {
    unsigned long long* best = nullptr;
    float* qnorm = nullptr;
};

std::mutex g_static_mu;
StaticScratch g_static_scratch[kMaxDevices];

// Device addresses of the fixed arrays on `device`, which must be current.
// Looked up on the first call per device and cached.
lookme_status static_scratch(int device, StaticScratch* out) {
    if (device < 0 || device >= kMaxDevices) return fail(LOOKME_ERR_UNSUPPORTED, "device %d out of range", device);
    std::lock_guard<std::mutex> lock(g_static_mu);
    StaticScratch& sc = g_static_scratch[device];
    if (!sc.best) {
        void* pb = nullptr;
        void* pq = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&pb, g_static_best);
        if (e != cudaSuccess) return fail(LOOKME_ERR_CUDA, "cudaGetSymbolAddress(best): %s", cudaGetErrorString(e));
        e = cudaGetSymbolAddress(&pq, g_static_qnorm);
        if (e != cudaSuccess) return fail(LOOKME_ERR_CUDA, "cudaGetSymbolAddress(qnorm): %s", cudaGetErrorString(e));
        sc.best = static_cast<unsigned long long*>(pb);
        sc.qnorm = static_cast<float*>(pq);
    }
    *out = sc;
    return LOOKME_OK;
}

// A token whose key is still 0 was never scored (the routing kernel gave up a
// bounded wait and set the status word): it gets scene -1, never a valid id.
__global__ void k_route_static_decode(const unsigned long long* __restrict__ best, int64_t N, int64_t S,
                                      int32_t* __restrict__ scene_out) {
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (t < N) {
        const unsigned long long k = best[t];
        scene_out[t] = k == 0ull ? -1 : unpack_scene(k, S);
    }
}

}  // namespace

extern "C" lookme_status lookme_route_scenes_static(lookme_table* t, const void* queries, int64_t N,
                                                    int32_t* scene_out, lookme_stream stream) {
    lookme_status st = check_table(t);
    if (st != LOOKME_OK) return st;
    const lookme_table_desc& d = t->d;
    if (N < 0 || N > LOOKME_ROUTE_STATIC_MAX_TOKENS)
        return fail(LOOKME_ERR_INVALID_ARG, "n_tokens %lld outside [0, %d], the size of the fixed scratch",
                    (long long)N, LOOKME_ROUTE_STATIC_MAX_TOKENS);
    if (N > 0 && (!queries || !scene_out)) return fail(LOOKME_ERR_INVALID_ARG, "queries and scene_out are required");
    if (N > 0 && !aligned16(queries)) return fail(LOOKME_ERR_INVALID_ARG, "queries must be 16-byte aligned");
    if (t->n_loaded != d.n_scenes)
        return fail(LOOKME_ERR_STATE, "%lld of %lld scenes loaded", (long long)t->n_loaded, (long long)d.n_scenes);
    if (N == 0) return LOOKME_OK;
    DeviceGuard guard(d.device);
    StaticScratch sc;
    if ((st = static_scratch(d.device, &sc)) != LOOKME_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    LaunchCtx ctx{s, t->num_sms};
    const int dk = (int)d.d_key;
    const float* bias = t->has_bias ? t->bias : nullptr;
    // Every key the routing kernel reduces into starts at 0, so leftovers of an
    // earlier call never leak into this one: cleared by a memset (allocates
    // nothing) before the tensor-core kernel, which computes the query norms
    // itself, or by the prep kernel, which also computes them, before the
    // CUDA-core one.
    if (t->tc_route) {
        cudaError_t e = cudaMemsetAsync(sc.best, 0, (size_t)N * sizeof(unsigned long long), s);
        if (e != cudaSuccess) return cuda_fail(t, e, "clear routing keys");
    } else {
        st = launch(t, s, KID_PREP, [&] { return launch_prep(ctx, d.dtype, queries, N, dk, sc.qnorm, nullptr, sc.best); });
        if (st != LOOKME_OK) return st;
    }
    if (t->tc_route) {
        CUtensorMap mq;
        if (!encode_bf16_2d(&mq, queries, N, dk, 128))
            return fail(LOOKME_ERR_CUDA, "cuTensorMapEncodeTiled failed for the queries");
        const void* mc[3] = {&t->tmap_c[0], &t->tmap_c[1], &t->tmap_c[2]};
        st = launch(t, s, KID_ROUTE_TC, [&] {
            return launch_route_tc(ctx, &mq, mc, N, d.n_scenes, dk, t->inv_cnorm, bias, sc.qnorm, nullptr, sc.best,
                                   t->status);
        });
    } else {
        st = launch(t, s, KID_ROUTE_SIMT, [&] {
            return launch_route_simt(ctx, d.dtype, queries, t->cent, N, d.n_scenes, dk, t->inv_cnorm, bias, sc.qnorm,
                                     sc.best);
        });
    }
    if (st != LOOKME_OK) return st;
    return launch(t, s, KID_ROUTE_DECODE, [&] {
        k_route_static_decode<<<(unsigned)((N + 255) / 256), 256, 0, s>>>(sc.best, N, d.n_scenes, scene_out);
        return cudaGetLastError();
    });
}
