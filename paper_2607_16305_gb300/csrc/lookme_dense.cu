// Host entry points of the pieces around the two-level lookup, declared in
// lookme.h: the paper-exact level 2 with its scene-shared ranker MLP, the SKA
// gate, injection on a given gate, the text pathway, the fusion f with the
// inter-layer propagation, the projection into the embedding space and the
// multi-scale router.  Same rules as the rest of the runtime: arguments are
// checked on the host first, the caller's device and stream are used, and
// nothing synchronises except the documented set-up calls.
#include "api_internal.cuh"

using namespace lookme_host;

namespace {

constexpr int kTmapBoxA = 128;

// D = A B^T on the tensor cores: A [M][K] and B [Nn][K] row-major bf16.
lookme_status gemm(lookme_table* t, cudaStream_t s, int num_sms, const void* A, const void* B, int64_t M,
                   int64_t Nn, int64_t K, GemmArgs g) {
    if (M == 0 || Nn == 0) return LOOKME_OK;
    if (K % 8 || (reinterpret_cast<uintptr_t>(A) & 15) || (reinterpret_cast<uintptr_t>(B) & 15))
        return fail(LOOKME_ERR_INVALID_ARG, "GEMM operands need 16-byte alignment and K %% 8 == 0");
    const int bn = gemm_tile_n(M, g.mode == EPI_SWIGLU ? Nn : Nn, num_sms);
    CUtensorMap ma, mb;
    if (!encode_bf16_2d(&ma, A, M, K, kTmapBoxA) || !encode_bf16_2d(&mb, B, Nn, K, bn))
        return fail(LOOKME_ERR_CUDA, "cuTensorMapEncodeTiled failed for a GEMM operand");
    g.M = M;
    g.Nn = Nn;
    g.K = K;
    LaunchCtx ctx{s, num_sms};
    if (t) return launch(t, s, KID_GEMM, [&] { return launch_gemm_tc(ctx, &ma, &mb, bn, g); });
    cudaError_t e = launch_gemm_tc(ctx, &ma, &mb, bn, g);
    if (e != cudaSuccess) return fail(LOOKME_ERR_CUDA, "gemm: %s", cudaGetErrorString(e));
    return LOOKME_OK;
}

GemmArgs gemm_args(int mode, void* out, int64_t ld_out, uint32_t* status) {
    GemmArgs g;
    memset(&g, 0, sizeof(g));
    g.mode = mode;
    g.out = out;
    g.ld_out = ld_out;
    g.status = status;
    return g;
}

int current_sms() {
    int dev = 0, n = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n > 0 ? n : 1;
}

int64_t round_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

// Ranker scratch for up to `cap` tokens: H [cap][d_m] bf16, r [cap][ld_r] fp32.
lookme_status ensure_ranker_scratch(lookme_table* t, int64_t n, cudaStream_t s) {
    if (n <= t->rk_cap && t->rk_scratch) return LOOKME_OK;
    if (s && capturing(s))
        return fail(LOOKME_ERR_STATE, "ranker scratch must grow to %lld tokens while the stream is captured",
                    (long long)n);
    const int64_t cap = std::max<int64_t>(n, 1);
    const int64_t ld_r = round_up(t->d.n_prims, 4);
    const size_t bytes = align_up(cap * t->rk_dm * 2, 256) + cap * ld_r * 4;
    void* buf = nullptr;
    if (cudaDeviceSynchronize() != cudaSuccess || cudaMalloc(&buf, bytes) != cudaSuccess) {
        cudaGetLastError();
        return fail(LOOKME_ERR_OOM, "ranker scratch of %zu bytes", bytes);
    }
    if (t->rk_scratch) cudaFree(t->rk_scratch);
    t->rk_scratch = buf;
    t->rk_cap = cap;
    return LOOKME_OK;
}

}  // namespace

extern "C" {

lookme_status lookme_set_ranker(lookme_table* t, int64_t d_hidden, const void* W1, const float* b1, const void* W2,
                                const float* b2, lookme_stream stream) {
    lookme_status st = check_table(t);
    if (st != LOOKME_OK) return st;
    const lookme_table_desc& d = t->d;
    if (d.dtype != LOOKME_BF16) return fail(LOOKME_ERR_UNSUPPORTED, "the ranker runs on bf16 tables");
    if (d_hidden < 8 || d_hidden % 8 || d_hidden > 4096)
        return fail(LOOKME_ERR_INVALID_ARG, "d_hidden %lld: a multiple of 8 in [8, 4096]", (long long)d_hidden);
    if (!W1 || !b1 || !W2 || !b2) return fail(LOOKME_ERR_INVALID_ARG, "W1, b1, W2 and b2 are required");
    DeviceGuard guard(d.device);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int64_t dm = d_hidden, de = d.d_key, P = d.n_prims, S = d.n_scenes;
    if (t->rk_mem) {
        cudaStreamSynchronize(s);
        cudaFree(t->rk_mem);
        t->rk_mem = nullptr;
    }
    if (t->rk_scratch && t->rk_dm != dm) {
        cudaStreamSynchronize(s);
        cudaFree(t->rk_scratch);
        t->rk_scratch = nullptr;
        t->rk_cap = 0;
    }
    const size_t o_w1v = 0, o_w1c = align_up(o_w1v + dm * de * 2, 256), o_b1 = align_up(o_w1c + dm * de * 2, 256),
                 o_w2 = align_up(o_b1 + dm * 4, 256), o_b2 = align_up(o_w2 + P * dm * 2, 256),
                 o_c1 = align_up(o_b2 + P * 4, 256), total = align_up(o_c1 + S * dm * 4, 256);
    void* mem = nullptr;
    if (cudaMalloc(&mem, total) != cudaSuccess) {
        cudaGetLastError();
        return fail(LOOKME_ERR_OOM, "ranker weights of %zu bytes", total);
    }
    char* m = static_cast<char*>(mem);
    t->rk_mem = mem;
    t->rk_dm = dm;
    t->rk_w1v = reinterpret_cast<__nv_bfloat16*>(m + o_w1v);
    t->rk_w1c = reinterpret_cast<__nv_bfloat16*>(m + o_w1c);
    t->rk_b1 = reinterpret_cast<float*>(m + o_b1);
    t->rk_w2 = reinterpret_cast<__nv_bfloat16*>(m + o_w2);
    t->rk_b2 = reinterpret_cast<float*>(m + o_b2);
    t->rk_c1 = reinterpret_cast<float*>(m + o_c1);
    // W1 [d_m][2 d_k]: columns [0, d_k) multiply the query, [d_k, 2 d_k) the centroid.
    const char* w1 = static_cast<const char*>(W1);
    cudaError_t e = cudaMemcpy2DAsync(t->rk_w1v, de * 2, w1, 2 * de * 2, de * 2, dm, cudaMemcpyDefault, s);
    if (e == cudaSuccess)
        e = cudaMemcpy2DAsync(t->rk_w1c, de * 2, w1 + de * 2, 2 * de * 2, de * 2, dm, cudaMemcpyDefault, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(t->rk_b1, b1, dm * 4, cudaMemcpyDefault, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(t->rk_w2, W2, P * dm * 2, cudaMemcpyDefault, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(t->rk_b2, b2, P * 4, cudaMemcpyDefault, s);
    if (e != cudaSuccess) return cuda_fail(t, e, "ranker weights");
    t->rk_c1_stale = true;
    return LOOKME_OK;
}

lookme_status lookme_lookup_ranked(lookme_table* t, const void* queries, int64_t N, int32_t top_t, int32_t* scene_out,
                                   int32_t* prim_out, float* weight_out, lookme_stream stream) {
    lookme_status st = check_table(t);
    if (st != LOOKME_OK) return st;
    const lookme_table_desc& d = t->d;
    if (!t->rk_mem) return fail(LOOKME_ERR_STATE, "no ranker: call lookme_set_ranker first");
    if (N < 0 || N > INT32_MAX / 2) return fail(LOOKME_ERR_INVALID_ARG, "n_tokens %lld out of range", (long long)N);
    if (top_t < 1 || top_t > LOOKME_MAX_TOP_K || top_t > d.n_prims)
        return fail(LOOKME_ERR_INVALID_ARG, "top_t %d outside [1, min(n_prims, %d)]", top_t, LOOKME_MAX_TOP_K);
    if (N > 0 && (!queries || !scene_out || !prim_out || !weight_out))
        return fail(LOOKME_ERR_INVALID_ARG, "queries, scene_out, prim_out and weight_out are required");
    if (N > 0 && !aligned16(queries)) return fail(LOOKME_ERR_INVALID_ARG, "queries must be 16-byte aligned");
    if (t->n_loaded != d.n_scenes)
        return fail(LOOKME_ERR_STATE, "%lld of %lld scenes loaded", (long long)t->n_loaded, (long long)d.n_scenes);
    if (N == 0) return LOOKME_OK;
    DeviceGuard guard(d.device);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if ((st = ensure_scratch(t, N, s)) != LOOKME_OK) return st;
    if ((st = ensure_ranker_scratch(t, N, s)) != LOOKME_OK) return st;
    LaunchCtx ctx{s, t->num_sms};
    // lookme_set_grids: the routing grid and the GEMM tiles sized for route_sms SMs.
    const int gsms = t->small_sms > 0 ? std::min(t->small_sms, t->num_sms) : t->num_sms;
    const LaunchCtx rctx{s, gsms};
    const int dk = (int)d.d_key;
    const float* bias = t->has_bias ? t->bias : nullptr;
    const int64_t dm = t->rk_dm, P = d.n_prims, ld_r = round_up(P, 4);
    __nv_bfloat16* H = static_cast<__nv_bfloat16*>(t->rk_scratch);
    float* r = reinterpret_cast<float*>(static_cast<char*>(t->rk_scratch) + align_up(t->rk_cap * dm * 2, 256));

    // Level 1 (Sec. "Level-1: scene retrieval"): argmax keys, then scenes.
    if (t->tc_route) {
        CUtensorMap mq;
        if (!encode_bf16_2d(&mq, queries, N, dk, 128))
            return fail(LOOKME_ERR_CUDA, "cuTensorMapEncodeTiled failed for the queries");
        const void* mc[3] = {&t->tmap_c[0], &t->tmap_c[1], &t->tmap_c[2]};
        st = launch(t, s, KID_ROUTE_TC, [&] {
            return launch_route_tc(rctx, &mq, mc, N, d.n_scenes, dk, t->inv_cnorm, bias, t->qnorm, nullptr, t->best,
                                   t->status);
        });
    } else {
        st = launch(t, s, KID_PREP,
                    [&] { return launch_prep(rctx, d.dtype, queries, N, dk, t->qnorm, nullptr, t->best); });
        if (st == LOOKME_OK)
            st = launch(t, s, KID_ROUTE_SIMT, [&] {
                return launch_route_simt(rctx, d.dtype, queries, t->cent, N, d.n_scenes, dk, t->inv_cnorm, bias,
                                         t->qnorm, t->best);
            });
    }
    if (st != LOOKME_OK) return st;
    st = launch(t, s, KID_DECODE, [&] { return launch_decode_reset(ctx, t->best, N, d.n_scenes, scene_out); });
    if (st != LOOKME_OK) return st;
    // The ranker's per-scene term c1[s] = W1c e_img[s] + b1, once per change
    // of the centroids or the weights.
    if (t->rk_c1_stale) {
        GemmArgs g = gemm_args(EPI_F32, t->rk_c1, dm, t->status);
        g.colbias = t->rk_b1;
        if ((st = gemm(t, s, t->num_sms, t->cent, t->rk_w1c, d.n_scenes, dm, dk, g)) != LOOKME_OK) return st;
        t->rk_c1_stale = false;
    }
    // H = silu(q W1v^T + c1[scene]) (bf16), r = H W2^T + b2 (fp32).
    {
        GemmArgs g = gemm_args(EPI_BF16, H, dm, t->status);
        g.rowbias = t->rk_c1;
        g.rowsel = scene_out;
        g.ld_rowbias = dm;
        g.act = 1;
        if ((st = gemm(t, s, gsms, queries, t->rk_w1v, N, dm, dk, g)) != LOOKME_OK) return st;
    }
    {
        GemmArgs g = gemm_args(EPI_F32, r, ld_r, t->status);
        g.colbias = t->rk_b2;
        if ((st = gemm(t, s, gsms, H, t->rk_w2, N, P, dm, g)) != LOOKME_OK) return st;
    }
    // Top-T by r and the cos + tanh softmax, reading only the selected key rows.
    KeyView kv;
    kv.keys = static_cast<const uint8_t*>(t->keys);
    kv.block_bytes = t->kblock;
    kv.P = (int)P;
    kv.dk = dk;
    kv.tiled = t->tc_score ? 1 : 0;
    kv.ntile = (int)((P + 127) / 128);
    kv.nkb = (dk + 63) / 64;
    st = launch(t, s, KID_RANKED_SELECT, [&] {
        return launch_ranked_select(ctx, r, ld_r, N, top_t, static_cast<const __nv_bfloat16*>(queries), kv, scene_out,
                                    prim_out, weight_out);
    });
    if (st != LOOKME_OK) return st;
    t->last_tokens = N;
    return LOOKME_OK;
}

lookme_status lookme_ska_gate(const void* delta, const void* w_g, int64_t N, int64_t d_hidden, int32_t dtype,
                              uint8_t* gate_out, float* logit_out, lookme_stream stream) {
    if (dtype != LOOKME_BF16 && dtype != LOOKME_FP32) return fail(LOOKME_ERR_INVALID_ARG, "bad dtype %d", dtype);
    const int vec = dtype == LOOKME_BF16 ? 8 : 4;
    if (N < 0 || d_hidden < 1 || d_hidden % vec)
        return fail(LOOKME_ERR_INVALID_ARG, "N >= 0 and d_hidden a positive multiple of %d", vec);
    if (N == 0) return LOOKME_OK;
    if (!delta || !w_g || !gate_out) return fail(LOOKME_ERR_INVALID_ARG, "delta, w_g and gate_out are required");
    if (!aligned16(delta) || !aligned16(w_g)) return fail(LOOKME_ERR_INVALID_ARG, "delta and w_g: 16-byte aligned");
    LaunchCtx ctx{static_cast<cudaStream_t>(stream), current_sms()};
    cudaError_t e = launch_ska_gate(ctx, dtype, delta, w_g, N, d_hidden, gate_out, logit_out);
    if (e != cudaSuccess) return fail(LOOKME_ERR_CUDA, "ska_gate: %s", cudaGetErrorString(e));
    return LOOKME_OK;
}

lookme_status lookme_inject_gated(lookme_table* t, const int32_t* scene, const int32_t* prim, const float* weight,
                                  int64_t N, int32_t top_k, const uint8_t* gate, void* const* hidden, int32_t n_layers,
                                  lookme_stream stream) {
    lookme_status st = check_table(t);
    if (st != LOOKME_OK) return st;
    const lookme_table_desc& d = t->d;
    if (N < 0 || N > INT32_MAX / 2) return fail(LOOKME_ERR_INVALID_ARG, "n_tokens %lld out of range", (long long)N);
    if (top_k < 1 || top_k > LOOKME_MAX_TOP_K || top_k > d.n_prims)
        return fail(LOOKME_ERR_INVALID_ARG, "top_k %d outside [1, min(n_prims, %d)]", top_k, LOOKME_MAX_TOP_K);
    if (n_layers < 1 || n_layers > LOOKME_MAX_LAYERS || !hidden)
        return fail(LOOKME_ERR_INVALID_ARG, "hidden must list 1..%d layers", LOOKME_MAX_LAYERS);
    if (N == 0) return LOOKME_OK;
    if (!scene || !prim || !weight || !gate) return fail(LOOKME_ERR_INVALID_ARG, "scene, prim, weight and gate");
    for (int l = 0; l < n_layers; ++l)
        if (!hidden[l] || !aligned16(hidden[l])) return fail(LOOKME_ERR_INVALID_ARG, "hidden[%d]: NULL or unaligned", l);
    DeviceGuard guard(d.device);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    LaunchCtx ctx{s, t->num_sms};
    InjectArgs a;
    memset(&a, 0, sizeof(a));
    a.dtype = d.dtype;
    a.values = t->values;
    a.P = d.n_prims;
    a.dv = (int)d.d_value;
    a.top_k = top_k;
    a.scene = scene;
    a.prim = prim;
    a.weight = weight;
    a.N = N;
    a.S = d.n_scenes;
    a.n_layers = n_layers;
    for (int l = 0; l < n_layers; ++l) a.hidden[l] = hidden[l];
    return launch(t, s, KID_INJECT_GATED, [&] { return launch_inject_gated(ctx, a, gate); });
}

lookme_status lookme_combine(lookme_table* t, const int32_t* scene, const int32_t* prim, const float* weight,
                             int64_t n_tokens, int32_t top_k, const int32_t* rows, int64_t n_rows, void* R_out,
                             lookme_stream stream) {
    lookme_status st = check_table(t);
    if (st != LOOKME_OK) return st;
    const lookme_table_desc& d = t->d;
    if (d.dtype != LOOKME_BF16) return fail(LOOKME_ERR_UNSUPPORTED, "lookme_combine writes bf16 rows: bf16 tables only");
    if (top_k < 1 || top_k > LOOKME_MAX_TOP_K || top_k > d.n_prims)
        return fail(LOOKME_ERR_INVALID_ARG, "top_k %d outside [1, min(n_prims, %d)]", top_k, LOOKME_MAX_TOP_K);
    if (n_rows < 0 || n_rows > INT32_MAX / 2) return fail(LOOKME_ERR_INVALID_ARG, "n_rows out of range");
    if (n_rows == 0) return LOOKME_OK;
    if (!scene || !prim || !weight || !rows || !R_out || !aligned16(R_out))
        return fail(LOOKME_ERR_INVALID_ARG, "scene, prim, weight, rows and a 16-byte aligned R_out are required");
    DeviceGuard guard(d.device);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    LaunchCtx ctx{s, t->num_sms};
    InjectArgs a;
    memset(&a, 0, sizeof(a));
    a.dtype = d.dtype;
    a.values = t->values;
    a.P = d.n_prims;
    a.dv = (int)d.d_value;
    a.top_k = top_k;
    a.scene = scene;
    a.prim = prim;
    a.weight = weight;
    a.S = d.n_scenes;
    a.N = n_tokens;
    return launch(t, s, KID_COMBINE,
                  [&] { return launch_combine(ctx, a, rows, n_rows, static_cast<__nv_bfloat16*>(R_out)); });
}

lookme_status lookme_text_inject(const void* E, int64_t vocab, int64_t d, int32_t dtype, const int32_t* ids,
                                 const uint8_t* gate, int64_t N, void* const* hidden, int32_t n_layers,
                                 lookme_stream stream) {
    if (dtype != LOOKME_BF16 && dtype != LOOKME_FP32) return fail(LOOKME_ERR_INVALID_ARG, "bad dtype %d", dtype);
    const int vec = dtype == LOOKME_BF16 ? 8 : 4;
    if (N < 0 || N > INT32_MAX / 2 || vocab < 1 || d < 1 || d % vec)
        return fail(LOOKME_ERR_INVALID_ARG, "N >= 0, vocab >= 1, d a positive multiple of %d", vec);
    if (n_layers < 1 || n_layers > LOOKME_MAX_LAYERS || !hidden)
        return fail(LOOKME_ERR_INVALID_ARG, "hidden must list 1..%d layers", LOOKME_MAX_LAYERS);
    if (N == 0) return LOOKME_OK;
    if (!E || !ids || !aligned16(E)) return fail(LOOKME_ERR_INVALID_ARG, "a 16-byte aligned E and ids are required");
    for (int l = 0; l < n_layers; ++l)
        if (!hidden[l] || !aligned16(hidden[l])) return fail(LOOKME_ERR_INVALID_ARG, "hidden[%d]: NULL or unaligned", l);
    LaunchCtx ctx{static_cast<cudaStream_t>(stream), current_sms()};
    cudaError_t e = launch_text_inject(ctx, dtype, E, vocab, d, ids, gate, N, hidden, n_layers);
    if (e != cudaSuccess) return fail(LOOKME_ERR_CUDA, "text_inject: %s", cudaGetErrorString(e));
    return LOOKME_OK;
}

lookme_status lookme_project(const void* x, const void* W, const float* bias, int64_t N, int64_t d_in, int64_t d_out,
                             void* out, lookme_stream stream) {
    if (N < 0 || d_in < 8 || d_in % 8 || d_out < 8 || d_out % 8)
        return fail(LOOKME_ERR_INVALID_ARG, "N >= 0; d_in and d_out positive multiples of 8");
    if (N == 0) return LOOKME_OK;
    if (!x || !W || !out || !aligned16(out)) return fail(LOOKME_ERR_INVALID_ARG, "x, W and an aligned out are required");
    GemmArgs g = gemm_args(EPI_BF16, out, d_out, nullptr);
    g.colbias = bias;
    return gemm(nullptr, static_cast<cudaStream_t>(stream), current_sms(), x, W, N, d_out, d_in, g);
}

lookme_status lookme_scale_router(const void* H, const void* W_he, const void* const* R_scales, int32_t n_scales,
                                  int64_t N, int64_t d_hidden, int64_t d_embed, float* workspace, void* out,
                                  float* att_out, lookme_stream stream) {
    if (n_scales < 1 || n_scales > kRouterMaxScales)
        return fail(LOOKME_ERR_INVALID_ARG, "n_scales %d outside [1, %d]", n_scales, kRouterMaxScales);
    if (N < 0 || d_hidden < 8 || d_hidden % 8 || d_embed < 8 || d_embed % 8)
        return fail(LOOKME_ERR_INVALID_ARG, "N >= 0; d_hidden and d_embed positive multiples of 8");
    if (N == 0) return LOOKME_OK;
    if (!H || !W_he || !R_scales || !workspace || !out || !aligned16(workspace) || !aligned16(out))
        return fail(LOOKME_ERR_INVALID_ARG, "H, W_he, R_scales, an aligned workspace and out are required");
    const __nv_bfloat16* Rs[kRouterMaxScales];
    for (int m = 0; m < n_scales; ++m) {
        if (!R_scales[m] || !aligned16(R_scales[m]))
            return fail(LOOKME_ERR_INVALID_ARG, "R_scales[%d]: NULL or unaligned", m);
        Rs[m] = static_cast<const __nv_bfloat16*>(R_scales[m]);
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int sms = current_sms();
    // q = H W_he^T (fp32), then the per-token softmax over the scales.
    lookme_status st = gemm(nullptr, s, sms, H, W_he, N, d_embed, d_hidden, gemm_args(EPI_F32, workspace, d_embed, nullptr));
    if (st != LOOKME_OK) return st;
    LaunchCtx ctx{s, sms};
    cudaError_t e = launch_scale_router(ctx, workspace, Rs, n_scales, N, d_embed, static_cast<__nv_bfloat16*>(out), att_out);
    if (e != cudaSuccess) return fail(LOOKME_ERR_CUDA, "scale_router: %s", cudaGetErrorString(e));
    return LOOKME_OK;
}

// ------------------------------------------------- fusion f and propagation
}  // extern "C"

struct lookme_fusion {
    int32_t n_stages = 0;
    int64_t de = 0, dff = 0, dh = 0, max_rows = 0;
    int device = 0, num_sms = 0;
    void* mem = nullptr;                     // weights of every stage, then scratch
    std::vector<__nv_bfloat16*> w_ab, w_o, w_p;  // per stage
    std::vector<uint8_t> loaded;
    __nv_bfloat16* u = nullptr;              // [max_rows][d_ff]
    __nv_bfloat16* r[2] = {nullptr, nullptr};  // [max_rows][d_e] each
    uint32_t* status = nullptr;
};

extern "C" {

lookme_status lookme_fusion_create(int32_t n_stages, int64_t d_embed, int64_t d_ff, int64_t d_hidden, int32_t device,
                                   int64_t max_rows, lookme_fusion** out) {
    if (!out) return fail(LOOKME_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    if (n_stages < 1 || n_stages > LOOKME_MAX_LAYERS)
        return fail(LOOKME_ERR_INVALID_ARG, "n_stages %d outside [1, %d]", n_stages, LOOKME_MAX_LAYERS);
    if (d_embed < 8 || d_embed % 8 || d_hidden < 8 || d_hidden % 8 || d_ff < 32 || d_ff % 32 || max_rows < 1)
        return fail(LOOKME_ERR_INVALID_ARG, "d_embed, d_hidden: multiples of 8; d_ff: a multiple of 32; max_rows >= 1");
    DeviceGuard guard(device);
    if (!guard.ok) return fail(LOOKME_ERR_INVALID_ARG, "device %d not available", device);
    lookme_fusion* f = new lookme_fusion();
    f->n_stages = n_stages;
    f->de = d_embed;
    f->dff = d_ff;
    f->dh = d_hidden;
    f->max_rows = max_rows;
    f->device = device;
    cudaDeviceGetAttribute(&f->num_sms, cudaDevAttrMultiProcessorCount, device);
    const size_t per_stage = align_up(2 * d_ff * d_embed * 2, 256) + align_up(d_hidden * d_ff * 2, 256) +
                             align_up(d_embed * d_embed * 2, 256);
    const size_t scratch = align_up(max_rows * d_ff * 2, 256) + 2 * align_up(max_rows * d_embed * 2, 256) + 256;
    const size_t total = per_stage * n_stages + scratch;
    cudaError_t e = configure_gemm_kernels();
    if (e != cudaSuccess || cudaMalloc(&f->mem, total) != cudaSuccess) {
        cudaGetLastError();
        delete f;
        return fail(LOOKME_ERR_OOM, "fusion of %zu bytes", total);
    }
    char* m = static_cast<char*>(f->mem);
    for (int k = 0; k < n_stages; ++k) {
        f->w_ab.push_back(reinterpret_cast<__nv_bfloat16*>(m));
        m += align_up(2 * d_ff * d_embed * 2, 256);
        f->w_o.push_back(reinterpret_cast<__nv_bfloat16*>(m));
        m += align_up(d_hidden * d_ff * 2, 256);
        f->w_p.push_back(reinterpret_cast<__nv_bfloat16*>(m));
        m += align_up(d_embed * d_embed * 2, 256);
    }
    f->u = reinterpret_cast<__nv_bfloat16*>(m);
    m += align_up(max_rows * d_ff * 2, 256);
    f->r[0] = reinterpret_cast<__nv_bfloat16*>(m);
    m += align_up(max_rows * d_embed * 2, 256);
    f->r[1] = reinterpret_cast<__nv_bfloat16*>(m);
    m += align_up(max_rows * d_embed * 2, 256);
    f->status = reinterpret_cast<uint32_t*>(m);
    f->loaded.assign(n_stages, 0);
    if (cudaMemset(f->status, 0, 256) != cudaSuccess) {
        cudaFree(f->mem);
        delete f;
        return fail(LOOKME_ERR_CUDA, "fusion initialisation");
    }
    *out = f;
    return LOOKME_OK;
}

lookme_status lookme_fusion_load(lookme_fusion* f, int32_t stage, const void* W_a, const void* W_b, const void* W_o,
                                 const void* W_p, lookme_stream stream) {
    if (!f) return fail(LOOKME_ERR_INVALID_ARG, "fusion is NULL");
    if (stage < 0 || stage >= f->n_stages) return fail(LOOKME_ERR_INVALID_ARG, "stage %d outside [0, %d)", stage, f->n_stages);
    if (!W_a || !W_b || !W_o || (stage > 0 && !W_p))
        return fail(LOOKME_ERR_INVALID_ARG, "W_a, W_b, W_o (and W_p for stages after the first) are required");
    DeviceGuard guard(f->device);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int64_t de = f->de, dff = f->dff;
    // The gate and up projections interleaved per 32 features: rows 64 g .. 64 g + 31 of
    // the stacked operand are W_a's rows 32 g .., rows 64 g + 32 .. + 63 W_b's.
    const size_t blk = 32 * de * 2;
    char* ab = reinterpret_cast<char*>(f->w_ab[stage]);
    cudaError_t e = cudaMemcpy2DAsync(ab, 2 * blk, W_a, blk, blk, dff / 32, cudaMemcpyDefault, s);
    if (e == cudaSuccess) e = cudaMemcpy2DAsync(ab + blk, 2 * blk, W_b, blk, blk, dff / 32, cudaMemcpyDefault, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(f->w_o[stage], W_o, f->dh * dff * 2, cudaMemcpyDefault, s);
    if (e == cudaSuccess && stage > 0) e = cudaMemcpyAsync(f->w_p[stage], W_p, de * de * 2, cudaMemcpyDefault, s);
    if (e != cudaSuccess) return fail(LOOKME_ERR_CUDA, "fusion weights: %s", cudaGetErrorString(e));
    f->loaded[stage] = 1;
    return LOOKME_OK;
}

lookme_status lookme_fusion_apply(lookme_fusion* f, const void* R, const int32_t* rows, int64_t n_rows,
                                  void* const* hidden, lookme_stream stream) {
    if (!f) return fail(LOOKME_ERR_INVALID_ARG, "fusion is NULL");
    for (int k = 0; k < f->n_stages; ++k)
        if (!f->loaded[k]) return fail(LOOKME_ERR_STATE, "stage %d has no weights", k);
    if (n_rows < 0 || n_rows > f->max_rows)
        return fail(LOOKME_ERR_INVALID_ARG, "n_rows %lld outside [0, %lld]", (long long)n_rows, (long long)f->max_rows);
    if (n_rows == 0) return LOOKME_OK;
    if (!R || !rows || !hidden || !aligned16(R)) return fail(LOOKME_ERR_INVALID_ARG, "R (aligned), rows and hidden");
    for (int k = 0; k < f->n_stages; ++k)
        if (!hidden[k] || !aligned16(hidden[k])) return fail(LOOKME_ERR_INVALID_ARG, "hidden[%d]: NULL or unaligned", k);
    DeviceGuard guard(f->device);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const void* Rk = R;
    lookme_status st;
    for (int k = 0; k < f->n_stages; ++k) {
        if (k > 0) {
            // R^(k) = R^(k-1) W_p + R^(k-1) (Sec. "Inter-Layer Sparse Activation").
            __nv_bfloat16* dst = f->r[k & 1];
            GemmArgs g = gemm_args(EPI_RESID, dst, f->de, f->status);
            g.resid = Rk;
            g.ld_resid = f->de;
            if ((st = gemm(nullptr, s, f->num_sms, Rk, f->w_p[k], n_rows, f->de, f->de, g)) != LOOKME_OK) return st;
            Rk = dst;
        }
        // f(R) = (silu(R W_a^T) * (R W_b^T)) W_o^T, added to the gated rows of layer k.
        if ((st = gemm(nullptr, s, f->num_sms, Rk, f->w_ab[k], n_rows, 2 * f->dff, f->de,
                       gemm_args(EPI_SWIGLU, f->u, f->dff, f->status))) != LOOKME_OK)
            return st;
        GemmArgs g = gemm_args(EPI_SCATTER_ADD, hidden[k], f->dh, f->status);
        g.rowidx = rows;
        if ((st = gemm(nullptr, s, f->num_sms, f->u, f->w_o[k], n_rows, f->dh, f->dff, g)) != LOOKME_OK) return st;
    }
    return LOOKME_OK;
}

lookme_status lookme_fusion_status(lookme_fusion* f, uint32_t* status, lookme_stream stream) {
    if (!f || !status) return fail(LOOKME_ERR_INVALID_ARG, "NULL argument");
    DeviceGuard guard(f->device);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaMemcpyAsync(status, f->status, sizeof(uint32_t), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return fail(LOOKME_ERR_CUDA, "read fusion status: %s", cudaGetErrorString(e));
    return LOOKME_OK;
}

lookme_status lookme_fusion_destroy(lookme_fusion* f) {
    if (!f) return LOOKME_OK;
    DeviceGuard guard(f->device);
    cudaDeviceSynchronize();
    if (f->mem) cudaFree(f->mem);
    delete f;
    return LOOKME_OK;
}

}  // extern "C"
