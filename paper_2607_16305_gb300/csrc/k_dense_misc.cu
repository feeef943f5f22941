// Latency-bound kernels around the dense GEMMs:
//  - argmax-key decode for the paper-exact level 2 (which needs no bucketing);
//  - the paper's level-2 selection and weighting from the ranker's relevance
//    (Sec. "Level-2: scene-primitive retrieval": top-T of r, weights
//    softmax(cos(v_e, e_{j,p}) + tanh r_j[p]));
//  - the SKA gate at inference (Sec. "Intra-Layer Sparse Activation":
//    g = sigmoid(Delta W_g) > 0.5, i.e. Delta W_g > 0);
//  - injection on a given gate, the text pathway's ID lookup (Sec. "Text"),
//    the retrieved embeddings of listed tokens (input of the fusion f);
//  - the token-wise softmax router of the multi-scale retrieval (Sec.
//    "Multi-scale image retrieval").
#include <cfloat>
#include <climits>

#include "common.cuh"

namespace lookme {

// --------------------------------------------------------------- decode
__global__ void __launch_bounds__(256) k_decode_reset(unsigned long long* best, int64_t N, int64_t S,
                                                       int32_t* __restrict__ scene_out) {
    pdl_trigger();
    pdl_wait();
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (t < N) {
        scene_out[t] = unpack_scene(best[t], S);  // an unscored key decodes to 0 (the status word is set)
        best[t] = 0ull;
    }
}

cudaError_t launch_decode_reset(const LaunchCtx& c, unsigned long long* best, int64_t N, int64_t S,
                                int32_t* scene_out) {
    if (N == 0) return cudaSuccess;
    return launch_pdl(k_decode_reset, dim3((unsigned)((N + 255) / 256)), dim3(256), 0, c.stream, best, N, S, scene_out);
}

// ---------------------------------------------------------- ranked select
namespace kr {
constexpr int kWarps = 8;
// Address of 16-byte chunk kc of key row p of scene s.  Tiled: per scene, for
// each N-tile of two 128-row tiles (the last may hold one), for each 64-wide
// k-block, the N-tile's sub-blocks of 128 rows x 128 bytes, chunk c of row r
// at position c ^ (r & 7).
__device__ __forceinline__ const uint4* key_chunk(const KeyView& kv, int64_t s, int p, int kc) {
    if (!kv.tiled) return reinterpret_cast<const uint4*>(kv.keys + s * kv.block_bytes + ((int64_t)p * kv.dk + kc * 8) * 2);
    const int tile = p >> 7, r = p & 127, nt = tile >> 1;
    const int ns = (2 * nt + 1 < kv.ntile) ? 2 : 1;
    const int kb = kc >> 3;
    const int sb = nt * 2 * kv.nkb + kb * ns + (tile - 2 * nt);
    const int pos = (kc & 7) ^ (r & 7);
    return reinterpret_cast<const uint4*>(kv.keys + s * kv.block_bytes + (int64_t)sb * 16384 + r * 128 + pos * 16);
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    return v;
}
}  // namespace kr

__global__ void __launch_bounds__(kr::kWarps * 32) k_ranked_select(const float* __restrict__ r, int64_t ld_r, int64_t N, int T,
                                                                    const __nv_bfloat16* __restrict__ q, KeyView kv,
                                                                    const int32_t* __restrict__ scene,
                                                                    int32_t* __restrict__ prim_out,
                                                                    float* __restrict__ weight_out) {
    pdl_trigger();
    pdl_wait();
    const int lane = threadIdx.x & 31;
    const int64_t t = (int64_t)blockIdx.x * kr::kWarps + (threadIdx.x >> 5);
    if (t >= N) return;
    const int P = kv.P;
    const float* rt = r + t * ld_r;
    // Top-T by r, larger first, lower primitive on ties: T rounds of a warp
    // argmax over the entries after the previous winner in that order.  A
    // lane's entries (p = lane + 32 i) are read once, up to 64 of them into
    // registers (P <= 2,048); larger P re-reads the row from L1.
    constexpr int kReg = 8;
    float rl[kReg];
#pragma unroll
    for (int i = 0; i < kReg; ++i) {
        const int p = lane + 32 * i;
        rl[i] = p < P ? rt[p] : -INFINITY;
    }
    int sel[LOOKME_MAX_TOP_K];
    float rv[LOOKME_MAX_TOP_K];
    float last_v = INFINITY;
    int last_p = -1;
    for (int j = 0; j < T; ++j) {
        float bv = -INFINITY;
        int bp = INT_MAX;
#pragma unroll
        for (int i = 0; i < kReg; ++i) {
            const int p = lane + 32 * i;
            const float v = rl[i];
            const bool after = v < last_v || (v == last_v && p > last_p);
            if (p < P && after && (v > bv || (v == bv && p < bp))) {
                bv = v;
                bp = p;
            }
        }
        for (int p = lane + 32 * kReg; p < P; p += 32) {
            const float v = rt[p];
            const bool after = v < last_v || (v == last_v && p > last_p);
            if (after && (v > bv || (v == bv && p < bp))) {
                bv = v;
                bp = p;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float ov = __shfl_xor_sync(0xFFFFFFFFu, bv, o);
            const int op = __shfl_xor_sync(0xFFFFFFFFu, bp, o);
            if (ov > bv || (ov == bv && op < bp)) {
                bv = ov;
                bp = op;
            }
        }
        sel[j] = bp;
        rv[j] = bv;
        last_v = bv;
        last_p = bp;
    }
    // cos(q_t, K[scene_t, p]) for the selected p: lanes split d_k in 16-byte chunks.
    const int64_t s = scene[t];
    const int nch = kv.dk / 8;
    float qv[8 * 4];  // up to 4 chunks per lane (d_k <= 1,024)
    float nq = 0.f;
    for (int u = 0; u * 32 + lane < nch && u < 4; ++u) {
        Vec16<__nv_bfloat16>::unpack(reinterpret_cast<const uint4*>(q + t * kv.dk)[u * 32 + lane], qv + 8 * u);
#pragma unroll
        for (int e = 0; e < 8; ++e) nq = fmaf(qv[8 * u + e], qv[8 * u + e], nq);
    }
    nq = sqrtf(kr::warp_sum(nq));
    float sc[LOOKME_MAX_TOP_K];
    float smax = -INFINITY;
    // Eight key rows at a time: every lane issues its chunk loads of the
    // eight rows before any arithmetic, then the warp reduces each row.
    for (int j0 = 0; j0 < T; j0 += 8) {
        float dot[8], nk[8];
#pragma unroll
        for (int jj = 0; jj < 8; ++jj) dot[jj] = nk[jj] = 0.f;
        for (int u = 0; u * 32 + lane < nch && u < 4; ++u) {
            uint4 kc[8];
#pragma unroll
            for (int jj = 0; jj < 8; ++jj)
                if (j0 + jj < T) kc[jj] = *kr::key_chunk(kv, s, sel[j0 + jj], u * 32 + lane);
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) {
                if (j0 + jj < T) {
                    float kf[8];
                    Vec16<__nv_bfloat16>::unpack(kc[jj], kf);
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        dot[jj] = fmaf(qv[8 * u + e], kf[e], dot[jj]);
                        nk[jj] = fmaf(kf[e], kf[e], nk[jj]);
                    }
                }
            }
        }
#pragma unroll
        for (int jj = 0; jj < 8; ++jj) {
            if (j0 + jj < T) {
                const float d = kr::warp_sum(dot[jj]);
                const float n = sqrtf(kr::warp_sum(nk[jj]));
                const float cosv = (nq > 0.f && n > 0.f) ? d / (nq * n) : 0.f;
                sc[j0 + jj] = cosv + tanhf(rv[j0 + jj]);
                smax = fmaxf(smax, sc[j0 + jj]);
            }
        }
    }
    float den = 0.f;
    for (int j = 0; j < T; ++j) {
        sc[j] = __expf(sc[j] - smax);
        den += sc[j];
    }
    const float inv = 1.f / den;
    for (int j = lane; j < T; j += 32) {
        prim_out[t * T + j] = sel[j];
        weight_out[t * T + j] = sc[j] * inv;
    }
}

cudaError_t launch_ranked_select(const LaunchCtx& c, const float* r, int64_t ld_r, int64_t N, int T, const __nv_bfloat16* q,
                                 const KeyView& kv, const int32_t* scene, int32_t* prim_out, float* weight_out) {
    if (N == 0) return cudaSuccess;
    if (T < 1 || T > LOOKME_MAX_TOP_K || kv.dk % 8 || kv.dk > 1024) return cudaErrorInvalidValue;
    return launch_pdl(k_ranked_select, dim3((unsigned)((N + kr::kWarps - 1) / kr::kWarps)), dim3(kr::kWarps * 32), 0,
                      c.stream, r, ld_r, N, T, q, kv, scene, prim_out, weight_out);
}

// --------------------------------------------------------------- SKA gate
template <typename T>
__global__ void __launch_bounds__(256) k_ska_gate(const T* __restrict__ delta, const T* __restrict__ wg, int64_t N,
                                                  int64_t dh, uint8_t* __restrict__ gate, float* __restrict__ logit) {
    pdl_trigger();
    pdl_wait();
    const int lane = threadIdx.x & 31;
    const int64_t t = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
    if (t >= N) return;
    constexpr int V = Vec16<T>::N;
    const int64_t nch = dh / V;
    float acc = 0.f;
    for (int64_t cidx = lane; cidx < nch; cidx += 32) {
        float a[V], b[V];
        Vec16<T>::unpack(reinterpret_cast<const uint4*>(delta + t * dh)[cidx], a);
        Vec16<T>::unpack(reinterpret_cast<const uint4*>(wg)[cidx], b);
#pragma unroll
        for (int e = 0; e < V; ++e) acc = fmaf(a[e], b[e], acc);
    }
    acc = kr::warp_sum(acc);
    if (lane == 0) {
        gate[t] = acc > 0.f ? 1 : 0;
        if (logit) logit[t] = acc;
    }
}

cudaError_t launch_ska_gate(const LaunchCtx& c, int dtype, const void* delta, const void* wg, int64_t N, int64_t dh,
                            uint8_t* gate, float* logit_out) {
    if (N == 0) return cudaSuccess;
    const dim3 grid((unsigned)((N + 7) / 8));
    if (dtype == LOOKME_BF16)
        return launch_pdl(k_ska_gate<__nv_bfloat16>, grid, dim3(256), 0, c.stream, (const __nv_bfloat16*)delta,
                          (const __nv_bfloat16*)wg, N, dh, gate, logit_out);
    return launch_pdl(k_ska_gate<float>, grid, dim3(256), 0, c.stream, (const float*)delta, (const float*)wg, N, dh, gate,
                      logit_out);
}

// ------------------------------------------------ injection on a given gate
// One CTA per token; gated-off tokens return at once.  Thread i handles the
// 16-byte chunks i, i + blockDim, ... of the row: the weighted sum of the
// token's value rows in fp32, then one rounding per layer.
struct GatedParams {
    const void* values;
    int64_t P;
    int dv, top_k, n_layers;
    const int32_t* scene;
    const int32_t* prim;
    const float* weight;
    const uint8_t* gate;
    const int32_t* rows;  // combine: token of each output row
    int64_t N;            // combine: tokens of the lookup (rows outside give zeros)
    void* out;            // combine: [n][dv] bf16
    void* hidden[LOOKME_MAX_LAYERS];
};

template <typename T, bool kCombine>
__global__ void __launch_bounds__(256) k_gated_rows(const __grid_constant__ GatedParams p) {
    pdl_trigger();
    pdl_wait();
    const int64_t i = blockIdx.x;
    const int64_t t = kCombine ? (int64_t)p.rows[i] : i;
    if (!kCombine && !p.gate[t]) return;
    const bool valid = !kCombine || (t >= 0 && t < p.N);
    constexpr int V = Vec16<T>::N;
    const int nch = p.dv / V;
    const int64_t s = valid ? p.scene[t] : 0;
    const T* vals = reinterpret_cast<const T*>(p.values);
    for (int cidx = threadIdx.x; cidx < nch; cidx += blockDim.x) {
        float acc[V];
#pragma unroll
        for (int e = 0; e < V; ++e) acc[e] = 0.f;
        const int kk = valid ? p.top_k : 0;
        for (int j0 = 0; j0 < kk; j0 += 8) {
            // Eight rows' chunks in flight before any is used.
            uint4 c8[8];
            float w8[8];
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) {
                if (j0 + jj < kk) {
                    const int64_t row = s * p.P + p.prim[t * p.top_k + j0 + jj];
                    w8[jj] = p.weight[t * p.top_k + j0 + jj];
                    c8[jj] = reinterpret_cast<const uint4*>(vals + row * p.dv)[cidx];
                }
            }
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) {
                if (j0 + jj < kk) {
                    float f[V];
                    Vec16<T>::unpack(c8[jj], f);
#pragma unroll
                    for (int e = 0; e < V; ++e) acc[e] = fmaf(w8[jj], f[e], acc[e]);
                }
            }
        }
        if (kCombine) {
            uint4 o;
            __nv_bfloat162* ob = reinterpret_cast<__nv_bfloat162*>(&o);
            static_assert(!kCombine || V == 8, "combine writes bf16 rows from bf16 tables");
#pragma unroll
            for (int e = 0; e < 4; ++e) ob[e] = __floats2bfloat162_rn(acc[2 * e], acc[2 * e + 1]);
            reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(p.out) + i * p.dv)[cidx] = o;
        } else {
            for (int l = 0; l < p.n_layers; ++l) {
                uint4* h = reinterpret_cast<uint4*>(reinterpret_cast<T*>(p.hidden[l]) + t * p.dv) + cidx;
                float f[V];
                Vec16<T>::unpack(*h, f);
#pragma unroll
                for (int e = 0; e < V; ++e) f[e] += acc[e];
                *h = Vec16<T>::pack(f);
            }
        }
    }
}

static GatedParams gated_params(const InjectArgs& a) {
    GatedParams p;
    memset(&p, 0, sizeof(p));
    p.values = a.values;
    p.P = a.P;
    p.dv = a.dv;
    p.top_k = a.top_k;
    p.n_layers = a.n_layers;
    p.scene = a.scene;
    p.prim = a.prim;
    p.weight = a.weight;
    for (int l = 0; l < a.n_layers; ++l) p.hidden[l] = a.hidden[l];
    return p;
}

static int row_threads(int dv, int vec) {
    int threads = (dv / vec + 31) / 32 * 32;
    return threads > 256 ? 256 : (threads < 32 ? 32 : threads);
}

cudaError_t launch_inject_gated(const LaunchCtx& c, const InjectArgs& a, const uint8_t* gate) {
    if (a.N == 0) return cudaSuccess;
    GatedParams p = gated_params(a);
    p.gate = gate;
    if (a.dtype == LOOKME_BF16)
        return launch_pdl(k_gated_rows<__nv_bfloat16, false>, dim3((unsigned)a.N), dim3(row_threads(a.dv, 8)), 0,
                          c.stream, p);
    return launch_pdl(k_gated_rows<float, false>, dim3((unsigned)a.N), dim3(row_threads(a.dv, 4)), 0, c.stream, p);
}

cudaError_t launch_combine(const LaunchCtx& c, const InjectArgs& a, const int32_t* rows, int64_t n,
                           __nv_bfloat16* R_out) {
    if (n == 0) return cudaSuccess;
    if (a.dtype != LOOKME_BF16) return cudaErrorInvalidValue;
    GatedParams p = gated_params(a);
    p.rows = rows;
    p.N = a.N;
    p.out = R_out;
    return launch_pdl(k_gated_rows<__nv_bfloat16, true>, dim3((unsigned)n), dim3(row_threads(a.dv, 8)), 0, c.stream,
                      p);
}

// ------------------------------------------------------------ text pathway
template <typename T>
__global__ void __launch_bounds__(256) k_text_inject(const T* __restrict__ E, int64_t V, int64_t d,
                                                     const int32_t* __restrict__ ids, const uint8_t* __restrict__ gate,
                                                     const __grid_constant__ GatedParams p) {
    pdl_trigger();
    pdl_wait();
    const int64_t t = blockIdx.x;
    const int32_t u = ids[t];
    if ((gate && !gate[t]) || u < 0 || u >= V) return;
    constexpr int VN = Vec16<T>::N;
    const int64_t nch = d / VN;
    for (int64_t cidx = threadIdx.x; cidx < nch; cidx += blockDim.x) {
        float e[VN];
        Vec16<T>::unpack(reinterpret_cast<const uint4*>(E + (int64_t)u * d)[cidx], e);
        for (int l = 0; l < p.n_layers; ++l) {
            uint4* h = reinterpret_cast<uint4*>(reinterpret_cast<T*>(p.hidden[l]) + t * d) + cidx;
            float f[VN];
            Vec16<T>::unpack(*h, f);
#pragma unroll
            for (int k = 0; k < VN; ++k) f[k] += e[k];
            *h = Vec16<T>::pack(f);
        }
    }
}

cudaError_t launch_text_inject(const LaunchCtx& c, int dtype, const void* E, int64_t V, int64_t d,
                               const int32_t* ids, const uint8_t* gate, int64_t N, void* const* hidden, int n_layers) {
    if (N == 0) return cudaSuccess;
    GatedParams p;
    memset(&p, 0, sizeof(p));
    p.n_layers = n_layers;
    for (int l = 0; l < n_layers; ++l) p.hidden[l] = hidden[l];
    if (dtype == LOOKME_BF16)
        return launch_pdl(k_text_inject<__nv_bfloat16>, dim3((unsigned)N), dim3(row_threads((int)d, 8)), 0, c.stream,
                          (const __nv_bfloat16*)E, V, d, ids, gate, p);
    return launch_pdl(k_text_inject<float>, dim3((unsigned)N), dim3(row_threads((int)d, 4)), 0, c.stream,
                      (const float*)E, V, d, ids, gate, p);
}

// ------------------------------------------------------ multi-scale router
struct RouterParams {
    const __nv_bfloat16* R[kRouterMaxScales];
};

__global__ void __launch_bounds__(256) k_scale_router(const float* __restrict__ q, const __grid_constant__ RouterParams rp,
                                                      int M, int64_t N, int64_t de, __nv_bfloat16* __restrict__ out,
                                                      float* __restrict__ att) {
    pdl_trigger();
    pdl_wait();
    const int lane = threadIdx.x & 31;
    const int64_t t = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
    if (t >= N) return;
    const float inv = rsqrtf((float)de);
    const int64_t nch = de / 8;
    float s[kRouterMaxScales];
    float smax = -INFINITY;
    for (int m = 0; m < M; ++m) {
        float acc = 0.f;
        for (int64_t cidx = lane; cidx < nch; cidx += 32) {
            float f[8];
            Vec16<__nv_bfloat16>::unpack(reinterpret_cast<const uint4*>(rp.R[m] + t * de)[cidx], f);
            const float4 q0 = reinterpret_cast<const float4*>(q + t * de)[2 * cidx];
            const float4 q1 = reinterpret_cast<const float4*>(q + t * de)[2 * cidx + 1];
            acc += q0.x * f[0] + q0.y * f[1] + q0.z * f[2] + q0.w * f[3] + q1.x * f[4] + q1.y * f[5] + q1.z * f[6] +
                   q1.w * f[7];
        }
        s[m] = kr::warp_sum(acc) * inv;
        smax = fmaxf(smax, s[m]);
    }
    float den = 0.f;
    for (int m = 0; m < M; ++m) {
        s[m] = __expf(s[m] - smax);
        den += s[m];
    }
    const float rden = 1.f / den;
    for (int m = 0; m < M; ++m) s[m] *= rden;
    if (att && lane < M) {
        for (int m = 0; m < M; ++m)
            if (m == lane) att[t * M + m] = s[m];
    }
    for (int64_t cidx = lane; cidx < nch; cidx += 32) {
        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        for (int m = 0; m < M; ++m) {
            float f[8];
            Vec16<__nv_bfloat16>::unpack(reinterpret_cast<const uint4*>(rp.R[m] + t * de)[cidx], f);
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[e] = fmaf(s[m], f[e], acc[e]);
        }
        reinterpret_cast<uint4*>(out + t * de)[cidx] = Vec16<__nv_bfloat16>::pack(acc);
    }
}

cudaError_t launch_scale_router(const LaunchCtx& c, const float* q, const __nv_bfloat16* const* Rs, int M, int64_t N,
                                int64_t de, __nv_bfloat16* out, float* att_out) {
    if (N == 0) return cudaSuccess;
    if (M < 1 || M > kRouterMaxScales || de % 8) return cudaErrorInvalidValue;
    RouterParams rp;
    memset(&rp, 0, sizeof(rp));
    for (int m = 0; m < M; ++m) rp.R[m] = Rs[m];
    return launch_pdl(k_scale_router, dim3((unsigned)((N + 7) / 8)), dim3(256), 0, c.stream, q, rp, M, N, de, out,
                      att_out);
}

}  // namespace lookme
