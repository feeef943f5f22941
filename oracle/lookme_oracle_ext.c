/*
 * LookME CPU oracle, second part: the paper-exact pieces around the lookup.
 * TEST INFRASTRUCTURE ONLY (same rules as lookme_oracle.c: only the tests,
 * the smoke check and the benchmark's CPU leg may load it; the CUDA library
 * shares no code with it).
 *
 *   - level 2 with the scene-shared MLP ranker and the cos + tanh weighting
 *     (Sec. "Level-2: scene-primitive retrieval", both equations);
 *   - the SKA gate at inference (Sec. "Intra-Layer Sparse Activation", first
 *     equation);
 *   - the text pathway's ID lookup (Sec. "Text", and the PLE equation of
 *     Sec. "Method");
 *   - the dense ends: the projection into the embedding space (Sec.
 *     "Level-1", W_{v->e}), the SwiGLU-style fusion f (Sec. "Intra-Layer
 *     Sparse Activation", second equation) and the bottleneck propagation
 *     R W_p + R (Sec. "Inter-Layer Sparse Activation");
 *   - the token-wise softmax router over the multi-scale results (Sec.
 *     "Multi-scale image retrieval").
 *
 * Conventions: float inputs hold exact values; every product and sum is in
 * double.  Weight matrices are row-major in the orientation each function
 * states.  Readings where the paper is silent (listed in the design notes):
 *   - the ranker MLP is Linear(2 d_e -> d_m), SiLU, Linear(d_m -> N_p), with
 *     biases; its hidden activations are rounded to bf16 when round_hidden is
 *     set (the tensor-core path's operand precision);
 *   - the ranker's top-T orders by larger r then lower primitive index; the
 *     weights are softmax_p(cos(v_e, K[j,p]) + tanh(r_j[p])) over the T
 *     selected, with K the table's keys; a zero-norm vector has cosine 0;
 *   - the hard gate is g = 1 exactly when sigmoid(Delta . W_g) > 0.5, i.e.
 *     Delta . W_g > 0 (no Gumbel noise at inference);
 *   - SwiGLU: f(x) = (silu(x W_a^T) * (x W_b^T)) W_o^T, the product rounded
 *     to bf16 when round_mid is set.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

static double silu(double x) { return x / (1.0 + exp(-x)); }

/* Round-to-nearest-even of a double to the nearest bf16 value (returned as a
 * double).  Values past the largest finite bf16 become infinity. */
static double to_bf16(double v)
{
    if (isnan(v) || isinf(v) || v == 0.0) return v;
    int e;
    double m = frexp(fabs(v), &e); /* |v| = m 2^e, m in [0.5, 1) */
    double r;
    if (e - 1 >= -126)
        r = ldexp(nearbyint(ldexp(m, 8)), e - 8);
    else
        r = ldexp(nearbyint(ldexp(fabs(v), 133)), -133);
    if (r > 3.38953138925153547590470800371487866880e38) r = INFINITY;
    return v < 0 ? -r : r;
}

/* y[n][dout] = x[n][din] W^T + b, W row-major [dout][din] (b may be NULL). */
void lkx_linear(int64_t n, int64_t din, int64_t dout, const float* x, const float* W, const float* b, double* y)
{
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        for (int64_t o = 0; o < dout; ++o) {
            double acc = b ? (double)b[o] : 0.0;
            for (int64_t k = 0; k < din; ++k)
                acc += (double)x[i * din + k] * (double)W[o * din + k];
            y[i * dout + o] = acc;
        }
    }
}

/* Level-2 relevance of the scene-shared two-layer MLP (Sec. "Level-2", first
 * equation): r_t = W2 silu(W1 [v_t ; e_img[scene_t]] + b1) + b2.
 *   v [N][de], cent [S][de] (the scene-centred embeddings), W1 [dm][2 de]
 *   (columns 0..de-1 multiply v, de..2de-1 the centroid), b1 [dm],
 *   W2 [P][dm], b2 [P]  ->  r [N][P].
 * With round_hidden the hidden activations are rounded to bf16 first. */
void lkx_ranker_relevance(int64_t N, int64_t S, int64_t de, int64_t dm, int64_t P, const float* v,
                          const int32_t* scene, const float* cent, const float* W1, const float* b1,
                          const float* W2, const float* b2, int32_t round_hidden, double* r)
{
    (void)S;
#pragma omp parallel
    {
        double* h = (double*)malloc((size_t)dm * sizeof(double));
#pragma omp for schedule(dynamic, 4)
        for (int64_t t = 0; t < N; ++t) {
            const float* vt = v + t * de;
            const float* ct = cent + (int64_t)scene[t] * de;
            for (int64_t m = 0; m < dm; ++m) {
                const float* w = W1 + m * 2 * de;
                double acc = (double)b1[m];
                for (int64_t k = 0; k < de; ++k) acc += (double)w[k] * (double)vt[k];
                for (int64_t k = 0; k < de; ++k) acc += (double)w[de + k] * (double)ct[k];
                h[m] = silu(acc);
                if (round_hidden) h[m] = to_bf16(h[m]);
            }
            for (int64_t p = 0; p < P; ++p) {
                double acc = (double)b2[p];
                for (int64_t m = 0; m < dm; ++m) acc += (double)W2[p * dm + m] * h[m];
                r[t * P + p] = acc;
            }
        }
        free(h);
    }
}

typedef struct {
    double r;
    int32_t p;
} ranked;

/* Order: larger relevance first, then lower primitive index. */
static int by_r_desc_then_p(const void* a, const void* b)
{
    const ranked* x = (const ranked*)a;
    const ranked* y = (const ranked*)b;
    if (x->r > y->r) return -1;
    if (x->r < y->r) return 1;
    return (x->p < y->p) ? -1 : (x->p > y->p);
}

/* Level-2 selection and weighting of the paper (Sec. "Level-2", both
 * equations): I = the T primitives of largest r_t (scene j = scene_t), and
 *   w_p = softmax_{p in I}( cos(v_t, K[j,p]) + tanh(r_t[p]) ).
 * Outputs [N][T] in order of descending r: prim, weight; gap_T[t] =
 * r_(T) - r_(T+1) (+inf when T == P); gap_adj[t] = the smallest gap between
 * adjacent selected r (+inf when T == 1). */
void lkx_ranked_level2(int64_t N, int64_t P, int64_t de, int32_t T, const float* v, const int32_t* scene,
                       const float* key_blocks, const int64_t* block_of_scene, const double* r, int32_t* prim,
                       double* weight, double* gap_T, double* gap_adj)
{
#pragma omp parallel
    {
        ranked* rs = (ranked*)malloc((size_t)P * sizeof(ranked));
#pragma omp for schedule(dynamic, 8)
        for (int64_t t = 0; t < N; ++t) {
            for (int64_t p = 0; p < P; ++p) {
                rs[p].r = r[t * P + p];
                rs[p].p = (int32_t)p;
            }
            qsort(rs, (size_t)P, sizeof(ranked), by_r_desc_then_p);
            const float* vt = v + t * de;
            const float* Kj = key_blocks + block_of_scene[scene[t]] * P * de;
            double nv = 0.0;
            for (int64_t k = 0; k < de; ++k) nv += (double)vt[k] * (double)vt[k];
            nv = sqrt(nv);
            double s[64], smax = -INFINITY, den = 0.0, min_adj = INFINITY; /* T <= 64 */
            for (int32_t j = 0; j < T; ++j) {
                const float* kr = Kj + (int64_t)rs[j].p * de;
                double dot = 0.0, nk = 0.0;
                for (int64_t k = 0; k < de; ++k) {
                    dot += (double)vt[k] * (double)kr[k];
                    nk += (double)kr[k] * (double)kr[k];
                }
                nk = sqrt(nk);
                const double cosv = (nv > 0.0 && nk > 0.0) ? dot / (nv * nk) : 0.0;
                s[j] = cosv + tanh(rs[j].r);
                if (s[j] > smax) smax = s[j];
                if (j + 1 < T && rs[j].r - rs[j + 1].r < min_adj) min_adj = rs[j].r - rs[j + 1].r;
            }
            for (int32_t j = 0; j < T; ++j) den += exp(s[j] - smax);
            for (int32_t j = 0; j < T; ++j) {
                prim[t * T + j] = rs[j].p;
                weight[t * T + j] = exp(s[j] - smax) / den;
            }
            gap_T[t] = (T < P) ? rs[T - 1].r - rs[T].r : INFINITY;
            gap_adj[t] = min_adj;
        }
        free(rs);
    }
}

/* The weighting above for a primitive set that is given (conditional oracle). */
void lkx_ranked_weights_for(int64_t N, int64_t P, int64_t de, int32_t T, const float* v, const int32_t* scene,
                            const int32_t* prim, const float* key_blocks, const int64_t* block_of_scene,
                            const double* r, double* weight)
{
    for (int64_t t = 0; t < N; ++t) {
        const float* vt = v + t * de;
        const float* Kj = key_blocks + block_of_scene[scene[t]] * P * de;
        double nv = 0.0;
        for (int64_t k = 0; k < de; ++k) nv += (double)vt[k] * (double)vt[k];
        nv = sqrt(nv);
        double s[64], smax = -INFINITY, den = 0.0;
        for (int32_t j = 0; j < T; ++j) {
            const int64_t p = prim[t * T + j];
            const float* kr = Kj + p * de;
            double dot = 0.0, nk = 0.0;
            for (int64_t k = 0; k < de; ++k) {
                dot += (double)vt[k] * (double)kr[k];
                nk += (double)kr[k] * (double)kr[k];
            }
            nk = sqrt(nk);
            s[j] = ((nv > 0.0 && nk > 0.0) ? dot / (nv * nk) : 0.0) + tanh(r[t * P + p]);
            if (s[j] > smax) smax = s[j];
        }
        for (int32_t j = 0; j < T; ++j) den += exp(s[j] - smax);
        for (int32_t j = 0; j < T; ++j) weight[t * T + j] = exp(s[j] - smax) / den;
    }
}

/* SKA gate at inference (Sec. "Intra-Layer Sparse Activation"):
 * logit_t = Delta_t . W_g, g_t = 1 exactly when sigmoid(logit_t) > 0.5. */
void lkx_ska_gate(int64_t N, int64_t dh, const float* delta, const float* wg, uint8_t* gate, double* logit)
{
    for (int64_t t = 0; t < N; ++t) {
        double acc = 0.0;
        for (int64_t k = 0; k < dh; ++k) acc += (double)delta[t * dh + k] * (double)wg[k];
        logit[t] = acc;
        gate[t] = acc > 0.0 ? 1 : 0;
    }
}

/* Retrieved embedding of each token: R_t = sum_j w_tj V[scene_t, prim_tj, :]. */
void lkx_combine(int64_t N, int64_t P, int64_t dv, int32_t T, const int32_t* scene, const int32_t* prim,
                 const double* weight, const float* value_blocks, const int64_t* block_of_scene, double* R)
{
    for (int64_t t = 0; t < N; ++t) {
        const float* Vj = value_blocks + block_of_scene[scene[t]] * P * dv;
        for (int64_t d = 0; d < dv; ++d) R[t * dv + d] = 0.0;
        for (int32_t j = 0; j < T; ++j) {
            const float* row = Vj + (int64_t)prim[t * T + j] * dv;
            for (int64_t d = 0; d < dv; ++d) R[t * dv + d] += weight[t * T + j] * (double)row[d];
        }
    }
}

/* Text pathway with sparse injection (Sec. "Text": R_text = E_text[u]; Sec.
 * "Intra-Layer Sparse Activation": S(R) = g * f(R[g]), f the identity here):
 *   out[l,t,:] = h[l,t,:] + E[ids[t], :]  when gate[t] and 0 <= ids[t] < V,
 *   out[l,t,:] = h[l,t,:]                 otherwise (non-text positions carry
 *                                         an id outside the vocabulary). */
void lkx_text_inject(int64_t N, int64_t V, int64_t d, const float* E, const int32_t* ids, const uint8_t* gate,
                     int32_t n_layers, const float* hidden, double* out)
{
    for (int32_t l = 0; l < n_layers; ++l) {
        for (int64_t t = 0; t < N; ++t) {
            const int32_t u = ids[t];
            const int on = (!gate || gate[t]) && u >= 0 && u < V;
            for (int64_t k = 0; k < d; ++k) {
                const int64_t i = ((int64_t)l * N + t) * d + k;
                out[i] = (double)hidden[i] + (on ? (double)E[(int64_t)u * d + k] : 0.0);
            }
        }
    }
}

/* SwiGLU-style fusion f from the embedding width de to the hidden width dh
 * (Sec. "Intra-Layer Sparse Activation", second equation):
 *   u = silu(x W_a^T) * (x W_b^T)   (W_a, W_b [dff][de]; u rounded to bf16
 *                                    when round_mid is set)
 *   y = u W_o^T                      (W_o [dh][dff]). */
void lkx_swiglu(int64_t n, int64_t de, int64_t dff, int64_t dh, const float* x, const float* Wa, const float* Wb,
                const float* Wo, int32_t round_mid, double* y)
{
#pragma omp parallel
    {
        double* u = (double*)malloc((size_t)dff * sizeof(double));
#pragma omp for schedule(dynamic, 4)
        for (int64_t i = 0; i < n; ++i) {
            const float* xi = x + i * de;
            for (int64_t f = 0; f < dff; ++f) {
                double a = 0.0, b = 0.0;
                for (int64_t k = 0; k < de; ++k) {
                    a += (double)Wa[f * de + k] * (double)xi[k];
                    b += (double)Wb[f * de + k] * (double)xi[k];
                }
                u[f] = silu(a) * b;
                if (round_mid) u[f] = to_bf16(u[f]);
            }
            for (int64_t o = 0; o < dh; ++o) {
                double acc = 0.0;
                for (int64_t f = 0; f < dff; ++f) acc += (double)Wo[o * dff + f] * u[f];
                y[i * dh + o] = acc;
            }
        }
        free(u);
    }
}

/* Bottleneck propagation to the next non-LookME layer (Sec. "Inter-Layer
 * Sparse Activation", second equation): out = R W_p + R, with R [n][de] and
 * W_p [de][de] in the paper's orientation (row vector times matrix). */
void lkx_propagate(int64_t n, int64_t de, const float* R, const float* Wp, double* out)
{
    for (int64_t i = 0; i < n; ++i) {
        for (int64_t o = 0; o < de; ++o) {
            double acc = (double)R[i * de + o];
            for (int64_t k = 0; k < de; ++k) acc += (double)R[i * de + k] * (double)Wp[k * de + o];
            out[i * de + o] = acc;
        }
    }
}

/* Token-wise softmax router over M scales (Sec. "Multi-scale image
 * retrieval"): q_t = H_t W_he (H [N][dh], W_he [dh][de] in the paper's
 * orientation), a_tm = softmax_m(q_t . R^m_t / sqrt(de)), out_t =
 * sum_m a_tm R^m_t, with the scales' results Rs [M][N][de].  att [N][M]
 * receives the router weights. */
void lkx_scale_router(int64_t N, int64_t dh, int64_t de, int32_t M, const float* H, const float* Whe,
                      const float* Rs, double* out, double* att)
{
    const double inv = 1.0 / sqrt((double)de);
#pragma omp parallel
    {
        double* q = (double*)malloc((size_t)de * sizeof(double));
        double s[64];
#pragma omp for schedule(dynamic, 8)
        for (int64_t t = 0; t < N; ++t) {
            for (int64_t o = 0; o < de; ++o) {
                double acc = 0.0;
                for (int64_t k = 0; k < dh; ++k) acc += (double)H[t * dh + k] * (double)Whe[k * de + o];
                q[o] = acc;
            }
            double smax = -INFINITY, den = 0.0;
            for (int32_t m = 0; m < M; ++m) {
                const float* Rm = Rs + ((int64_t)m * N + t) * de;
                double dot = 0.0;
                for (int64_t o = 0; o < de; ++o) dot += q[o] * (double)Rm[o];
                s[m] = dot * inv;
                if (s[m] > smax) smax = s[m];
            }
            for (int32_t m = 0; m < M; ++m) den += exp(s[m] - smax);
            for (int64_t o = 0; o < de; ++o) out[t * de + o] = 0.0;
            for (int32_t m = 0; m < M; ++m) {
                const double a = exp(s[m] - smax) / den;
                att[t * M + m] = a;
                const float* Rm = Rs + ((int64_t)m * N + t) * de;
                for (int64_t o = 0; o < de; ++o) out[t * de + o] += a * (double)Rm[o];
            }
        }
        free(q);
    }
}
