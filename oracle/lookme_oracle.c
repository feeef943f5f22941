/*
 * LookME CPU oracle.  TEST INFRASTRUCTURE ONLY.
 *
 * This file restates, with plain loops in double precision, what the LookME
 * hierarchical two-level lookup and sparse injection compute (Sec. "Image
 * Embedding Hierarchical Two-Level Lookup" and Sec. "Sparse Injection" of
 * arXiv 2607.16305).  Only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg may load it.  The product path (the CUDA library) shares no
 * code with it and never calls it.
 *
 * Conventions
 *   - Every input array is float and holds the exact input values (a bf16
 *     value is exactly representable in float); every product and sum is
 *     formed in double.
 *   - Row-major layouts: queries q[N][d_k], centroids c[S][d_k],
 *     keys K[S][P][d_k] and values V[S][P][d_v], hidden h[L][N][d_v].
 *   - Scene blocks may be passed sparsely: key_blocks/value_blocks hold
 *     n_blocks blocks of P rows, and block_of_scene[s] gives the block index
 *     of scene s (or -1 if that scene's block was not provided).  For a full
 *     table block_of_scene[s] == s.
 *
 * Readings where the paper leaves a choice open (listed in the design notes):
 *   - Level-2 selection and weighting use z = q.k / sqrt(d_k) against the
 *     scene's primitive keys; the softmax runs over the selected top-k only.
 *   - Ties: level-1 argmax keeps the lowest scene index; level-2 top-k orders
 *     by larger z then lower primitive index; token selection orders by larger
 *     priority then lower token index.
 *   - A zero-norm query or centroid has cosine 0 against everything.
 *   - Token selection keeps r = floor(len * keep_ratio) tokens per segment.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* Level-1 scene-centred embedding: e_img[s] = (1/N_p) sum_i E_img[s, i, :]
 * (Sec. "Level-1: scene retrieval", first equation). */
void lkm_centroids(int64_t S, int64_t P, int64_t dk, const float* keys, double* cent)
{
    for (int64_t s = 0; s < S; ++s) {
        for (int64_t d = 0; d < dk; ++d) {
            double acc = 0.0;
            for (int64_t p = 0; p < P; ++p)
                acc += (double)keys[(s * P + p) * dk + d];
            cent[s * dk + d] = acc / (double)P;
        }
    }
}

/* Euclidean norm of a float row, in double. */
static double row_norm(const float* x, int64_t n)
{
    double acc = 0.0;
    for (int64_t i = 0; i < n; ++i)
        acc += (double)x[i] * (double)x[i];
    return sqrt(acc);
}

/* ||q_t||_2 of every query: the default gate priority of the token
 * selection (Sec. "Intra-Layer Sparse Activation", priority read as the
 * query norm).  The same value lkm_route reports. */
void lkm_query_norms(int64_t N, int64_t dk, const float* q, double* qnorm)
{
#pragma omp parallel for schedule(static)
    for (int64_t t = 0; t < N; ++t)
        qnorm[t] = row_norm(q + t * dk, dk);
}

/* Level-1 routing: scene_t = argmax_s ( cos(q_t, e_img[s]) + b_s )
 * (Sec. "Level-1: scene retrieval", second equation).
 * Outputs per token: the scene, its score, the gap between the best and the
 * second-best score (+inf when S == 1), and ||q_t||_2. */
void lkm_route(int64_t N, int64_t S, int64_t dk,
               const float* q, const float* cent, const float* bias,
               int32_t* scene, double* best_score, double* gap1, double* qnorm)
{
    double* cnorm = (double*)malloc((size_t)S * sizeof(double));
    for (int64_t s = 0; s < S; ++s)
        cnorm[s] = row_norm(cent + s * dk, dk);

#pragma omp parallel for schedule(dynamic, 8)
    for (int64_t t = 0; t < N; ++t) {
        const float* qt = q + t * dk;
        double nt = row_norm(qt, dk);
        double best = -INFINITY, second = -INFINITY;
        int32_t arg = 0;
        for (int64_t s = 0; s < S; ++s) {
            double dot = 0.0;
            for (int64_t d = 0; d < dk; ++d)
                dot += (double)qt[d] * (double)cent[s * dk + d];
            double cosv = (nt > 0.0 && cnorm[s] > 0.0) ? dot / (nt * cnorm[s]) : 0.0;
            double score = cosv + (bias ? (double)bias[s] : 0.0);
            if (score > best) {          /* strict: equal scores keep the lower s */
                second = best;
                best = score;
                arg = (int32_t)s;
            } else if (score > second) {
                second = score;
            }
        }
        scene[t] = arg;
        best_score[t] = best;
        gap1[t] = (S > 1) ? best - second : INFINITY;
        qnorm[t] = nt;
    }
    free(cnorm);
}

typedef struct {
    double z;
    int32_t p;
} scored_prim;

/* Order: larger z first, then lower primitive index. */
static int by_z_desc_then_p(const void* a, const void* b)
{
    const scored_prim* x = (const scored_prim*)a;
    const scored_prim* y = (const scored_prim*)b;
    if (x->z > y->z) return -1;
    if (x->z < y->z) return 1;
    return (x->p < y->p) ? -1 : (x->p > y->p);
}

/* Level-2 within the routed scene j = scene_t: z_p = q_t . K[j,p] / sqrt(d_k)
 * for every primitive p; I_t = the top_k primitives by z; weights
 * w = softmax over the selected z only (Sec. "Level-2: scene-primitive
 * retrieval", both equations, with the key-similarity reading).
 * Outputs per token t (row-major [N][top_k]): prim, weight, logit (the z of
 * each selected primitive, descending), gap_k[t] = z_(k) - z_(k+1)
 * (+inf when top_k == P) and gap_adj[t] = the smallest gap between adjacent
 * selected logits (+inf when top_k == 1). */
void lkm_primitives(int64_t N, int64_t P, int64_t dk, int32_t top_k,
                    const float* q, const int32_t* scene,
                    const float* key_blocks, const int64_t* block_of_scene,
                    int32_t* prim, double* weight, double* logit,
                    double* gap_k, double* gap_adj)
{
    const double inv_sqrt_dk = 1.0 / sqrt((double)dk);
#pragma omp parallel
    {
        scored_prim* zs = (scored_prim*)malloc((size_t)P * sizeof(scored_prim));
#pragma omp for schedule(dynamic, 8)
        for (int64_t t = 0; t < N; ++t) {
            const float* qt = q + t * dk;
            const float* Kj = key_blocks + block_of_scene[scene[t]] * P * dk;
            for (int64_t p = 0; p < P; ++p) {
                double dot = 0.0;
                for (int64_t d = 0; d < dk; ++d)
                    dot += (double)qt[d] * (double)Kj[p * dk + d];
                zs[p].z = dot * inv_sqrt_dk;
                zs[p].p = (int32_t)p;
            }
            qsort(zs, (size_t)P, sizeof(scored_prim), by_z_desc_then_p);

            double zmax = zs[0].z, denom = 0.0;
            for (int32_t j = 0; j < top_k; ++j)
                denom += exp(zs[j].z - zmax);
            double min_adj = INFINITY;
            for (int32_t j = 0; j < top_k; ++j) {
                prim[t * top_k + j] = zs[j].p;
                logit[t * top_k + j] = zs[j].z;
                weight[t * top_k + j] = exp(zs[j].z - zmax) / denom;
                if (j + 1 < top_k && zs[j].z - zs[j + 1].z < min_adj)
                    min_adj = zs[j].z - zs[j + 1].z;
            }
            gap_k[t] = (top_k < P) ? zs[top_k - 1].z - zs[top_k].z : INFINITY;
            gap_adj[t] = min_adj;
        }
        free(zs);
    }
}

/* The same weighting as lkm_primitives for a primitive set that is given
 * rather than chosen: w_j = softmax_j(q_t . K[scene_t, prim_tj] / sqrt(d_k)).
 * Used to evaluate the injection for another implementation's choices. */
void lkm_weights_for(int64_t N, int64_t P, int64_t dk, int32_t top_k,
                     const float* q, const int32_t* scene, const int32_t* prim,
                     const float* key_blocks, const int64_t* block_of_scene,
                     double* weight)
{
    const double inv_sqrt_dk = 1.0 / sqrt((double)dk);
    for (int64_t t = 0; t < N; ++t) {
        const float* qt = q + t * dk;
        const float* Kj = key_blocks + block_of_scene[scene[t]] * P * dk;
        double z[64], zmax = -INFINITY, denom = 0.0;  /* top_k <= 64 */
        for (int32_t j = 0; j < top_k; ++j) {
            int64_t p = prim[t * top_k + j];
            double dot = 0.0;
            for (int64_t d = 0; d < dk; ++d)
                dot += (double)qt[d] * (double)Kj[p * dk + d];
            z[j] = dot * inv_sqrt_dk;
            if (z[j] > zmax) zmax = z[j];
        }
        for (int32_t j = 0; j < top_k; ++j)
            denom += exp(z[j] - zmax);
        for (int32_t j = 0; j < top_k; ++j)
            weight[t * top_k + j] = exp(z[j] - zmax) / denom;
    }
}

typedef struct {
    double pi;
    int64_t t;
} prio_tok;

/* Order: larger priority first, then lower token index. */
static int by_pi_desc_then_t(const void* a, const void* b)
{
    const prio_tok* x = (const prio_tok*)a;
    const prio_tok* y = (const prio_tok*)b;
    if (x->pi > y->pi) return -1;
    if (x->pi < y->pi) return 1;
    return (x->t < y->t) ? -1 : (x->t > y->t);
}

/* Intra-layer sparse activation as top-r selection (Sec. "Intra-Layer Sparse
 * Activation"): in each segment [seg_off[i], seg_off[i+1]) keep the
 * r = floor(len * keep_ratio) tokens of largest priority.  mask[t] = 1 for a
 * kept token.  For each segment, pi_r[i] is the r-th largest priority
 * (+inf if r == 0) and pi_r1[i] the (r+1)-th (-inf if r == len). */
void lkm_select(int64_t N, const double* priority, int32_t n_seg, const int64_t* seg_off,
                double keep_ratio, uint8_t* mask, double* pi_r, double* pi_r1)
{
    memset(mask, 0, (size_t)N);
    for (int32_t i = 0; i < n_seg; ++i) {
        int64_t b = seg_off[i], len = seg_off[i + 1] - seg_off[i];
        int64_t r = (int64_t)floor((double)len * keep_ratio);
        prio_tok* v = (prio_tok*)malloc((size_t)(len > 0 ? len : 1) * sizeof(prio_tok));
        for (int64_t j = 0; j < len; ++j) {
            v[j].pi = priority[b + j];
            v[j].t = b + j;
        }
        qsort(v, (size_t)len, sizeof(prio_tok), by_pi_desc_then_t);
        for (int64_t j = 0; j < r; ++j)
            mask[v[j].t] = 1;
        pi_r[i] = (r > 0) ? v[r - 1].pi : INFINITY;
        pi_r1[i] = (r < len) ? v[r].pi : -INFINITY;
        free(v);
    }
}

/* Sparse injection into every layer that shares the table (Sec. "Sparse
 * Injection", S(R) = g * f(R[g]) with f the identity, and Sec. "Inter-Layer
 * Sparse Activation" with the propagation W_p = 0):
 *   R_t = sum_j weight[t,j] * V[scene_t, prim[t,j], :]
 *   out[l,t,:] = h[l,t,:] + R_t   if mask[t],   h[l,t,:] otherwise. */
void lkm_inject(int64_t N, int64_t P, int64_t dv, int32_t top_k,
                const int32_t* scene, const int32_t* prim, const double* weight,
                const uint8_t* mask, const float* value_blocks, const int64_t* block_of_scene,
                int32_t n_layers, const float* hidden, double* out)
{
#pragma omp parallel
    {
        double* R = (double*)malloc((size_t)dv * sizeof(double));
#pragma omp for schedule(dynamic, 8)
        for (int64_t t = 0; t < N; ++t) {
            if (mask[t]) {
                for (int64_t d = 0; d < dv; ++d)
                    R[d] = 0.0;
                const float* Vj = value_blocks + block_of_scene[scene[t]] * P * dv;
                for (int32_t j = 0; j < top_k; ++j) {
                    const float* row = Vj + (int64_t)prim[t * top_k + j] * dv;
                    for (int64_t d = 0; d < dv; ++d)
                        R[d] += weight[t * top_k + j] * (double)row[d];
                }
            }
            for (int32_t l = 0; l < n_layers; ++l) {
                const float* h = hidden + ((int64_t)l * N + t) * dv;
                double* o = out + ((int64_t)l * N + t) * dv;
                for (int64_t d = 0; d < dv; ++d)
                    o[d] = (double)h[d] + (mask[t] ? R[d] : 0.0);
            }
        }
        free(R);
    }
}

/* Round-to-nearest-even of a double to bfloat16 (1 sign, 8 exponent and 7
 * stored mantissa bits), returned as the bf16 bit pattern. */
void lkm_round_bf16(int64_t n, const double* x, uint16_t* out)
{
    for (int64_t i = 0; i < n; ++i) {
        double v = x[i];
        float f;
        if (isnan(v)) {
            out[i] = 0x7FC0;
            continue;
        }
        if (v == 0.0 || isinf(v)) {
            f = (float)v;
        } else {
            int e;
            double m = frexp(fabs(v), &e);          /* |v| = m * 2^e, m in [0.5, 1) */
            double r;
            if (e - 1 >= -126) {
                r = ldexp(nearbyint(ldexp(m, 8)), e - 8);   /* keep 8 significant bits */
            } else {
                r = ldexp(nearbyint(ldexp(fabs(v), 133)), -133);  /* subnormal quantum 2^-133 */
            }
            if (r > 3.38953138925153547590470800371487866880e38)   /* above the largest finite bf16 */
                r = INFINITY;
            f = (float)(v < 0 ? -r : r);            /* exact: r has at most 8 significant bits */
        }
        uint32_t bits;
        memcpy(&bits, &f, sizeof(bits));
        out[i] = (uint16_t)(bits >> 16);
    }
}
