/*
 * lookme.h - C ABI of the LookME lookup + sparse-injection library (GB300, sm_103a).
 *
 * LookME (arXiv 2607.16305) enhances a vision-language model's hidden states
 * with rows retrieved from a large external table.  The image and cross-modal
 * pathways look up continuous embeddings in two levels (Sec. "Image Embedding
 * Hierarchical Two-Level Lookup"):
 *   level 1  scene_t = argmax_s ( cos(q_t, e_img[s]) + b_s )
 *   level 2  z_tp = q_t . K[scene_t, p] / sqrt(d_k) for every primitive p of
 *            that scene, I_t = top-k of z_t, w_t = softmax(z_t[I_t]),
 *            R_t = sum_j w_tj * V[scene_t, I_tj, :]
 * and inject R only into the hidden rows of the highest-priority tokens
 * (Sec. "Sparse Injection"), reusing one lookup across the neighbouring
 * layers that share a table (Sec. "Inter-Layer Sparse Activation").
 *
 * Conventions for every entry point
 *   - All pointers are plain addresses.  "device" means CUDA device memory of
 *     the table's device (or host memory the device can address); "host"
 *     means ordinary CPU memory.  Layouts are row-major and dense.
 *   - The element type of queries, centroids, keys, values and hidden states
 *     is the table's dtype (bf16 = IEEE bfloat16 bit patterns, or fp32).
 *     Indices are int32, weights, norms and priorities fp32.
 *   - All work is asynchronous on the given stream (a cudaStream_t; NULL is
 *     the legacy default stream).  No entry point synchronises the stream
 *     unless its comment says so.  Results are valid once the stream has
 *     reached the point of the call.
 *   - The caller owns every buffer it passes; the library never frees or
 *     keeps caller memory past the call (except the table storage it owns).
 *   - Errors are return codes; nothing throws or aborts across the ABI.
 *     lookme_last_error() gives a thread-local message for the last failure.
 *     An asynchronous CUDA error seen by a later call is returned as
 *     LOOKME_ERR_CUDA and makes the table unusable (sticky).
 *   - One table may be used from one stream at a time.
 */
#ifndef LOOKME_H
#define LOOKME_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    LOOKME_OK = 0,
    LOOKME_ERR_INVALID_ARG = 1,  /* an argument failed validation; nothing was launched */
    LOOKME_ERR_CUDA = 2,         /* a CUDA call failed (sticky on the table) */
    LOOKME_ERR_OOM = 3,          /* a device or pinned-host allocation failed */
    LOOKME_ERR_TIMEOUT = 4,      /* a bounded device-side wait gave up (see lookme_device_status) */
    LOOKME_ERR_STATE = 5,        /* call out of order (e.g. lookup before every scene is loaded) */
    LOOKME_ERR_UNSUPPORTED = 6   /* valid request this build does not handle */
} lookme_status;

typedef enum { LOOKME_BF16 = 0, LOOKME_FP32 = 1 } lookme_dtype;

/* Where the keys and values of a table live.  Centroids always live in HBM.
 *   DEVICE       keys and values in HBM.
 *   HOST_STAGED  keys and values in pinned host memory (the paper's
 *                partitioned storage with on-demand loading, Sec. "Level-2:
 *                scene-primitive retrieval", last sentence): each lookup
 *                copies the key blocks of the routed scenes into an HBM slot
 *                cache on a side stream, and the injection reads the selected
 *                value rows straight from host memory. */
typedef enum { LOOKME_RES_DEVICE = 0, LOOKME_RES_HOST_STAGED = 1 } lookme_residency;

typedef void* lookme_stream; /* cudaStream_t */

/* Shape of a two-level table E_img in R^{N_s x N_p x d_e} (Sec. "Two-level
 * embedding table"), split into keys (scored) and values (injected).  Setting
 * d_key == d_value and passing the same array for both recovers the paper's
 * single table. */
typedef struct {
    int64_t n_scenes;     /* N_s >= 1 */
    int64_t n_prims;      /* N_p >= 1 (primitives per scene) */
    int64_t d_key;        /* key / query width d_k >= 1 (bf16: multiple of 8; fp32: multiple of 4) */
    int64_t d_value;      /* value / hidden width >= 1 (bf16: multiple of 8; fp32: multiple of 4) */
    int32_t dtype;        /* lookme_dtype */
    int32_t residency;    /* lookme_residency */
    int32_t device;       /* CUDA device ordinal */
    int32_t reserved0;    /* must be 0 */
    int64_t max_tokens;   /* scratch is sized for this many tokens per call; 0 = grow on demand */
    int64_t stage_slots;  /* HOST_STAGED: scenes the HBM slot cache holds (0 = n_scenes); a call
                           * may route to at most this many distinct scenes, so it must be at
                           * least min(n_tokens, n_scenes) of every lookup */
} lookme_table_desc;

typedef struct lookme_table lookme_table; /* opaque, owned by the library */

/* Limits of this build. */
#define LOOKME_MAX_TOP_K 64        /* top_k <= min(n_prims, 64) */
#define LOOKME_MAX_LAYERS 64       /* layers sharing one table per inject call */
#define LOOKME_MAX_SEGMENTS 1024   /* token-selection segments per inject call */
#define LOOKME_MAX_SCENES 49152    /* n_scenes (bucketing keeps one counter per scene on chip) */
#define LOOKME_MAX_PRIMS 2048      /* n_prims (level-2 keeps one logit per primitive on chip) */
#define LOOKME_MAX_DKEY 1024       /* d_key */

/* Create a table on desc->device.  Allocates the table storage (HBM, or
 * pinned host for HOST_STAGED), the centroids and, if desc->max_tokens > 0,
 * the per-call scratch.  *out receives the handle; on failure *out is NULL.
 * Errors: INVALID_ARG (bad shape or limits), OOM, CUDA. */
lookme_status lookme_table_create(const lookme_table_desc* desc, lookme_table** out);

/* Free everything the table owns.  Synchronises the device first.  NULL is a no-op. */
lookme_status lookme_table_destroy(lookme_table* table);

/* Copy scenes [scene_begin, scene_begin + n) into the table (Sec. "Two-level
 * embedding table").
 *   centroids  [n][d_key] scene-centred embeddings e_img, or NULL: then each
 *              centroid is the mean of its scene's keys (Sec. "Level-1: scene
 *              retrieval", first equation), accumulated in fp32 and stored
 *              in the table dtype.
 *   keys       [n][n_prims][d_key]     (required)
 *   values     [n][n_prims][d_value]   (required)
 *   bias       [n] fp32 routing bias b (Sec. "Level-1", second equation) or
 *              NULL for 0.  A table with any nonzero bias routes by
 *              cos + b; without bias by cos alone.
 *   src_on_device  1 if the sources are device memory, 0 if host memory.
 * The sources may be reused once the stream reaches the end of the call.
 * Errors: INVALID_ARG (range, NULL keys/values), CUDA. */
lookme_status lookme_load_scenes(lookme_table* table, int64_t scene_begin, int64_t n,
                                 const void* centroids, const void* keys, const void* values,
                                 const float* bias, int src_on_device, lookme_stream stream);

/* Two-level lookup for n_tokens queries (Sec. "Image Embedding Hierarchical
 * Two-Level Lookup"; the cross-modal pathway is the same call with the
 * decoder output as queries):
 *   queries     device [n_tokens][d_key]
 *   scene_out   device [n_tokens] int32: level-1 scene (ties: lowest index)
 *   prim_out    device [n_tokens][top_k] int32: primitives of that scene by
 *               descending z (ties: lower index)
 *   weight_out  device [n_tokens][top_k] fp32: softmax over the selected z
 *   qnorm_out   device [n_tokens] fp32 ||q_t||_2, or NULL (the table keeps
 *               its own copy for lookme_inject's default priority)
 * Every token is looked up; selection happens in lookme_inject.
 * HOST_STAGED tables (Sec. "Level-2: scene-primitive retrieval", last
 * sentence: scene blocks are loaded on demand): after bucketing, the routed
 * scenes are looked up in the table's HBM slot cache, which persists across
 * calls; the key blocks of the misses are copied from pinned host memory over
 * the host link on the table's own staging stream (forked from and joined to
 * the caller's stream with events), evicting scenes that this call does not
 * route to (clock order); level 2 then reads the slots, and the injection
 * reads the selected value rows from host memory directly.
 * Errors: INVALID_ARG, STATE (a scene not loaded yet, or scratch would have to
 * grow while the stream is being captured), UNSUPPORTED (HOST_STAGED with
 * fewer staging slots than min(n_tokens, n_scenes)), OOM, CUDA. */
lookme_status lookme_lookup(lookme_table* table, const void* queries, int64_t n_tokens, int32_t top_k,
                            int32_t* scene_out, int32_t* prim_out, float* weight_out, float* qnorm_out,
                            lookme_stream stream);

/* Sparse injection (Sec. "Sparse Injection", S(R) = g * f(R[g]) with f the
 * identity, and Sec. "Inter-Layer Sparse Activation" with the same gate and
 * R reused by every layer that shares the table):
 *   scene, prim, weight   device outputs of lookme_lookup for these tokens
 *   priority   device [n_tokens] fp32 gate signal, or NULL for the query
 *              norms of this table's most recent lookup (which must have had
 *              n_tokens tokens)
 *   seg_offsets  HOST [n_seg + 1] int64, 0 = off[0] <= ... <= off[n_seg] =
 *              n_tokens, or NULL for one segment.  Segment i keeps its
 *              r_i = floor(len_i * keep_ratio) tokens of largest priority
 *              (ties: lower token index); keep_ratio in [0, 1].
 *   hidden     HOST array of n_layers device pointers, each [n_tokens][d_value]
 *              in the table dtype, updated in place: every kept row gets
 *              + sum_j w_tj V[scene_t, prim_tj, :] (accumulated in fp32,
 *              rounded once); every other row is left untouched.
 *   mask_out   device [n_tokens] uint8 (1 = kept) or NULL
 *   sel_out    device [sum r_i] int32 kept token ids (ascending within each
 *              segment, segments in order) or NULL
 * Errors: INVALID_ARG, STATE, OOM, CUDA. */
lookme_status lookme_inject(lookme_table* table, const int32_t* scene, const int32_t* prim,
                            const float* weight, int64_t n_tokens, int32_t top_k,
                            const float* priority, const int64_t* seg_offsets, int32_t n_seg,
                            double keep_ratio, void* const* hidden, int32_t n_layers,
                            uint8_t* mask_out, int32_t* sel_out, lookme_stream stream);

/* lookme_lookup followed by lookme_inject in one call, on one stream, with
 * the same results (Sec. "Hierarchical Lookup" then Sec. "Sparse Injection").
 * The arguments mean what they mean there; priority NULL = the query norms of
 * these queries; mask_out (device [n_tokens] uint8, or NULL) receives the
 * gate.  With at most 64 segments of at most 8,192 tokens, the gate is
 * decided during the lookup (beside the bucketing) and the injection visits
 * only the kept tokens; on HBM-resident bf16 tables with top_k <= 16 the
 * level-2 kernel hands each kept token's value rows and weights to the
 * injection directly.  Errors: those of lookme_lookup and lookme_inject
 * (the injection arguments are checked before anything runs). */
lookme_status lookme_lookup_inject(lookme_table* table, const void* queries, int64_t n_tokens, int32_t top_k,
                                   const float* priority, const int64_t* seg_offsets, int32_t n_seg,
                                   double keep_ratio, void* const* hidden, int32_t n_layers, int32_t* scene_out,
                                   int32_t* prim_out, float* weight_out, uint8_t* mask_out, lookme_stream stream);

/* Size the per-call scratch for up to max_tokens tokens now, so that later
 * calls (for example under CUDA graph capture) never allocate.  Synchronous. */
lookme_status lookme_reserve(lookme_table* table, int64_t max_tokens);

/* Empty the HOST_STAGED slot cache, so that the next lookup copies every
 * routed scene's key block again (for cold-cache measurements, or after the
 * host copy of the table was changed other than through lookme_load_scenes,
 * which empties the cache itself).  Asynchronous on the stream; no effect on
 * HBM-resident tables.  Errors: INVALID_ARG, CUDA. */
lookme_status lookme_stage_invalidate(lookme_table* table, lookme_stream stream);

/* Grid sizes of later calls, for running several calls at once (Sec.
 * "Hierarchical Lookup" over independent batches on different streams).
 * route_sms: the SM count that the level-1 routing and the bucketing + gate
 * size their grids for (0: the whole device).  level2_ctas: the CTAs of the
 * tcgen05 level-2 kernel (0: one per SM; values above the SM count act as 0).
 * One call at a time, the defaults spread every step over the whole device.
 * With several calls in flight, each CTA of one call's routing or gate holds an
 * SM that another call's level 2 would stream on, and each level-2 CTA pays a
 * ramp (first copy) and a tail (last item's top-k) per call; fewer, fuller
 * CTAs then cost less SM time for the same work, while the calls in flight
 * together keep HBM busy.  Results do not depend on either value.  The fused
 * single-launch form ignores both.  lookme_lookup_ranked takes route_sms for
 * its routing grid and its ranker GEMM tiles.  Not thread-safe with calls in
 * flight on the host.  Errors: INVALID_ARG (a negative value). */
lookme_status lookme_set_grids(lookme_table* table, int32_t route_sms, int32_t level2_ctas);

/* Statistics of the table's most recent lookup, read back synchronously on
 * the given stream: routed scenes, level-2 work items, largest bucket. */
typedef struct {
    int64_t n_tokens;
    int32_t n_routed_scenes;  /* distinct scenes that received a token */
    int32_t n_work_items;     /* level-2 work items (scene, token chunk) */
    int64_t staged_bytes;     /* HOST_STAGED: key bytes copied host -> HBM (the slot cache's misses) */
    int32_t staged_hits;      /* HOST_STAGED: routed scenes found in the slot cache */
    int32_t reserved0;
} lookme_lookup_stats;
lookme_status lookme_last_lookup_stats(lookme_table* table, lookme_lookup_stats* out, lookme_stream stream);

/* Device status word of the table (bit 0: a bounded wait inside a kernel
 * gave up; the kernel then skipped its remaining work; bit 1: it was the
 * level-1 kernel, bit 2: a level-2 kernel; bit 4: more routed scenes than
 * HBM slots; bit 6: a kernel met an index outside its range, such as an
 * injection record naming no token, and skipped that access).  Synchronises
 * the stream.  reset != 0 clears it afterwards. */
lookme_status lookme_device_status(lookme_table* table, uint32_t* status, int reset, lookme_stream stream);

/* Number of CUDA kernels this table has launched since creation. */
uint64_t lookme_launch_count(const lookme_table* table);

/* Per-kernel tracing.  While enabled, every kernel the table launches is
 * bracketed by two CUDA events on its stream.  lookme_trace_read
 * synchronises those events and copies out up to max records (kernel id and
 * milliseconds), then clears the log.  lookme_kernel_name maps an id to a name. */
typedef struct {
    int32_t kernel;
    float ms;
} lookme_trace_record;
lookme_status lookme_trace_enable(lookme_table* table, int enable);
lookme_status lookme_trace_read(lookme_table* table, lookme_trace_record* out, int32_t max, int32_t* n_out);
const char* lookme_kernel_name(int32_t kernel);

/* Level-1 routing only (scene_out[t] for every query, exactly as
 * lookme_lookup's scene_out) without allocating anything.  The paper has no
 * counterpart: this entry point exists for callers that cannot allocate
 * device memory when they route, such as a serving loop whose device memory
 * belongs to another allocator or a path that must avoid the device-wide
 * synchronisation an allocation can cause.  Its per-token scratch lives in
 * fixed device arrays built into the library, sized for
 * LOOKME_ROUTE_STATIC_MAX_TOKENS tokens (768 KiB per device, held by every
 * GPU that loads the library until the process exits).
 *   queries    device [n_tokens][d_key], n_tokens <= LOOKME_ROUTE_STATIC_MAX_TOKENS
 *              (larger requests fail with INVALID_ARG before anything runs)
 *   scene_out  device [n_tokens] int32
 * The first call on a device looks up the arrays' device addresses
 * (cudaGetSymbolAddress) with that device current; make that first call
 * before any stream capture.  All calls share the one scratch and each call
 * re-initialises the part it uses, so calls that may overlap on the GPU (on
 * different streams, or from different tables on the same device) race and
 * must be serialised by the caller.
 * Errors: INVALID_ARG, STATE (a scene not loaded yet), CUDA.  A bounded
 * device-side wait that gave up is not a return code of this call (it
 * happens after the call returns): it sets the table's status word, read with
 * lookme_device_status, and the tokens it left unrouted get scene -1. */
#define LOOKME_ROUTE_STATIC_MAX_TOKENS 65536
lookme_status lookme_route_scenes_static(lookme_table* table, const void* queries, int64_t n_tokens,
                                         int32_t* scene_out, lookme_stream stream);

/* ------------------------------------------------------------------------
 * Paper-exact level 2 (Sec. "Level-2: scene-primitive retrieval").
 *
 * Install the scene-shared two-layer MLP ranker of a bf16 table:
 *   r_j = W2 silu(W1 [v_e ; e_img[j]] + b1) + b2     (first equation)
 *   W1  [d_hidden][2 d_key] bf16 (columns [0, d_key) multiply the query,
 *       [d_key, 2 d_key) the scene's centroid), b1 [d_hidden] fp32,
 *   W2  [n_prims][d_hidden] bf16, b2 [n_prims] fp32; host or device memory,
 *       copied (the sources may be reused once the stream reaches the call).
 * The activation is SiLU (the paper does not name it).  The per-scene term
 * W1[:, d_key:] e_img[j] + b1 is computed by the next lookme_lookup_ranked
 * and again after any lookme_load_scenes.  Synchronous when it replaces an
 * earlier ranker.  Errors: INVALID_ARG (d_hidden not a multiple of 8 in
 * [8, 4096], NULL weights), UNSUPPORTED (fp32 table), OOM, CUDA. */
lookme_status lookme_set_ranker(lookme_table* table, int64_t d_hidden, const void* W1, const float* b1,
                                const void* W2, const float* b2, lookme_stream stream);

/* Level 1 as lookme_lookup, then the paper's level 2: the ranker's relevance
 * r_t over the scene's n_prims primitives (two bf16 GEMMs on the tensor
 * cores, the hidden activations rounded to bf16), the top_t primitives of
 * largest r (ties: lower index; output in descending r), and the weights
 *   w = softmax over the selected of cos(q_t, K[scene_t, p]) + tanh(r_t[p])
 * (second equation; K is the table's keys, read only for the selected rows).
 *   queries [n_tokens][d_key] bf16, scene_out [n_tokens], prim_out and
 *   weight_out [n_tokens][top_t] (device).
 * The table keeps ||q_t|| for lookme_inject's default priority.
 * Errors: INVALID_ARG, STATE (no ranker, scenes not loaded, or scratch must
 * grow under stream capture), OOM, CUDA. */
lookme_status lookme_lookup_ranked(lookme_table* table, const void* queries, int64_t n_tokens, int32_t top_t,
                                   int32_t* scene_out, int32_t* prim_out, float* weight_out, lookme_stream stream);

/* SKA gate at inference (Sec. "Intra-Layer Sparse Activation", first
 * equation): g_t = 1 exactly when sigmoid(Delta_t . w_g) > 0.5, i.e.
 * Delta_t . w_g > 0 (the Gumbel-Sigmoid without noise).
 *   delta [n_tokens][d_hidden], w_g [d_hidden] (dtype: LOOKME_BF16 or
 *   LOOKME_FP32, d_hidden a multiple of 8 or 4), gate_out [n_tokens] u8,
 *   logit_out [n_tokens] fp32 or NULL; device memory, current device.
 * Errors: INVALID_ARG, CUDA. */
lookme_status lookme_ska_gate(const void* delta, const void* w_g, int64_t n_tokens, int64_t d_hidden, int32_t dtype,
                              uint8_t* gate_out, float* logit_out, lookme_stream stream);

/* Sparse injection on a given gate (Sec. "Intra-Layer Sparse Activation",
 * second equation, f the identity): for every t with gate[t] != 0,
 *   h_l[t] += sum_j weight[t][j] V[scene[t], prim[t][j]]   for each layer l,
 * accumulated in fp32 and rounded once; other rows are not touched.
 *   scene [n_tokens], prim/weight [n_tokens][top_k], gate [n_tokens] u8,
 *   hidden: host array of n_layers device pointers [n_tokens][d_value].
 * Errors: INVALID_ARG, CUDA. */
lookme_status lookme_inject_gated(lookme_table* table, const int32_t* scene, const int32_t* prim, const float* weight,
                                  int64_t n_tokens, int32_t top_k, const uint8_t* gate, void* const* hidden,
                                  int32_t n_layers, lookme_stream stream);

/* Retrieved embeddings of listed tokens, the input of the fusion f:
 *   R_out[i] = sum_j weight[t][j] V[scene[t], prim[t][j]],  t = rows[i]
 * in fp32, written as bf16 [n_rows][d_value] (bf16 tables); scene, prim and
 * weight are a lookup's outputs for n_tokens tokens, and a row id outside
 * [0, n_tokens) yields a row of zeros.
 * Errors: INVALID_ARG, UNSUPPORTED (fp32 table), CUDA. */
lookme_status lookme_combine(lookme_table* table, const int32_t* scene, const int32_t* prim, const float* weight,
                             int64_t n_tokens, int32_t top_k, const int32_t* rows, int64_t n_rows, void* R_out,
                             lookme_stream stream);

/* Text pathway (Sec. "Text", and the text-only PLE equation of Sec.
 * "Method"): R_text = E_text[u], injected on the gated text positions:
 *   h_l[t] += E[ids[t]] for every layer l, when (gate is NULL or gate[t])
 *   and 0 <= ids[t] < vocab; positions whose id is outside the vocabulary
 *   (image positions, say -1) are left untouched.
 *   E [vocab][d] and hidden [n_tokens][d] in dtype (bf16 or fp32), ids
 *   [n_tokens] int32, gate [n_tokens] u8 or NULL; device memory.
 * Errors: INVALID_ARG, CUDA. */
lookme_status lookme_text_inject(const void* E, int64_t vocab, int64_t d, int32_t dtype, const int32_t* ids,
                                 const uint8_t* gate, int64_t n_tokens, void* const* hidden, int32_t n_layers,
                                 lookme_stream stream);

/* Projection into the embedding space (Sec. "Level-1": v_e = v W_{v->e}):
 *   out[N][d_out] (bf16) = x[N][d_in] W^T + bias,
 * with W [d_out][d_in] bf16 (the transpose of the paper's d_v x d_e matrix:
 * a linear layer's weight) and bias [d_out] fp32 or NULL; tensor cores,
 * fp32 accumulation.  d_in and d_out multiples of 8.  Errors: INVALID_ARG, CUDA. */
lookme_status lookme_project(const void* x, const void* W, const float* bias, int64_t n_tokens, int64_t d_in,
                             int64_t d_out, void* out, lookme_stream stream);

/* Token-wise softmax router over the multi-scale results (Sec. "Multi-scale
 * image retrieval"):
 *   q_t = H_t W_he^T,  a_tm = softmax_m(q_t . R^m_t / sqrt(d_embed)),
 *   out_t = sum_m a_tm R^m_t.
 *   H [n_tokens][d_hidden] bf16; W_he [d_embed][d_hidden] bf16 (the
 *   transpose of the paper's W_{h->e}); R_scales: host array of n_scales
 *   (<= 16) device pointers [n_tokens][d_embed] bf16; workspace
 *   [n_tokens][d_embed] fp32 (caller-owned, receives q); out
 *   [n_tokens][d_embed] bf16; att_out [n_tokens][n_scales] fp32 or NULL.
 * Errors: INVALID_ARG, CUDA. */
lookme_status lookme_scale_router(const void* H, const void* W_he, const void* const* R_scales, int32_t n_scales,
                                  int64_t n_tokens, int64_t d_hidden, int64_t d_embed, float* workspace, void* out,
                                  float* att_out, lookme_stream stream);

/* Fusion f and inter-layer propagation (Sec. "Intra-Layer Sparse
 * Activation", second equation; Sec. "Inter-Layer Sparse Activation"): a
 * stack of n_stages layers sharing one retrieval.  Stage 0 is the LookME
 * layer, stage k >= 1 the k-th layer after it:
 *   R^(0) = R,  R^(k) = R^(k-1) W_p^k + R^(k-1),
 *   h_k[rows[i]] += f^k(R^(k)_i),  f^k(x) = (silu(x W_a^T) * (x W_b^T)) W_o^T,
 * on tensor cores with fp32 accumulation; R^(k) and the SwiGLU product are
 * rounded to bf16 between the GEMMs.  The object owns its weights and
 * scratch (rows up to max_rows).  bf16 only; d_embed and d_hidden multiples
 * of 8, d_ff a multiple of 32. */
typedef struct lookme_fusion lookme_fusion;
lookme_status lookme_fusion_create(int32_t n_stages, int64_t d_embed, int64_t d_ff, int64_t d_hidden, int32_t device,
                                   int64_t max_rows, lookme_fusion** out);
/* Weights of one stage, copied (host or device memory): W_a and W_b
 * [d_ff][d_embed], W_o [d_hidden][d_ff], W_p [d_embed][d_embed] given as a
 * linear layer's weight, i.e. the transpose of the paper's W_p (NULL for
 * stage 0).  Errors: INVALID_ARG, CUDA. */
lookme_status lookme_fusion_load(lookme_fusion* fusion, int32_t stage, const void* W_a, const void* W_b,
                                 const void* W_o, const void* W_p, lookme_stream stream);
/* R [n_rows][d_embed] bf16 (e.g. from lookme_combine), rows [n_rows] the
 * token of each row (distinct), hidden: host array of n_stages device
 * pointers [n_tokens][d_hidden] bf16, updated in place on the listed rows.
 * Errors: INVALID_ARG, STATE (a stage without weights), CUDA. */
lookme_status lookme_fusion_apply(lookme_fusion* fusion, const void* R, const int32_t* rows, int64_t n_rows,
                                  void* const* hidden, lookme_stream stream);
/* The fusion's device status word (bounded-wait timeouts), synchronously. */
lookme_status lookme_fusion_status(lookme_fusion* fusion, uint32_t* status, lookme_stream stream);
lookme_status lookme_fusion_destroy(lookme_fusion* fusion);

const char* lookme_status_string(lookme_status status);
const char* lookme_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* LOOKME_H */
