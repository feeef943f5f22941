// The whole lookup + sparse injection of one call in a single persistent
// launch (bf16 tables resident in HBM): level-1 routing (Sec. "Level-1: scene
// retrieval"), bucketing by scene, level-2 scoring with top-k and softmax over
// the selected (Sec. "Level-2: scene-primitive retrieval", key-similarity
// form), the gate as top-r by priority per segment (Sec. "Intra-Layer Sparse
// Activation") and the injection of R into every layer sharing the table
// (Sec. "Sparse Injection", "Inter-Layer Sparse Activation").
//
// One CTA per SM, all resident at once (cooperative launch).  Phases:
//  1 routing: (128-token tile, BN-scene tile) units, each CTA a contiguous run
//    of them; TMA token and centroid tiles, tcgen05.mma into TMEM, and an
//    epilogue that keeps the best (score, scene) per token and merges it with
//    one 64-bit atomicMax into this call's key array.  The CTA that takes
//    scene tile 0 of a token tile also stores the tokens' query norms (the
//    default gate priority).
//  2 one grid-wide barrier: every token's key is final.
//  3 bucketing, redundantly in every CTA: all N keys -> per-scene counts in
//    shared memory -> block scan -> work items (scene, <= 8 tokens) in scene
//    order.  The counts do not depend on the order they are taken in, so every
//    CTA derives the same list.  CTA b owns the scenes whose first item lies
//    in [I b / G, I (b + 1) / G) of the I items: it writes those scenes' work
//    entries, places their tokens and writes their tokens' scenes.  Then, still
//    before any key copy, it ranks its tokens for the gate (the priorities came
//    with the keys, one round trip) and builds the token tiles of its first
//    items: once an SM's copy ring is full, a small load issued by that SM
//    waits about as long as the ring takes to drain, so nothing small is read
//    while the keys stream.
//  4 level 2 over the owned items with the pipeline of the level-2 kernel
//    (bulk-copied key tiles, MMAs into two TMEM buffers, two epilogue groups
//    taking alternate items), without work taking.  A kept token's value rows
//    are sent into L2 right after its top-k and its record is queued in shared
//    memory; when the CTA's last item is scored its sixteen epilogue warps
//    inject every queued token at once, with no key copy left in flight.
// The argmax keys and the grid-barrier counter alternate between two buffers
// by the parity of an epoch word that the last CTA to exit advances; each
// call clears the buffers the next call uses, so no reset launch is needed.
// Every wait is bounded (1 s); a timeout drains the CTA's copies and MMAs,
// frees TMEM and sets the table's status word.
#include <cuda.h>

#include <algorithm>
#include <climits>

#include "score_tc.cuh"

namespace lookme {

namespace kst {
// Warps: 0 producer, 1 MMA issuer, 2..9 epilogue (two groups of four, which
// are also the routing epilogue), 10 token tiles.  Eleven warps leave each
// thread about 168 registers, so the epilogue (read-out, top-k, injection)
// runs without spilling: a spill reload behind a full copy ring costs
// microseconds.
constexpr int kGroupWarps = 4;            // epilogue warps per item group
constexpr int kEpiWarps = 2 * kGroupWarps;
constexpr int kTokWarp = 2 + kEpiWarps;
constexpr int kThreads = (kTokWarp + 1) * 32;
constexpr int kWarps = kThreads / 32;
constexpr int kRouteEpi = 8;              // routing epilogue: warps 2..9
constexpr int kRouteBM = 128;
constexpr int kItemCache = 32;            // owned items kept in shared memory (the rest in the work array)
constexpr int kTileCache = 16;            // token tiles built before the key stream (ring of tiles after)
constexpr int kKeptCap = 32;              // kept tokens queued for the end-of-CTA injection
constexpr int kRStagesMax = 4;
constexpr int kBarBytes = 1024;
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr uint64_t kTimeoutNs = 1000000000ull;
constexpr int kSmemLimit = k3tc::kSmemLimit;

// Control block in shared memory (after the barriers).
struct Ctl {
    WorkItem items[k3tc::kISlots];              // item metadata handed to MMA and epilogue
    int32_t toks[k3tc::kISlots * k3tc::kTok];   // and the items' token ids
    uint32_t tmem_slot;
    int abort;
    uint32_t epoch;
    int i0, i1;                                 // owned items [i0, i1)
    int maxb;
    int n_kept;                                 // kept tokens queued
    int2 warp_buf[33];
    WorkItem ic_w[kItemCache];                  // the first owned items,
    int32_t ic_tok[kItemCache * k3tc::kTok];    // their tokens
    uint32_t ic_keep[kItemCache];               // and which of them the gate keeps
    int gcnt[kItemCache * k3tc::kTok];          // gate: larger-or-earlier priorities per cached token
    int32_t kept_t[kKeptCap];                   // queued kept tokens: id, value rows, weights
    int32_t kept_row[kKeptCap][kRecMaxTopK];
    float kept_w[kKeptCap][kRecMaxTopK];
};

struct Geo {
    // level 2 (the geometry rules of the level-2 kernel)
    int nkb, ntile, nnt, spi, group, gshift, slot_bytes, n_stages, chunks, row_bytes, b_bytes, tmem_cols, zbytes;
    int off_b, off_z, off_bar, off_x, smem, ring_bytes;
    // routing
    int BN, rstages, units_per_cta, r_off_b, r_off_c;
    int tmem_alloc;
};

inline int pow2_at_least(int v) {
    int c = 32;
    while (c < v) c <<= 1;
    return c;
}

inline bool geometry(int64_t N, int64_t S, int64_t P, int dk, int num_sms, Geo& g) {
    using namespace k3tc;
    g.nkb = (dk + BK - 1) / BK;
    g.ntile = (int)((P + kSubRows - 1) / kSubRows);
    g.nnt = (g.ntile + 1) / 2;
    g.spi = g.ntile * g.nkb;
    g.row_bytes = dk * 2;
    g.b_bytes = g.nkb * kAtomBytes;
    const int nmax = (int)std::min<int64_t>(kNTile, (P + 15) / 16 * 16);
    g.tmem_cols = pow2_at_least(2 * nmax);
    g.zbytes = ((int)P * kZStride * 4 + 15) / 16 * 16;
    const int ctl = ((int)sizeof(Ctl) + 15) / 16 * 16;
    const int tiles = kTileCache * g.b_bytes;
    const int fixed = tiles + 2 * g.zbytes + kBarBytes + ctl + 1024 /*alignment*/;
    // 32 KiB copies (two 16 KiB sub-blocks: one N-tile k-block), four in
    // flight: enough bytes in flight to keep HBM busy, few enough that a
    // copy issued behind them is not held for long.
    g.gshift = g.spi >= 2 ? 1 : 0;
    g.group = 1 << g.gshift;
    g.slot_bytes = g.group * kSubBytes;
    g.chunks = (g.spi + g.group - 1) / g.group;
    g.n_stages = std::min(4, (kSmemLimit - fixed) / g.slot_bytes);
    g.ring_bytes = g.n_stages * g.slot_bytes;
    g.off_b = g.ring_bytes;
    g.off_z = g.off_b + tiles;
    g.off_bar = g.off_z + 2 * g.zbytes;
    g.off_x = g.off_bar + kBarBytes;
    g.smem = g.off_x + ctl + 1024;
    // Routing: the scene-tile width of the level-1 kernel's rule (narrow tiles
    // when there are few token tiles, so more CTAs share the work).  Its tiles
    // use the ring and the tile cache, both free until the bucketing.
    const int64_t m_tiles = (N + kRouteBM - 1) / kRouteBM;
    if (m_tiles * ((S + 255) / 256) >= num_sms) g.BN = 256;
    else if (m_tiles * ((S + 127) / 128) >= num_sms) g.BN = 128;
    else g.BN = 64;
    const int route_room = g.ring_bytes + tiles;
    g.r_off_b = g.nkb * kRouteBM * 128;
    g.rstages = kRStagesMax;
    while (g.rstages > 2 && g.r_off_b + g.rstages * g.BN * 128 + 4 * g.BN * 4 > route_room) --g.rstages;
    g.r_off_c = g.r_off_b + g.rstages * g.BN * 128;
    const int64_t units = m_tiles * ((S + g.BN - 1) / g.BN);
    g.units_per_cta = (int)((units + num_sms - 1) / num_sms);
    g.tmem_alloc = std::max(g.tmem_cols, pow2_at_least(2 * g.BN));
    // Bucketing: scene counts and token scenes in the tile cache, priorities in the logit area.
    return g.n_stages >= 2 && g.smem <= kSmemLimit && g.tmem_alloc <= 512 && (dk % 8) == 0 && dk <= 512 &&
           (g.ntile < 2 || g.group >= 2) && g.r_off_c + 4 * g.BN * 4 <= route_room &&
           (S * 4 + 15) / 16 * 16 + N * 4 <= tiles && N * 4 <= 2 * g.zbytes && N <= kStepMaxTokens &&
           g.n_stages <= kMaxStages;
}

// The kernel's arguments (StepArgs without the host-only parts).
struct Params {
    int64_t N, S, P;
    int dk, dv, top_k;
    float scale;
    const __nv_bfloat16* q;
    const uint8_t* keys_t;
    int64_t block_bytes;
    const uint8_t* values;
    const float* inv_cnorm;
    const float* bias;
    int32_t* scene_out;
    int32_t* prim_out;
    float* weight_out;
    float* qnorm;
    float* qnorm_out;
    int gate;
    int n_seg;
    const float* priority;
    uint8_t* mask_out;
    int64_t seg_off[kMaxGateSegments + 1];
    int64_t seg_r[kMaxGateSegments];
    int n_layers;
    void* hidden[LOOKME_MAX_LAYERS];
    StepState* state;
    WorkItem* work;
    int32_t* item_tok;
    int32_t* counters;
    uint32_t* status;
    int32_t* rec_row;
    float* rec_w;
    int32_t* ovf_tok;
};

__device__ __forceinline__ uint32_t ld_acquire_gpu(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Named barrier 1 over the routing epilogue warps, returning the OR of v.
__device__ __forceinline__ bool route_epi_sync_or(bool v) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.or.pred q, 1, %2, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)v), "n"(32 * kRouteEpi)
        : "memory");
    return r != 0;
}

// Named barrier 1 + grp over one epilogue group, returning the OR of v.
template <int ID>
__device__ __forceinline__ bool group_bar_or(bool v) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.or.pred q, %2, %3, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)v), "n"(ID), "n"(kGroupWarps * 32)
        : "memory");
    return r != 0;
}
__device__ __forceinline__ bool group_sync_or(int grp, bool v) { return grp == 0 ? group_bar_or<1>(v) : group_bar_or<2>(v); }

// Exclusive scan of two counters over the CTA's kThreads threads.
__device__ void block_scan2(int2 v, int2& excl, int2& total, int2* wb) {
    const int lane = threadIdx.x % 32, warp = threadIdx.x / 32;
    int2 inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int a = __shfl_up_sync(0xFFFFFFFFu, inc.x, o);
        const int b = __shfl_up_sync(0xFFFFFFFFu, inc.y, o);
        if (lane >= o) {
            inc.x += a;
            inc.y += b;
        }
    }
    if (lane == 31) wb[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        const int2 w = lane < kWarps ? wb[lane] : make_int2(0, 0);
        int2 wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int a = __shfl_up_sync(0xFFFFFFFFu, wi.x, o);
            const int b = __shfl_up_sync(0xFFFFFFFFu, wi.y, o);
            if (lane >= o) {
                wi.x += a;
                wi.y += b;
            }
        }
        if (lane < kWarps) wb[lane] = make_int2(wi.x - w.x, wi.y - w.y);
        if (lane == kWarps - 1) wb[32] = wi;
    }
    __syncthreads();
    const int2 wbv = wb[warp];
    excl = make_int2(wbv.x + inc.x - v.x, wbv.y + inc.y - v.y);
    total = wb[32];
}

// The gate segment holding token t.
__device__ __forceinline__ int segment_of(const Params& p, int64_t t) {
    int lo = 0, hi = p.n_seg;
    while (hi - lo > 1) {
        const int mid = (lo + hi) / 2;
        if (p.seg_off[mid] <= t) lo = mid;
        else hi = mid;
    }
    return lo;
}

// The gate (Sec. "Intra-Layer Sparse Activation", as top-r by priority):
// token t is kept iff its rank in its segment, larger priority first and the
// lower index on equal priorities,
//   rank_t = #{ j in segment : pi_j > pi_t, or pi_j == pi_t and j < t },
// is below r_seg = floor(len * keep_ratio).  One warp per token; `prio`
// holds the segment's priorities (shared memory, or global memory read
// through L2 since other CTAs of this launch may have written them).
template <bool kShared>
__device__ __forceinline__ bool gate_keep(const Params& p, const float* prio, int64_t t, int lane) {
    const int lo = segment_of(p, t);
    const int64_t b = p.seg_off[lo], len = p.seg_off[lo + 1] - b, r = p.seg_r[lo];
    if (r <= 0) return false;
    if (r >= len) return true;
    const float* pb = prio + b;
    const uint32_t kt = orderable(kShared ? pb[t - b] : __ldcg(pb + (t - b)));
    const int64_t tl = t - b;
    int cnt = 0;
    constexpr int U = 8;
    for (int64_t j0 = lane; j0 < len; j0 += 32 * U) {
        float v[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t j = j0 + 32 * u;
            v[u] = j < len ? (kShared ? pb[j] : __ldcg(pb + j)) : 0.f;
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t j = j0 + 32 * u;
            const uint32_t kj = orderable(v[u]);
            cnt += (j < len) && ((kj > kt) || (kj == kt && j < tl));
        }
    }
    cnt = __reduce_add_sync(0xFFFFFFFFu, cnt);
    return cnt < r;
}

// One 16-byte chunk of token t's injection: R = sum_j w_j V[row_j] in fp32 (j
// in order, one fma per element and row: the arithmetic of the injection
// kernels), added into every layer sharing the table with one rounding.
__device__ __forceinline__ void inject_chunk(const Params& p, int64_t t, const int32_t* rows, const float* w, int ch) {
    const int64_t vrow = (int64_t)p.dv * 2;
    const int64_t max_row = p.S * p.P - 1;
    const uint4 hv0 = *(reinterpret_cast<const uint4*>(reinterpret_cast<const uint8_t*>(p.hidden[0]) + t * vrow) + ch);
    float acc[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] = 0.f;
    for (int j0 = 0; j0 < p.top_k; j0 += 4) {
        uint4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            if (j0 + u < p.top_k) {
                const int64_t r = min(max((int64_t)rows[j0 + u], (int64_t)0), max_row);
                v[u] = __ldg(reinterpret_cast<const uint4*>(p.values + r * vrow) + ch);
            }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            if (j0 + u < p.top_k) {
                float f[8];
                Vec16<__nv_bfloat16>::unpack(v[u], f);
                const float wu = w[j0 + u];
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[e] = fmaf(wu, f[e], acc[e]);
            }
        }
    }
    for (int l = 0; l < p.n_layers; ++l) {
        uint4* h = reinterpret_cast<uint4*>(reinterpret_cast<uint8_t*>(p.hidden[l]) + t * vrow) + ch;
        float f[8];
        Vec16<__nv_bfloat16>::unpack(l == 0 ? hv0 : *h, f);
#pragma unroll
        for (int e = 0; e < 8; ++e) f[e] += acc[e];
        *h = Vec16<__nv_bfloat16>::pack(f);
    }
}

// The 8 token rows of one item into a token tile (128-byte swizzle, one 1 KiB
// atom per 64-wide k-block): row j's 16-byte chunk c of k-block kb at
// kb * 1 KiB + j * 128 + (c ^ j) * 16; rows past the item's count and columns
// past d_k are zero.  Threads [0, nthr) of the caller share the work.
__device__ __forceinline__ void build_tile(uint32_t tile, const uint8_t* q, int row_bytes, int nkb,
                                           const int32_t* toks, int count, int idx0, int nthr) {
    const int cpr = row_bytes / 16;
    for (int idx = idx0; idx < nkb * 8 * k3tc::kTok; idx += nthr) {
        const int kb = idx / (8 * k3tc::kTok), rem = idx - kb * 8 * k3tc::kTok;
        const int j = rem / 8, c = rem % 8;
        const int cc = kb * 8 + c;
        const uint32_t dst = tile + (uint32_t)(kb * k3tc::kAtomBytes + j * 128 + ((c ^ j) * 16));
        if (j < count && cc < cpr)
            ptx::cp_async16(dst, q + (int64_t)toks[j] * row_bytes + cc * 16);
        else
            asm volatile("st.shared.v4.u32 [%0], {%1, %1, %1, %1};" ::"r"(dst), "r"(0u) : "memory");
    }
}

// The kernel's shared-memory regions and mbarriers.
struct Shm {
    uint8_t* ring;
    uint8_t* btile;
    float* zs;
    Ctl* x;
    uint64_t *full, *empty, *bfull, *bempty, *ifull, *iempty, *dready, *tempty, *drain;
    uint64_t *r_full, *r_empty, *a_full, *a_empty, *t_full, *t_empty, *r_drain;
};
__device__ __forceinline__ Shm shm_of(uint8_t* smem, const Geo& g) {
    Shm m;
    m.ring = smem;
    m.btile = smem + g.off_b;
    m.zs = reinterpret_cast<float*>(smem + g.off_z);
    m.x = reinterpret_cast<Ctl*>(smem + g.off_x);
    uint64_t* b = reinterpret_cast<uint64_t*>(smem + g.off_bar);
    m.full = b;
    m.empty = m.full + k3tc::kMaxStages;
    m.bfull = m.empty + k3tc::kMaxStages;
    m.bempty = m.bfull + kTileCache;
    m.ifull = m.bempty + kTileCache;
    m.iempty = m.ifull + k3tc::kISlots;
    m.dready = m.iempty + k3tc::kISlots;  // [2 group + buffer]
    m.tempty = m.dready + 4;
    m.drain = m.tempty + 2;
    m.r_full = m.drain + 1;
    m.r_empty = m.r_full + kRStagesMax;
    m.a_full = m.r_empty + kRStagesMax;
    m.a_empty = m.a_full + 1;
    m.t_full = m.a_empty + 1;
    m.t_empty = m.t_full + 2;
    m.r_drain = m.t_empty + 2;
    return m;
}

// The level-2 roles.  Their code, with the rest of the kernel's, is kept
// small enough (well under the ~96 KiB an SM's instruction cache holds from
// one launch to the next) to stay cached across calls: an instruction fetched
// behind an SM's full copy ring waits for microseconds.
__device__ __forceinline__ WorkItem item_at(const Params& p, const Ctl* x, int i0, int j) {
    if (j < kItemCache) return x->ic_w[j];
    WorkItem w;
    const int4 v = __ldcg(reinterpret_cast<const int4*>(p.work + i0 + j));
    w.scene = v.x;
    w.begin = v.y;
    w.count = v.z;
    w.slot = v.w;
    return w;
}

__device__ __forceinline__ int nt_cols_of(int64_t P, int nt) {
    const int64_t rows = P - (int64_t)nt * k3tc::kNTile;
    return (int)(rows >= k3tc::kNTile ? k3tc::kNTile : (rows + 15) / 16 * 16);
}

__device__ __forceinline__ void producer_role(const Params& p, const Geo& g, uint8_t* smem, int n_mine, int i0) {
    const Shm m = shm_of(smem, g);
    volatile int* abort = &m.x->abort;
    const int lane = threadIdx.x % 32;
    int64_t stage_seq = 0;
    int slot = 0;
    uint32_t phase = 0;
    bool ok = true;
    const uint64_t policy = ptx::l2_policy_evict_first();
    for (int j = 0; j < n_mine && ok; ++j) {
        const WorkItem w = item_at(p, m.x, i0, j);
        const uint8_t* blk = p.keys_t + (int64_t)w.scene * p.block_bytes;
        for (int c = 0; c < g.chunks && ok; ++c, ++stage_seq) {
            const uint32_t bytes = (uint32_t)(min(g.group, g.spi - c * g.group) * k3tc::kSubBytes);
            if (lane == 0) {
                ok = ptx::mbar_wait(&m.empty[slot], phase ^ 1u, abort, kTimeoutNs);
                if (ok) {
                    ptx::mbar_arrive_expect_tx(&m.full[slot], bytes);
                    ptx::bulk_g2s_hint(m.ring + (int64_t)slot * g.slot_bytes, blk + (int64_t)c * g.slot_bytes, bytes,
                                       &m.full[slot], policy);
                }
            }
            ok = __shfl_sync(0xFFFFFFFFu, (int)ok, 0) != 0;
            if (++slot == g.n_stages) {
                slot = 0;
                phase ^= 1u;
            }
        }
    }
    if (!ok && lane == 0) {
        for (int64_t s = stage_seq - g.n_stages; s < stage_seq; ++s)
            if (s >= 0) ptx::mbar_wait_drain(&m.full[s % g.n_stages], (uint32_t)((s / g.n_stages) & 1), kTimeoutNs);
    }
}

__device__ __forceinline__ void mma_role(const Params& p, const Geo& g, uint8_t* smem, uint32_t tmem_base) {
    const Shm m = shm_of(smem, g);
    volatile int* abort = &m.x->abort;
    if (threadIdx.x % 32 != 0) return;
    const uint32_t a_tiles = ptx::smem_u32(m.btile);
    int slot = 0;
    uint32_t phase = 0;
    int qn = 0;
    bool ok = true;
    for (int i = 0; ok; ++i) {
        const int bs = i % kTileCache;
        if (!(ok = ptx::mbar_wait(&m.bfull[bs], (i / kTileCache) & 1, abort, kTimeoutNs))) break;
        if (m.x->items[i % k3tc::kISlots].count < 0) break;
        ptx::tc_fence_after();
        const uint64_t ad0 = k3tc::sw128_desc(a_tiles + (uint32_t)(bs * g.b_bytes), 0);
        int cur_chunk = -1;
        for (int nt = 0; nt < g.nnt && ok; ++nt, ++qn) {
            const int buf = qn & 1;
            if (!(ok = ptx::mbar_wait(&m.tempty[buf], ((qn >> 1) & 1) ^ 1, abort, kTimeoutNs))) break;
            ptx::tc_fence_after();
            const uint32_t d = tmem_base + (uint32_t)(buf * (g.tmem_cols >> 1));
            const uint32_t idesc = k3tc::idesc_m128(nt_cols_of(p.P, nt));
            const int ns = (nt == g.nnt - 1 && (g.ntile & 1)) ? 1 : 2;
            for (int kb = 0; kb < g.nkb; ++kb) {
                const int sb = nt * 2 * g.nkb + kb * ns;
                const int ch = sb >> g.gshift;
                if (ch != cur_chunk) {
                    if (cur_chunk >= 0) {
                        ptx::mma_commit(&m.empty[slot]);
                        if (++slot == g.n_stages) {
                            slot = 0;
                            phase ^= 1u;
                        }
                    }
                    if (!(ok = ptx::mbar_wait(&m.full[slot], phase, abort, kTimeoutNs))) break;
                    ptx::tc_fence_after();
                    cur_chunk = ch;
                }
                const uint32_t b_addr =
                    ptx::smem_u32(m.ring + (int64_t)slot * g.slot_bytes + (int64_t)(sb - (ch << g.gshift)) * k3tc::kSubBytes);
                k3tc::mma_kblock(1u, d, ad0 + (uint64_t)(kb * (k3tc::kAtomBytes >> 4)), k3tc::sw128_desc(b_addr, 1024),
                                 idesc, kb == 0 ? 1u : 0u);
            }
            if (ok) ptx::mma_commit(&m.dready[(i & 1) * 2 + buf]);
        }
        if (!ok) break;
        ptx::mma_commit(&m.empty[slot]);
        if (++slot == g.n_stages) {
            slot = 0;
            phase ^= 1u;
        }
        ptx::mma_commit(&m.bempty[bs]);
    }
    ptx::mma_commit(m.drain);
    ptx::mbar_wait_drain(m.drain, 0, kTimeoutNs);
}

// Top-k + softmax of one token for the fused step: the register-resident
// variants (a round rescans a lane's elements), whose code is a fraction of the
// sorted-list variants' and gives the same result.
__device__ __forceinline__ k3::TopkLane step_topk(const float* z, int64_t P, int top_k, int lane, int64_t t,
                                                  int32_t* prim_out, float* weight_out) {
    if (P <= 32) return k3tc::topk_regs_fn<1>(z, P, top_k, lane, t, prim_out, weight_out);
    if (P <= 64) return k3tc::topk_regs_fn<2>(z, P, top_k, lane, t, prim_out, weight_out);
    if (P <= 128) return k3tc::topk_regs_fn<4>(z, P, top_k, lane, t, prim_out, weight_out);
    if (P <= 256) return k3tc::topk_regs_fn<8>(z, P, top_k, lane, t, prim_out, weight_out);
    if (P <= 512) return k3tc::topk_regs_fn<16>(z, P, top_k, lane, t, prim_out, weight_out);
    if (P <= 1024) return k3tc::topk_regs_fn<32>(z, P, top_k, lane, t, prim_out, weight_out);
    return k3tc::topk_scan_fn(z, P, top_k, lane, t, prim_out, weight_out);
}

// The end-of-CTA injection of the queued kept tokens by the eight epilogue
// warps, every 16-byte chunk of every queued token spread over them, two
// chunks in flight per thread.
__device__ __noinline__ void inject_queued(const Params& p, Ctl* x, int i0, int e, int lane) {
    const int nk = x->n_kept;
    const int chunks = p.dv / 8;
#pragma unroll 1
    for (int idx = e * 32 + lane; idx < nk * chunks; idx += kEpiThreads) {
        const int u = idx / chunks;
        const int32_t* rows;
        const float* w;
        int64_t t;
        if (u < kKeptCap) {
            t = x->kept_t[u];
            rows = x->kept_row[u];
            w = x->kept_w[u];
        } else {
            t = __ldcg(p.ovf_tok + (int64_t)i0 * k3tc::kTok + (u - kKeptCap));
            rows = p.rec_row + t * kRecMaxTopK;
            w = p.rec_w + t * kRecMaxTopK;
        }
        inject_chunk(p, t, rows, w, idx - u * chunks);
    }
}

__device__ __forceinline__ void epilogue_role(const Params& p, const Geo& g, uint8_t* smem, uint32_t tmem_base, int i0) {
    using k3tc::kTok;
    const Shm m = shm_of(smem, g);
    Ctl* x = m.x;
    volatile int* abort = &x->abort;
    const int lane = threadIdx.x % 32, warp = threadIdx.x / 32;
    const int e = warp - 2;
    const int grp = e / kGroupWarps;
    const int eg = e % kGroupWarps;
    const int quarter = warp & 3;
    const float* prio_g = p.priority ? p.priority : p.qnorm;
    float* zg = m.zs + grp * (g.zbytes / 4);
    const int P = (int)p.P;
    for (int i = grp;; i += 2) {
        const int ms = i % k3tc::kISlots;
        const bool ok0 = __all_sync(0xFFFFFFFFu, ptx::mbar_wait(&m.ifull[ms], (i / k3tc::kISlots) & 1, abort, kTimeoutNs));
        if (group_sync_or(grp, !ok0 || *abort)) break;
        if (x->items[ms].count < 0) break;
        const int nb = min(x->items[ms].count, kTok);
        // The gate of this warp's tokens eg and eg + 4: from the bucketing for
        // cached items, else ranked here from global memory.
        uint32_t keep = 0;
        if (p.gate) {
#pragma unroll 1
            for (int h = 0; h < 2; ++h) {
                const int u = eg + h * kGroupWarps;
                if (u >= nb) break;
                if (i < kItemCache) {
                    keep |= ((x->ic_keep[i] >> u) & 1u) << h;
                } else {
                    const int64_t tg = x->toks[ms * kTok + u];
                    const bool kk = gate_keep<false>(p, prio_g, tg, lane);
                    if (lane == 0 && p.mask_out) p.mask_out[tg] = (uint8_t)kk;
                    keep |= (uint32_t)kk << h;
                }
            }
        }
        for (int nt = 0; nt < g.nnt; ++nt) {
            const int qn = i * g.nnt + nt, buf = qn & 1;
            const int mm = i >> 1;
            const int per_item = (g.nnt & 1) ? (g.nnt + (((buf ^ grp) & 1) ? -1 : 1)) / 2 : g.nnt / 2;
            const uint32_t par = (uint32_t)(mm * per_item + (nt >> 1)) & 1u;
            const bool ok = __all_sync(0xFFFFFFFFu, ptx::mbar_wait(&m.dready[grp * 2 + buf], par, abort, kTimeoutNs));
            const int ncols = nt_cols_of(p.P, nt);
            // Warp eg reads columns [64 eg, 64 eg + 64) of its TMEM lane quarter
            // (16 at a time; N is a multiple of 16); lane j < 8 of any quarter
            // holds token j (D row r is token r % 8).
            ptx::tc_fence_after();
#pragma unroll 1
            for (int c0 = eg * 64; ok && c0 < min(ncols, eg * 64 + 64); c0 += 16) {
                uint32_t r[16];
                ptx::tmem_ld_32x32b_x16(tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(buf * (g.tmem_cols >> 1) + c0), r);
                ptx::tmem_wait_ld();
                const int p0 = nt * k3tc::kNTile + c0;
                if (lane < nb) {
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        if (p0 + j < P) zg[(p0 + j) * k3tc::kZStride + lane] = __uint_as_float(r[j]) * p.scale;
                }
            }
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&m.tempty[buf]);
        }
        if (group_sync_or(grp, *abort)) break;  // all logits of the item are in shared memory
#pragma unroll 1
        for (int h = 0; h < 2; ++h) {
            const int u = eg + h * kGroupWarps;
            if (u >= nb) break;
            const int64_t t = x->toks[ms * kTok + u];
            const k3::TopkLane r = step_topk(zg + u, p.P, p.top_k, lane, t, p.prim_out, p.weight_out);
            if ((keep >> h) & 1u) {
                // Queue the kept token for the end-of-CTA injection and send its
                // value rows into L2 meanwhile.
                int q = 0;
                if (lane == 0) q = atomicAdd(&x->n_kept, 1);
                q = __shfl_sync(0xFFFFFFFFu, q, 0);
                const int64_t row = (int64_t)x->items[ms].scene * p.P + r.p;
                if (lane < p.top_k) {
                    if (q < kKeptCap) {
                        x->kept_row[q][lane] = (int32_t)row;
                        x->kept_w[q][lane] = r.w;
                    } else {
                        // Past the queue's room: the record by token id in global memory.
                        p.rec_row[t * kRecMaxTopK + lane] = (int32_t)row;
                        p.rec_w[t * kRecMaxTopK + lane] = r.w;
                    }
                    k3tc::prefetch_row_l2(p.values + row * (int64_t)p.dv * 2, (int64_t)p.dv * 2);
                }
                if (lane == 0) {
                    if (q < kKeptCap) x->kept_t[q] = (int32_t)t;
                    else p.ovf_tok[(int64_t)i0 * kTok + (q - kKeptCap)] = (int32_t)t;
                }
            }
        }
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(&m.iempty[ms]);
    }
    // Every epilogue warp has scored its last item: inject the queued tokens.
    if (p.gate) {
        asm volatile("bar.sync 3, %0;" ::"n"(kEpiThreads) : "memory");
        inject_queued(p, x, i0, e, lane);
    }
}

__device__ __forceinline__ void token_role(const Params& p, const Geo& g, uint8_t* smem, int n_mine, int i0) {
    using k3tc::kTok;
    const Shm m = shm_of(smem, g);
    Ctl* x = m.x;
    volatile int* abort = &x->abort;
    const int lane = threadIdx.x % 32;
    // The first kTileCache tiles were built before the key stream; later items
    // reuse a tile once the MMAs of the item kTileCache before are done.
    const uint32_t bt0 = ptx::smem_u32(m.btile);
    bool ok = true;
    int ends = 0;
    for (int i = 0; ends < 2; ++i) {
        const int ms = i % k3tc::kISlots, bs = i % kTileCache;
        if (lane == 0 && i >= k3tc::kISlots)
            ok = ptx::mbar_wait(&m.iempty[ms], ((i / k3tc::kISlots) & 1) ^ 1, abort, kTimeoutNs);
        if (lane == 0 && ok && i >= kTileCache)
            ok = ptx::mbar_wait(&m.bempty[bs], ((i / kTileCache) & 1) ^ 1, abort, kTimeoutNs);
        if (!__shfl_sync(0xFFFFFFFFu, (int)ok, 0)) break;
        if (i >= n_mine) {
            if (lane == 0) {
                x->items[ms].count = -1;
                ptx::mbar_arrive(&m.ifull[ms]);
                if (ends == 0) ptx::mbar_arrive(&m.bfull[bs]);
            }
            ++ends;
            continue;
        }
        const WorkItem w = item_at(p, x, i0, i);
        const int nb = min(w.count, kTok);
        int32_t tok = 0;
        if (lane < nb)
            tok = i < kItemCache ? x->ic_tok[i * kTok + lane] : __ldcg(p.item_tok + (int64_t)(i0 + i) * kTok + lane);
        if (lane < nb) x->toks[ms * kTok + lane] = tok;
        if (i >= kTileCache) {
            __syncwarp();
            build_tile(bt0 + (uint32_t)(bs * g.b_bytes), reinterpret_cast<const uint8_t*>(p.q), g.row_bytes, g.nkb,
                       x->toks + ms * kTok, nb, lane, 32);
            ptx::cp_async_wait_all();
            ptx::fence_proxy_async_smem();
        }
        if (lane == 0) x->items[ms] = w;
        __syncwarp();
        if (lane == 0) {
            ptx::mbar_arrive(&m.ifull[ms]);
            ptx::mbar_arrive(&m.bfull[bs]);
        }
    }
}

}  // namespace kst

__global__ void __launch_bounds__(kst::kThreads, 1)
    k_step_tc(const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_c,
              const __grid_constant__ kst::Params p, const __grid_constant__ kst::Geo g) {
    using namespace kst;
    using k3tc::kTok;
    using k3tc::kISlots;
    using k3tc::kMaxStages;
    using k3tc::kSubBytes;
    using k3tc::kAtomBytes;
    using k3tc::kNTile;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* ring = smem;
    uint8_t* btile = smem + g.off_b;
    float* zs = reinterpret_cast<float*>(smem + g.off_z);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + g.off_bar);
    // level 2
    uint64_t* full = bars;
    uint64_t* empty = full + kMaxStages;
    uint64_t* bfull = empty + kMaxStages;
    uint64_t* bempty = bfull + kTileCache;
    uint64_t* ifull = bempty + kTileCache;
    uint64_t* iempty = ifull + kISlots;
    uint64_t* dready = iempty + kISlots;  // [2 group + buffer]
    uint64_t* tempty = dready + 4;
    uint64_t* drain = tempty + 2;
    // routing
    uint64_t* r_full = drain + 1;
    uint64_t* r_empty = r_full + kRStagesMax;
    uint64_t* a_full = r_empty + kRStagesMax;
    uint64_t* a_empty = a_full + 1;
    uint64_t* t_full = a_empty + 1;
    uint64_t* t_empty = t_full + 2;
    uint64_t* r_drain = t_empty + 2;
    Ctl* x = reinterpret_cast<Ctl*>(smem + g.off_x);
    volatile int* abort = &x->abort;

    const int tid = threadIdx.x, lane = tid % 32, warp = tid / 32;
    const int G = gridDim.x, cta = blockIdx.x;
    StepState* st = p.state;

    if (tid == 0) {
        ptx::prefetch_tmap(&tmap_q);
        ptx::prefetch_tmap(&tmap_c);
        for (int i = 0; i < g.n_stages; ++i) {
            ptx::mbar_init(&full[i], 1);
            ptx::mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < kTileCache; ++i) {
            ptx::mbar_init(&bfull[i], 1);
            ptx::mbar_init(&bempty[i], 1);
        }
        for (int i = 0; i < kISlots; ++i) {
            ptx::mbar_init(&ifull[i], 1);
            ptx::mbar_init(&iempty[i], kGroupWarps);
        }
        for (int i = 0; i < 4; ++i) ptx::mbar_init(&dready[i], 1);
        for (int i = 0; i < 2; ++i) ptx::mbar_init(&tempty[i], kGroupWarps);
        ptx::mbar_init(drain, 1);
        for (int i = 0; i < g.rstages; ++i) {
            ptx::mbar_init(&r_full[i], 1);
            ptx::mbar_init(&r_empty[i], 1);
        }
        ptx::mbar_init(a_full, 1);
        ptx::mbar_init(a_empty, 1 + kRouteEpi);  // the MMA issuer's commit and each routing epilogue warp
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(&t_full[i], 1);
            ptx::mbar_init(&t_empty[i], kRouteEpi);
        }
        ptx::mbar_init(r_drain, 1);
        x->abort = 0;
        x->epoch = *reinterpret_cast<volatile uint32_t*>(&st->epoch);
        x->i0 = INT_MAX;
        x->i1 = -1;
        x->maxb = 0;
        ptx::fence_mbar_init();
    }
    if (warp == 1) ptx::tmem_alloc(&x->tmem_slot, g.tmem_alloc);
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem_base = x->tmem_slot;
    const uint32_t eb = x->epoch & 1u;
    unsigned long long* best = st->best[eb];

    // ================================================================ phase 1
    {
        const int BN = g.BN, nkb = g.nkb;
        uint8_t* sA = ring;
        uint8_t* sB = ring + g.r_off_b;
        float* s_ic = reinterpret_cast<float*>(ring + g.r_off_c);
        float* s_bias = s_ic + 2 * BN;
        const int n_tiles = (int)((p.S + BN - 1) / BN);
        const int64_t n_units = (int64_t)((p.N + kRouteBM - 1) / kRouteBM) * n_tiles;
        const int64_t u0 = (int64_t)cta * g.units_per_cta;
        const int64_t u1 = min(n_units, u0 + g.units_per_cta);
        if (warp == 0) {
            if (lane == 0 && u0 < u1) {
                int stage = 0;
                uint32_t phase = 0, issued = 0, last_par = 0;
                int seg = -1;
                int64_t m_cur = -1;
                bool ok = true;
                for (int64_t u = u0; u < u1 && ok; ++u) {
                    const int64_t m = u / n_tiles;
                    const int nt = (int)(u - m * n_tiles);
                    if (m != m_cur) {
                        if (seg >= 0 && !(ok = ptx::mbar_wait(a_empty, (uint32_t)(seg & 1), abort, kTimeoutNs))) break;
                        ++seg;
                        m_cur = m;
                        ptx::mbar_arrive_expect_tx(a_full, (uint32_t)(nkb * kRouteBM * 128));
                        for (int kb = 0; kb < nkb; ++kb)
                            ptx::tma_load_2d(sA + kb * kRouteBM * 128, &tmap_q, kb * 64, (int32_t)(m * kRouteBM), a_full);
                    }
                    for (int kb = 0; kb < nkb; ++kb) {
                        if (!(ok = ptx::mbar_wait(&r_empty[stage], phase ^ 1u, abort, kTimeoutNs))) break;
                        ptx::mbar_arrive_expect_tx(&r_full[stage], (uint32_t)(BN * 128));
                        ptx::tma_load_2d(sB + stage * BN * 128, &tmap_c, kb * 64, nt * BN, &r_full[stage]);
                        issued |= 1u << stage;
                        last_par = (last_par & ~(1u << stage)) | (phase << stage);
                        if (++stage == g.rstages) {
                            stage = 0;
                            phase ^= 1u;
                        }
                    }
                }
                // Every copy issued has landed before the ring is reused.
                if (seg >= 0) ptx::mbar_wait_drain(a_full, (uint32_t)(seg & 1), kTimeoutNs);
                for (int i = 0; i < g.rstages; ++i)
                    if (issued & (1u << i)) ptx::mbar_wait_drain(&r_full[i], (last_par >> i) & 1u, kTimeoutNs);
            }
        } else if (warp == 1) {
            if (lane == 0 && u0 < u1) {
                const uint32_t idesc = k3tc::idesc_m128(BN);
                bool ok = true;
                int stage = 0;
                uint32_t phase = 0;
                int seg = -1;
                int64_t m_cur = -1;
                for (int64_t u = u0, it = 0; u < u1 && ok; ++u, ++it) {
                    const int64_t m = u / n_tiles;
                    if (m != m_cur) {
                        if (seg >= 0) ptx::mma_commit(a_empty);
                        ++seg;
                        m_cur = m;
                        if (!(ok = ptx::mbar_wait(a_full, (uint32_t)(seg & 1), abort, kTimeoutNs))) break;
                    }
                    const int buf = (int)(it & 1);
                    const uint32_t use = (uint32_t)(it >> 1);
                    if (!(ok = ptx::mbar_wait(&t_empty[buf], (use & 1u) ^ 1u, abort, kTimeoutNs))) break;
                    ptx::tc_fence_after();
                    const uint32_t d_tmem = tmem_base + (uint32_t)(buf * BN);
                    for (int kb = 0; kb < nkb; ++kb) {
                        if (!(ok = ptx::mbar_wait(&r_full[stage], phase, abort, kTimeoutNs))) break;
                        ptx::tc_fence_after();
                        const uint32_t a0 = ptx::smem_u32(sA + kb * kRouteBM * 128);
                        const uint32_t b0 = ptx::smem_u32(sB + stage * BN * 128);
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            ptx::mma_bf16(d_tmem, ptx::sw128_kmajor_desc(a0 + k * 32), ptx::sw128_kmajor_desc(b0 + k * 32),
                                          idesc, (kb | k) != 0);
                        ptx::mma_commit(&r_empty[stage]);
                        if (++stage == g.rstages) {
                            stage = 0;
                            phase ^= 1u;
                        }
                    }
                    if (ok) ptx::mma_commit(&t_full[buf]);
                }
                ptx::mma_commit(r_drain);
                ptx::mbar_wait_drain(r_drain, 0, kTimeoutNs);
            }
        } else if (warp < 2 + kRouteEpi) {
            // Warp w owns TMEM lane quarter (w % 4) and column half (w - 2) / 4 of every tile.
            const int quarter = warp & 3;
            const int half = (warp - 2) / 4;
            const int HC = BN / 2;
            const int et = tid - 64;  // 0 .. 255; BN <= 256, so one scene constant per thread and tile
            const float nan = __int_as_float(0x7fc00000);
            float ic_next = nan, b_next = 0.f;
            auto load_consts = [&](int nt) {
                const int64_t s = (int64_t)nt * BN + et;
                const bool in = et < BN && s < p.S;
                ic_next = in ? __ldg(p.inv_cnorm + s) : nan;
                b_next = (in && p.bias) ? __ldg(p.bias + s) : 0.f;
            };
            auto store_consts = [&](int buf) {
                if (et < BN) {
                    s_ic[buf * BN + et] = ic_next;
                    s_bias[buf * BN + et] = b_next;
                }
            };
            if (u0 < u1) {
                load_consts((int)(u0 % n_tiles));
                store_consts(0);
            }
            float best_v = -INFINITY;
            int64_t best_s = -1, row = -1;
            float inv_q = 1.f;
            int seg = -1;
            int64_t m_cur = -1;
            for (int64_t u = u0, it = 0; u < u1; ++u, ++it) {
                const int64_t m = u / n_tiles;
                const int nt = (int)(u - m * n_tiles);
                const int buf = (int)(it & 1);
                const uint32_t use = (uint32_t)(it >> 1);
                if (u + 1 < u1) load_consts((int)((u + 1) % n_tiles));
                if (m != m_cur) {
                    if (row >= 0 && row < p.N && best_s >= 0 && !*abort)
                        atomicMax(&best[row], pack_argmax(best_v, (uint32_t)best_s));
                    best_v = -INFINITY;
                    best_s = -1;
                    ++seg;
                    m_cur = m;
                    row = m * kRouteBM + quarter * 32 + lane;
                    const bool ready = ptx::mbar_wait(a_full, (uint32_t)(seg & 1), abort, kTimeoutNs);
                    const bool store = nt == 0 && half == 0;
                    if (ready && (store || p.bias)) {
                        // ||q_row||_2 from the token tile in shared memory (the
                        // swizzle permutes 16-byte chunks within the row).
                        float ss = 0.f;
                        const int r = quarter * 32 + lane;
                        for (int kb = 0; kb < nkb; ++kb) {
#pragma unroll 2
                            for (int c = 0; c < 8; ++c) {
                                float f[8];
                                Vec16<__nv_bfloat16>::unpack(
                                    *reinterpret_cast<const uint4*>(sA + kb * kRouteBM * 128 + r * 128 + (((c + lane) & 7) * 16)),
                                    f);
#pragma unroll
                                for (int i = 0; i < 8; ++i) ss = fmaf(f[i], f[i], ss);
                            }
                        }
                        const float n = sqrtf(ss);
                        if (store && row < p.N) {
                            p.qnorm[row] = n;
                            if (p.qnorm_out) p.qnorm_out[row] = n;
                        }
                        if (p.bias) inv_q = n > 0.f ? 1.f / n : 0.f;
                    }
                    __syncwarp();
                    if (lane == 0) ptx::mbar_arrive(a_empty);
                }
                const bool ready = ptx::mbar_wait(&t_full[buf], use & 1u, abort, kTimeoutNs);
                if (route_epi_sync_or(!__all_sync(0xFFFFFFFFu, ready))) break;
                ptx::tc_fence_after();
                const int c0 = half * HC;
                const float* ic = s_ic + buf * BN + c0;
                const float* bs = s_bias + buf * BN + c0;
                float tv = -INFINITY;
                int tc = -1;
#pragma unroll 1
                for (int c = 0; c < HC; c += 16) {
                    uint32_t r[16];
                    ptx::tmem_ld_32x32b_x16(tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(buf * BN + c0 + c), r);
                    ptx::tmem_wait_ld();
                    if (p.bias) {
#pragma unroll 4
                        for (int j = 0; j < 16; ++j) {
                            const float score = fmaf(__uint_as_float(r[j]) * ic[c + j], inv_q, bs[c + j]);
                            if (score > tv) {
                                tv = score;
                                tc = c + j;
                            }
                        }
                    } else {
#pragma unroll 4
                        for (int j = 0; j < 16; ++j) {
                            const float score = __uint_as_float(r[j]) * ic[c + j];
                            if (score > tv) {
                                tv = score;
                                tc = c + j;
                            }
                        }
                    }
                }
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(&t_empty[buf]);
                if (u + 1 < u1) store_consts(buf ^ 1);
                if (tc >= 0 && tv > best_v) {  // later tiles of a token tile hold larger scene indices
                    best_v = tv;
                    best_s = (int64_t)nt * BN + c0 + tc;
                }
            }
            if (row >= 0 && row < p.N && best_s >= 0 && !*abort) atomicMax(&best[row], pack_argmax(best_v, (uint32_t)best_s));
        } else if (warp == kTokWarp) {
            // The buffers of the next call: its argmax keys and barrier counter.
            unsigned long long* nb = st->best[eb ^ 1u];
            const int64_t per = (kStepMaxTokens + G - 1) / G;
            for (int64_t i = (int64_t)cta * per + lane; i < min(kStepMaxTokens, (int64_t)(cta + 1) * per); i += 32)
                nb[i] = 0ull;
            if (cta == 0 && lane == 0) st->bar[eb ^ 1u] = 0u;
        }
    }
    ptx::tc_fence_before();
    __syncthreads();

    // ================================================================ phase 2
    if (tid == 0) {
        __threadfence();
        atomicAdd(&st->bar[eb], 1u);
    }
    int n_mine = 0, i0 = 0;
    ptx::tc_fence_before();
    if (tid == 0) {
        const uint64_t t0 = ptx::globaltimer_ns();
        while (ld_acquire_gpu(&st->bar[eb]) < (uint32_t)G) {
            if (ptx::globaltimer_ns() - t0 > kTimeoutNs) {
                x->abort = 1;
                break;
            }
        }
        __threadfence();
    }
    __syncthreads();
    ptx::tc_fence_after();

    // ================================================================ phase 3
    // (32-bit indices throughout: N <= kStepMaxTokens and S < 2^31 / P.)
    const int N = (int)p.N, S = (int)p.S;
    // The ring stays free for the key stream, which starts before the end of
    // this phase: scene counts and token scenes live in the tile cache (dead
    // before its tiles are built), the gate priorities in the logit area
    // (dead before the first logits arrive).
    int* hist = reinterpret_cast<int*>(btile);                                // [S] counts, then positions
    int32_t* tscene = reinterpret_cast<int32_t*>(btile + (S * 4 + 15) / 16 * 16);  // [N] every token's scene
    float* prio = zs;                                                         // [N] gate priorities
    const float* prio_g = p.priority ? p.priority : p.qnorm;
    for (int s = tid; s < S; s += kThreads) hist[s] = 0;
    if (tid < kItemCache) x->ic_keep[tid] = 0u;
    for (int k = tid; k < kItemCache * kTok; k += kThreads) x->gcnt[k] = 0;
    if (tid == 0) x->n_kept = 0;
    __syncthreads();
    // Keys (and priorities) in batches of kB per thread, every load of a batch
    // in flight at once.
    constexpr int kB = 4;
#pragma unroll 1
    for (int t0 = tid; t0 < N; t0 += kB * kThreads) {
        unsigned long long key[kB];
        float pv[kB];
#pragma unroll
        for (int u = 0; u < kB; ++u) {
            const int t = t0 + u * kThreads;
            key[u] = t < N ? __ldcg(&best[t]) : 0ull;
            pv[u] = (p.gate && t < N) ? __ldcg(prio_g + t) : 0.f;
        }
#pragma unroll
        for (int u = 0; u < kB; ++u) {
            const int t = t0 + u * kThreads;
            if (t < N) {
                const int32_t sc = unpack_scene(key[u], S);
                tscene[t] = sc;
                prio[t] = pv[u];
                atomicAdd(&hist[sc], 1);
            }
        }
    }
    __syncthreads();
    // Each thread a contiguous run of scenes: work items and routed scenes, scanned.
    const int per = (S + kThreads - 1) / kThreads;
    const int s0 = min(S, tid * per), s1 = min(S, s0 + per);
    int2 mine = make_int2(0, 0);
    int mx = 0;
    for (int s = s0; s < s1; ++s) {
        const int c = hist[s];
        mine.x += (c + kTokensPerItem - 1) / kTokensPerItem;
        mine.y += c > 0;
        mx = max(mx, c);
    }
    int2 base, total;
    block_scan2(mine, base, total, x->warp_buf);
    const int I = total.x;
    const int lo = (int)((int64_t)I * cta / G), hi = (int)((int64_t)I * (cta + 1) / G);
    {
        int wi = base.x;
        for (int s = s0; s < s1; ++s) {
            const int c = hist[s];
            if (c > 0) {
                const int ni = (c + kTokensPerItem - 1) / kTokensPerItem;
                if (lo <= wi && wi < hi) {
                    atomicMin(&x->i0, wi);
                    atomicMax(&x->i1, wi + ni);
                }
                wi += ni;
            }
        }
        mx = __reduce_max_sync(0xFFFFFFFFu, mx);
        if (lane == 0 && mx) atomicMax(&x->maxb, mx);
    }
    __syncthreads();
    i0 = x->i0;
    n_mine = (i0 == INT_MAX || *abort) ? 0 : x->i1 - i0;
    if (cta == 0 && tid == 0) {
        p.counters[0] = I;
        p.counters[1] = total.y;
        p.counters[2] = x->maxb;
    }
    {
        int wi = base.x, slot = base.y;
        for (int s = s0; s < s1; ++s) {
            const int c = hist[s];
            const int ni = (c + kTokensPerItem - 1) / kTokensPerItem;
            const bool m = c > 0 && lo <= wi && wi < hi;
            hist[s] = m ? wi * kTokensPerItem : -1;
            for (int j = 0; m && j < ni; ++j) {
                const WorkItem w{s, (wi + j) * kTokensPerItem, min(kTokensPerItem, c - j * kTokensPerItem), slot};
                p.work[wi + j] = w;
                if (wi + j - i0 < kItemCache) x->ic_w[wi + j - i0] = w;
            }
            if (c > 0) {
                wi += ni;
                ++slot;
            }
        }
    }
    __syncthreads();
    // The owned scenes' tokens into their items (order inside a scene is
    // free: only this CTA reads these items), and their scenes.
    for (int t = tid; t < N; t += kThreads) {
        const int32_t sc = tscene[t];
        if (hist[sc] >= 0) {
            const int pos = atomicAdd(&hist[sc], 1);
            p.item_tok[pos] = t;
            if (pos - i0 * kTokensPerItem < kItemCache * kTokensPerItem) x->ic_tok[pos - i0 * kTokensPerItem] = t;
            p.scene_out[t] = sc;
        }
    }
    __syncthreads();
    // The key stream starts now (warp 0); the other warps build the first
    // items' token tiles (their query-row loads issued before any key copy,
    // so they do not queue behind one) and decide the gate, then meet at
    // named barrier 5.
    if (warp == 0) {
        producer_role(p, g, smem, n_mine, i0);
    } else {
        constexpr int kRest = kThreads - 32;
        const int rt = tid - 32;
        {
            const int nt = min(n_mine, kTileCache);
            const uint32_t bt0 = ptx::smem_u32(btile);
            const int per_tile = g.nkb * 8 * kTok;
            for (int idx = rt; idx < nt * per_tile; idx += kRest) {
                const int j = idx / per_tile;
                build_tile(bt0 + (uint32_t)(j * g.b_bytes), reinterpret_cast<const uint8_t*>(p.q), g.row_bytes, g.nkb,
                           x->ic_tok + j * kTok, min(x->ic_w[j].count, kTok), idx - j * per_tile, per_tile);
            }
        }
        // The gate for the tokens of the cached items, one item (up to 8 tokens)
        // per pass: every thread compares its share of the priorities with the
        // item's tokens' (each against its own segment), then 8 warp reductions
        // and shared atomics.  A kept token's hidden rows go into L2 now.
        const int n_ci = min(n_mine, kItemCache);
        if (p.gate) {
#pragma unroll 1
            for (int j = 0; j < n_ci; ++j) {
                const int cnt = min(x->ic_w[j].count, kTok);  // uniform
                uint32_t kt[kTok];
                int tt[kTok], sb[kTok], se[kTok];
#pragma unroll
                for (int u = 0; u < kTok; ++u) {
                    tt[u] = u < cnt ? x->ic_tok[j * kTok + u] : 0;
                    const int sg = segment_of(p, tt[u]);
                    sb[u] = u < cnt ? (int)p.seg_off[sg] : 0;
                    se[u] = u < cnt ? (int)p.seg_off[sg + 1] : 0;  // empty range for unused slots
                    kt[u] = orderable(prio[tt[u]]);
                }
                int c[kTok];
#pragma unroll
                for (int u = 0; u < kTok; ++u) c[u] = 0;
                for (int jj = rt; jj < N; jj += kRest) {
                    const uint32_t kj = orderable(prio[jj]);
#pragma unroll
                    for (int u = 0; u < kTok; ++u)
                        c[u] += (jj >= sb[u] && jj < se[u]) && ((kj > kt[u]) || (kj == kt[u] && jj < tt[u]));
                }
#pragma unroll
                for (int u = 0; u < kTok; ++u) {
                    const int cu = __reduce_add_sync(0xFFFFFFFFu, c[u]);
                    if (lane == 0 && cu) atomicAdd(&x->gcnt[j * kTok + u], cu);
                }
            }
            asm volatile("bar.sync 5, %0;" ::"n"(kRest) : "memory");
            const int n_ck = n_ci * kTok;
            if (rt < n_ck && (rt & (kTok - 1)) < x->ic_w[rt / kTok].count) {
                const int t = x->ic_tok[rt];
                const bool keep = x->gcnt[rt] < p.seg_r[segment_of(p, t)];
                if (p.mask_out) p.mask_out[t] = (uint8_t)keep;
                if (keep) {
                    atomicOr(&x->ic_keep[rt / kTok], 1u << (rt & (kTok - 1)));
                    const int vrow = p.dv * 2;
                    for (int l = 0; l < p.n_layers; ++l)
                        for (int o = 0; o < vrow; o += 128)
                            asm volatile("prefetch.global.L2 [%0];" ::"l"(reinterpret_cast<const uint8_t*>(p.hidden[l]) +
                                                                          (int64_t)t * vrow + o));
                }
            }
        }
        ptx::cp_async_wait_all();
        // The tiles are read by the tensor core (async proxy), the logit area
        // is written by the epilogue next.
        ptx::fence_proxy_async_smem();
        asm volatile("bar.sync 5, %0;" ::"n"(kRest) : "memory");

        // ============================================================ phase 4
        if (warp == 1) mma_role(p, g, smem, tmem_base);
        else if (warp < kTokWarp) epilogue_role(p, g, smem, tmem_base, i0);
        else token_role(p, g, smem, n_mine, i0);
    }


    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem_base, g.tmem_alloc);
    }
    if (tid == 0) {
        if (*abort) atomicOr(p.status, STATUS_WAIT_TIMEOUT | STATUS_IN_STEP);
        // The last CTA out advances the epoch: the next call uses the other buffers.
        __threadfence();
        const uint32_t k = atomicAdd(&st->exit_cnt, 1u);
        if (k == (uint32_t)G - 1) {
            st->exit_cnt = 0u;
            __threadfence();
            atomicExch(&st->epoch, x->epoch + 1u);
        }
    }
}

bool step_shape_supported(int64_t N, int64_t S, int64_t P, int dk, int dv, int num_sms) {
    kst::Geo g;
    return N >= 1 && dv % 8 == 0 && kst::geometry(N, S, P, dk, num_sms, g);
}

cudaError_t launch_step(const LaunchCtx& c, const void* tmap_q, const void* const tmap_c[3], const StepArgs& a) {
    kst::Geo g;
    if (!kst::geometry(a.N, a.S, a.P, a.dk, c.num_sms, g) || a.top_k > kRecMaxTopK || a.n_seg > kMaxGateSegments)
        return cudaErrorInvalidConfiguration;
    kst::Params p;
    p.N = a.N;
    p.S = a.S;
    p.P = a.P;
    p.dk = a.dk;
    p.dv = a.dv;
    p.top_k = a.top_k;
    p.scale = a.scale;
    p.q = static_cast<const __nv_bfloat16*>(a.q);
    p.keys_t = static_cast<const uint8_t*>(a.keys_tiled);
    p.block_bytes = a.block_bytes;
    p.values = static_cast<const uint8_t*>(a.values);
    p.inv_cnorm = a.inv_cnorm;
    p.bias = a.bias;
    p.scene_out = a.scene_out;
    p.prim_out = a.prim_out;
    p.weight_out = a.weight_out;
    p.qnorm = a.qnorm;
    p.qnorm_out = a.qnorm_out;
    p.gate = a.gate;
    p.n_seg = a.n_seg;
    p.priority = a.priority;
    p.mask_out = a.mask_out;
    for (int i = 0; i <= kMaxGateSegments; ++i) p.seg_off[i] = a.seg_off[i];
    for (int i = 0; i < kMaxGateSegments; ++i) p.seg_r[i] = a.seg_r[i];
    p.n_layers = a.n_layers;
    for (int l = 0; l < LOOKME_MAX_LAYERS; ++l) p.hidden[l] = l < a.n_layers ? a.hidden[l] : nullptr;
    p.state = a.state;
    p.work = a.work;
    p.item_tok = a.item_tok;
    p.counters = a.counters;
    p.status = a.status;
    p.rec_row = a.rec_row;
    p.rec_w = a.rec_w;
    p.ovf_tok = a.ovf_tok;
    const int which = g.BN == 256 ? 2 : (g.BN == 128 ? 1 : 0);
    CUtensorMap mq, mc;
    memcpy(&mq, tmap_q, sizeof(CUtensorMap));
    memcpy(&mc, tmap_c[which], sizeof(CUtensorMap));
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(c.num_sms);
    cfg.blockDim = dim3(kst::kThreads);
    cfg.dynamicSmemBytes = (size_t)g.smem;
    cfg.stream = c.stream;
    // Cooperative: every CTA resident at once (the grid barrier needs it).
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k_step_tc, mq, mc, p, g);
}

cudaError_t configure_step_kernel() {
    return cudaFuncSetAttribute(k_step_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, kst::kSmemLimit);
}

}  // namespace lookme
