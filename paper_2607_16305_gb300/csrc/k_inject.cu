// Sparse injection (Sec. "Sparse Injection" and "Inter-Layer Sparse Activation").
//
// K5 select: the intra-layer gate as top-r selection.  In each segment the
//   r = floor(len * keep_ratio) tokens of largest priority are kept (ties:
//   lower token index).  One CTA per segment finds the r-th largest priority
//   with a 4-pass, 8-bit radix select over order-preserving integer keys,
//   keeps every token above it and the first tokens equal to it, and compacts
//   the kept ids in ascending order.
// K4 inject: for every kept token t, R_t = sum_j w_tj V[scene_t, prim_tj, :]
//   accumulated in fp32 from 16-byte vector loads, then h_l[t] += R_t for every
//   layer l sharing the table, rounded once to the hidden dtype.  Rows that are
//   not kept are never touched.
#include "common.cuh"
#include "select.cuh"

namespace lookme {

namespace k5 {
constexpr int kThreads = sel::kSelectThreads;

struct Params {
    const float* priority;
    uint8_t* mask;
    int32_t* sel;
    double keep_ratio;
    int n_seg;
    int64_t off[LOOKME_MAX_SEGMENTS + 1];
};

__device__ __forceinline__ uint32_t prio_key(float f) { return orderable(f); }

}  // namespace k5

__global__ void __launch_bounds__(k5::kThreads, 1) k5_select(const __grid_constant__ k5::Params p) {
    pdl_trigger();
    pdl_wait();
    const int seg = blockIdx.x;
    const int64_t b = p.off[seg], len = p.off[seg + 1] - p.off[seg];
    const int64_t r = (int64_t)floor((double)len * p.keep_ratio);
    int64_t sel_base = 0;
    for (int i = 0; i < seg; ++i) sel_base += (int64_t)floor((double)(p.off[i + 1] - p.off[i]) * p.keep_ratio);
    sel::select_segment(p.priority, b, len, r, sel_base, p.mask, p.sel);
}

cudaError_t launch_select(const LaunchCtx& c, const float* priority, int64_t N, const int64_t* seg_off_host,
                          int n_seg, double keep_ratio, uint8_t* mask, int32_t* sel) {
    if (N == 0 || n_seg == 0) return cudaSuccess;
    k5::Params p;
    p.priority = priority;
    p.mask = mask;
    p.sel = sel;
    p.keep_ratio = keep_ratio;
    p.n_seg = n_seg;
    for (int i = 0; i <= n_seg; ++i) p.off[i] = seg_off_host ? seg_off_host[i] : (i == 0 ? 0 : N);
    return launch_pdl(k5_select, dim3(n_seg), dim3(k5::kThreads), 0, c.stream, p);
}

// ---------------------------------------------------------------- K4 inject
namespace k4 {
constexpr int kThreads = 256;

struct Params {
    const void* values;
    int64_t P;
    int dv;
    int top_k;
    const int32_t* scene;
    const int32_t* prim;
    const float* weight;
    const int32_t* sel;
    int64_t N;
    int64_t S;
    int n_layers;
    void* hidden[LOOKME_MAX_LAYERS];
    uint32_t* status;
};
}  // namespace k4

// Row pointers and weights of token t's k value rows, in shared memory.
template <typename T>
__device__ __forceinline__ void load_rows(const k4::Params& p, int64_t t, const uint4** rows, float* w) {
    const int64_t s = min(max((int64_t)p.scene[t], (int64_t)0), p.S - 1);
    for (int j = threadIdx.x; j < p.top_k; j += blockDim.x) {
        const int64_t pr = min(max((int64_t)p.prim[t * p.top_k + j], (int64_t)0), p.P - 1);
        rows[j] = reinterpret_cast<const uint4*>(reinterpret_cast<const T*>(p.values) + (s * p.P + pr) * p.dv);
        w[j] = p.weight[t * p.top_k + j];
    }
}

// Weighted sum of the k rows (fp32) added into token t's row of every layer,
// one rounding; the CTA's threads stride over 16-byte chunks of the row.
template <typename T>
__device__ __forceinline__ void accumulate_store(const k4::Params& p, int64_t t, const uint4* const* rows,
                                                 const float* w) {
    constexpr int EPC = Vec16<T>::N;
    constexpr int BATCH = 8;  // value rows in flight per thread
    const int chunks = p.dv / EPC;
    for (int ch = threadIdx.x; ch < chunks; ch += blockDim.x) {
        uint4* h0 = reinterpret_cast<uint4*>(reinterpret_cast<T*>(p.hidden[0]) + t * p.dv) + ch;
        const uint4 hv0 = *h0;  // issued together with the value rows
        float acc[EPC];
#pragma unroll
        for (int e = 0; e < EPC; ++e) acc[e] = 0.f;
        for (int j0 = 0; j0 < p.top_k; j0 += BATCH) {
            uint4 v[BATCH];
#pragma unroll
            for (int u = 0; u < BATCH; ++u)
                if (j0 + u < p.top_k) v[u] = __ldg(rows[j0 + u] + ch);
#pragma unroll
            for (int u = 0; u < BATCH; ++u) {
                if (j0 + u < p.top_k) {
                    float f[EPC];
                    Vec16<T>::unpack(v[u], f);
                    const float wu = w[j0 + u];
#pragma unroll
                    for (int e = 0; e < EPC; ++e) acc[e] = fmaf(wu, f[e], acc[e]);
                }
            }
        }
        for (int l = 0; l < p.n_layers; ++l) {
            uint4* h = reinterpret_cast<uint4*>(reinterpret_cast<T*>(p.hidden[l]) + t * p.dv) + ch;
            float f[EPC];
            Vec16<T>::unpack(l == 0 ? hv0 : *h, f);
#pragma unroll
            for (int e = 0; e < EPC; ++e) f[e] += acc[e];
            *h = Vec16<T>::pack(f);
        }
    }
}

template <typename T>
__global__ void __launch_bounds__(k4::kThreads) k4_inject(const __grid_constant__ k4::Params p) {
    __shared__ const uint4* rows[LOOKME_MAX_TOP_K];
    __shared__ float w[LOOKME_MAX_TOP_K];
    pdl_trigger();
    pdl_wait();
    const int64_t t = p.sel[blockIdx.x];
    load_rows<T>(p, t, rows, w);
    __syncthreads();
    accumulate_store<T>(p, t, rows, w);
}

// Selection fused into the injection (segments of at most kFusedMaxSegment
// tokens): a CTA takes two consecutive tokens and computes each one's rank in
// its segment,
//   rank_t = #{ j : pi_j > pi_t, or pi_j == pi_t and j < t },
// which orders tokens exactly like the radix selection (larger priority
// first, lower index on ties); a token is kept iff rank_t < r.  The same CTA
// injects its kept tokens.  Every load the ranks and the row addresses need
// is issued before any is used (one L2 round trip for the gate, one HBM round
// trip per kept token), and two tokens per CTA keep the whole grid of a
// 1,024-token call resident at once.
namespace k45 {
constexpr int kThreads = 256;  // one 16-byte chunk of a 2,048-wide bf16 row per thread
constexpr int kTPC = 2;        // tokens per CTA (the code below spells out two)
constexpr int kUnroll = 4;     // priorities in flight per thread and pass
constexpr int kWarps = kThreads / 32;

struct Seg {
    int64_t b, len, r;
};
__device__ __forceinline__ Seg segment_of(const k5::Params& sp, int64_t t) {
    int lo = 0, hi = sp.n_seg;  // segment: off[lo] <= t < off[lo + 1]
    while (hi - lo > 1) {
        const int mid = (lo + hi) / 2;
        if (sp.off[mid] <= t) lo = mid;
        else hi = mid;
    }
    Seg g;
    g.b = sp.off[lo];
    g.len = sp.off[lo + 1] - g.b;
    g.r = (int64_t)floor((double)g.len * sp.keep_ratio);
    return g;
}
}  // namespace k45

template <typename T>
__global__ void __launch_bounds__(k45::kThreads) k45_select_inject(const __grid_constant__ k4::Params p,
                                                                   const __grid_constant__ k5::Params sp) {
    using namespace k45;
    __shared__ int warp_cnt[kTPC][kWarps];
    __shared__ const uint4* rows[kTPC][LOOKME_MAX_TOP_K];
    __shared__ float w[kTPC][LOOKME_MAX_TOP_K];
    pdl_trigger();
    pdl_wait();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    int64_t t[kTPC];
    Seg sg[kTPC];
    bool valid[kTPC], ranked[kTPC];
#pragma unroll
    for (int u = 0; u < kTPC; ++u) {
        t[u] = (int64_t)blockIdx.x * kTPC + u;
        valid[u] = t[u] < p.N;
        sg[u] = segment_of(sp, valid[u] ? t[u] : 0);
        ranked[u] = valid[u] && sg[u].r > 0 && sg[u].r < sg[u].len;
    }
    // Row addresses and weights: threads [64 u, 64 u + top_k) for token u.
    const int u_row = tid / LOOKME_MAX_TOP_K, j_row = tid % LOOKME_MAX_TOP_K;
    const bool row_thread = u_row < kTPC && j_row < p.top_k && (u_row == 0 ? valid[0] : valid[1]);
    int32_t sc = 0, pj = 0;
    float wj = 0.f;
    if (row_thread) {
        const int64_t tr = u_row == 0 ? t[0] : t[1];
        sc = p.scene[tr];
        pj = p.prim[tr * p.top_k + j_row];
        wj = p.weight[tr * p.top_k + j_row];
    }
    // Ranks: one pass over the segment when both tokens share it (the usual
    // case), else one pass per token.
    int cnt[kTPC] = {};
    uint32_t kt[kTPC];
#pragma unroll
    for (int u = 0; u < kTPC; ++u) kt[u] = ranked[u] ? k5::prio_key(sp.priority[t[u]]) : 0u;
    const bool shared_seg = ranked[0] && ranked[1] && sg[0].b == sg[1].b;
#pragma unroll
    for (int u = 0; u < kTPC; ++u) {
        if (!ranked[u] || (u == 1 && shared_seg)) continue;
        const float* pb = sp.priority + sg[u].b;
        const int64_t len = sg[u].len;
        for (int64_t j0 = tid; j0 < len; j0 += kUnroll * kThreads) {
            float v[kUnroll];
#pragma unroll
            for (int q = 0; q < kUnroll; ++q) {
                const int64_t j = j0 + q * kThreads;
                v[q] = j < len ? pb[j] : 0.f;
            }
#pragma unroll
            for (int q = 0; q < kUnroll; ++q) {
                const int64_t j = sg[u].b + j0 + q * kThreads;
                const uint32_t kj = k5::prio_key(v[q]);
                const bool in = j0 + q * kThreads < len;
                cnt[u] += in && ((kj > kt[u]) || (kj == kt[u] && j < t[u]));
                if (u == 0 && shared_seg) cnt[1] += in && ((kj > kt[1]) || (kj == kt[1] && j < t[1]));
            }
        }
    }
#pragma unroll
    for (int u = 0; u < kTPC; ++u) {
#pragma unroll
        for (int o = 16; o; o >>= 1) cnt[u] += __shfl_xor_sync(0xFFFFFFFFu, cnt[u], o);
        if (lane == 0) warp_cnt[u][warp] = cnt[u];
    }
    if (row_thread) {
        const int64_t s = min(max((int64_t)sc, (int64_t)0), p.S - 1);
        const int64_t pr = min(max((int64_t)pj, (int64_t)0), p.P - 1);
        rows[u_row][j_row] = reinterpret_cast<const uint4*>(reinterpret_cast<const T*>(p.values) + (s * p.P + pr) * p.dv);
        w[u_row][j_row] = wj;
    }
    __syncthreads();  // counts, row addresses and weights visible to every thread
#pragma unroll
    for (int u = 0; u < kTPC; ++u) {
        if (!valid[u]) continue;
        bool keep = sg[u].r >= sg[u].len;
        if (ranked[u]) {
            int total = 0;
#pragma unroll
            for (int i = 0; i < kWarps; ++i) total += warp_cnt[u][i];
            keep = total < sg[u].r;
        }
        if (tid == 0 && sp.mask) sp.mask[t[u]] = (uint8_t)keep;
        if (keep) accumulate_store<T>(p, t[u], rows[u], w[u]);
    }
}

cudaError_t launch_select_inject(const LaunchCtx& c, const InjectArgs& a, const float* priority,
                                 const int64_t* seg_off_host, int n_seg, double keep_ratio, uint8_t* mask) {
    if (a.N == 0) return cudaSuccess;
    k4::Params p;
    p.values = a.values;
    p.P = a.P;
    p.dv = a.dv;
    p.top_k = a.top_k;
    p.scene = a.scene;
    p.prim = a.prim;
    p.weight = a.weight;
    p.sel = nullptr;
    p.N = a.N;
    p.S = a.S;
    p.n_layers = a.n_layers;
    for (int l = 0; l < a.n_layers; ++l) p.hidden[l] = a.hidden[l];
    p.status = a.status;
    k5::Params sp;
    sp.priority = priority;
    sp.mask = mask;
    sp.sel = nullptr;
    sp.keep_ratio = keep_ratio;
    sp.n_seg = n_seg;
    for (int i = 0; i <= n_seg; ++i) sp.off[i] = seg_off_host ? seg_off_host[i] : (i == 0 ? 0 : a.N);
    const unsigned grid = (unsigned)((a.N + k45::kTPC - 1) / k45::kTPC);
    if (a.dtype == LOOKME_BF16)
        return launch_pdl(k45_select_inject<__nv_bfloat16>, dim3(grid), dim3(k45::kThreads), 0, c.stream, p, sp);
    return launch_pdl(k45_select_inject<float>, dim3(grid), dim3(k45::kThreads), 0, c.stream, p, sp);
}

// K4 from level-2 records: CTA b injects the token of kept slot b, whose id,
// value rows and weights the level-2 kernel wrote at slot b, so one round trip
// brings everything the value-row and hidden-row loads need.
template <typename T>
__global__ void __launch_bounds__(k4::kThreads) k4_inject_records(const __grid_constant__ k4::Params p,
                                                                   const int32_t* rec_t, const int32_t* rec_row,
                                                                   const float* rec_w) {
    __shared__ const uint4* rows[kRecMaxTopK];
    __shared__ float w[kRecMaxTopK];
    pdl_trigger();
    pdl_wait();
    const int64_t b = blockIdx.x;
    const int64_t t = rec_t[b];  // every thread, together with the rows and weights
    const int j = threadIdx.x;
    if (j < p.top_k) {
        const int64_t r = min(max((int64_t)rec_row[b * p.top_k + j], (int64_t)0), p.S * p.P - 1);
        rows[j] = reinterpret_cast<const uint4*>(reinterpret_cast<const T*>(p.values) + r * p.dv);
        w[j] = rec_w[b * p.top_k + j];
    }
    __syncthreads();
    if (t < 0 || t >= p.N) {  // a slot the level-2 kernel left unwritten: skip it (uniform for the CTA)
        if (threadIdx.x == 0 && p.status) atomicOr(p.status, STATUS_BAD_INDEX);
        return;
    }
    accumulate_store<T>(p, t, rows, w);
}

cudaError_t launch_inject_records(const LaunchCtx& c, const InjectArgs& a, const int32_t* rec_t,
                                  const int32_t* rec_row, const float* rec_w) {
    if (a.n_sel == 0) return cudaSuccess;
    if (a.top_k > kRecMaxTopK) return cudaErrorInvalidValue;
    k4::Params p;
    p.values = a.values;
    p.P = a.P;
    p.dv = a.dv;
    p.top_k = a.top_k;
    p.scene = a.scene;
    p.prim = a.prim;
    p.weight = a.weight;
    p.sel = a.sel;
    p.N = a.N;
    p.S = a.S;
    p.n_layers = a.n_layers;
    for (int l = 0; l < a.n_layers; ++l) p.hidden[l] = a.hidden[l];
    p.status = a.status;
    const int chunks = a.dv / (a.dtype == LOOKME_BF16 ? 8 : 4);
    int threads = (chunks + 31) / 32 * 32;
    if (threads > k4::kThreads) threads = k4::kThreads;
    if (a.dtype == LOOKME_BF16)
        return launch_pdl(k4_inject_records<__nv_bfloat16>, dim3((unsigned)a.n_sel), dim3(threads), 0, c.stream, p,
                          rec_t, rec_row, rec_w);
    return launch_pdl(k4_inject_records<float>, dim3((unsigned)a.n_sel), dim3(threads), 0, c.stream, p, rec_t,
                      rec_row, rec_w);
}

cudaError_t launch_inject(const LaunchCtx& c, const InjectArgs& a) {
    if (a.n_sel == 0) return cudaSuccess;
    k4::Params p;
    p.values = a.values;
    p.P = a.P;
    p.dv = a.dv;
    p.top_k = a.top_k;
    p.scene = a.scene;
    p.prim = a.prim;
    p.weight = a.weight;
    p.sel = a.sel;
    p.N = a.N;
    p.S = a.S;
    p.n_layers = a.n_layers;
    for (int l = 0; l < a.n_layers; ++l) p.hidden[l] = a.hidden[l];
    p.status = a.status;
    // One 16-byte chunk of the row per thread where the row allows it.
    const int chunks = a.dv / (a.dtype == LOOKME_BF16 ? 8 : 4);
    int threads = (chunks + 31) / 32 * 32;
    if (threads > k4::kThreads) threads = k4::kThreads;
    if (a.dtype == LOOKME_BF16)
        return launch_pdl(k4_inject<__nv_bfloat16>, dim3((unsigned)a.n_sel), dim3(threads), 0, c.stream, p);
    return launch_pdl(k4_inject<float>, dim3((unsigned)a.n_sel), dim3(threads), 0, c.stream, p);
}

}  // namespace lookme
