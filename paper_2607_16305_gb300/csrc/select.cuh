// Top-r selection of one segment (the intra-layer gate of Sec. "Sparse
// Injection"): the r = floor(len * keep_ratio) tokens of largest priority are
// kept, ties going to the lower token index.  One CTA of kSelectThreads
// threads finds the r-th largest priority with a 4-pass, 8-bit radix select
// over order-preserving integer keys, keeps every token above it and the
// first tokens equal to it, writes the mask and compacts the kept ids in
// ascending order to sel[sel_base ...].  Used by the selection kernel and by
// the gate CTAs of the bucketing kernel.
#pragma once

#include "common.cuh"

namespace lookme {
namespace sel {
constexpr int kSelectThreads = 1024;
constexpr int kRegKeys = 8;  // keys per thread kept in registers: segments up to 8,192 tokens

// Block-wide exclusive scan of one int (1024 threads).
static __device__ int block_excl_scan(int v, int& total, int* buf) {
    const int lane = threadIdx.x % 32, warp = threadIdx.x / 32;
    int inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int n = __shfl_up_sync(0xFFFFFFFFu, inc, o);
        if (lane >= o) inc += n;
    }
    if (lane == 31) buf[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        const int w = buf[lane];
        int wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int n = __shfl_up_sync(0xFFFFFFFFu, wi, o);
            if (lane >= o) wi += n;
        }
        buf[lane] = wi - w;
        if (lane == 31) buf[32] = wi;
    }
    __syncthreads();
    const int r = buf[warp] + inc - v;
    total = buf[32];
    __syncthreads();
    return r;
}

// Keys read from global memory on every pass (any segment length).
static __device__ __noinline__ void select_segment_global(const float* priority, int64_t b, int64_t len, int64_t r,
                                                   int64_t sel_base, uint8_t* mask, int32_t* sel) {
    constexpr int kThreads = kSelectThreads;
    __shared__ int hist[256];
    __shared__ int scan_buf[33];
    __shared__ uint32_t sh_prefix;
    __shared__ int sh_remaining;
    const int tid = threadIdx.x;

    uint32_t prefix = 0, pmask = 0;
    int remaining = (int)r;
    if (r > 0 && r < len) {
        for (int shift = 24; shift >= 0; shift -= 8) {
            for (int i = tid; i < 256; i += kThreads) hist[i] = 0;
            __syncthreads();
            for (int64_t i = tid; i < len; i += kThreads) {
                const uint32_t k = orderable(priority[b + i]);
                if ((k & pmask) == prefix) atomicAdd(&hist[(k >> shift) & 255u], 1);
            }
            __syncthreads();
            // One warp finds the digit holding the r-th largest key: lane l
            // owns bins 255 - 8 l ... 248 - 8 l (descending), an exclusive
            // prefix over lanes gives the count above each lane's bins.
            if (tid < 32) {
                const int top = 255 - 8 * tid;
                int local = 0;
#pragma unroll
                for (int i = 0; i < 8; ++i) local += hist[top - i];
                int inc = local;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int n = __shfl_up_sync(0xFFFFFFFFu, inc, o);
                    if (tid >= o) inc += n;
                }
                const int excl = inc - local;
                if (excl < remaining && remaining <= inc) {
                    int above = excl, d = top;
                    for (int i = 0; i < 8; ++i) {
                        d = top - i;
                        if (above + hist[d] >= remaining) break;
                        above += hist[d];
                    }
                    sh_prefix = prefix | ((uint32_t)d << shift);
                    sh_remaining = remaining - above;
                }
            }
            __syncthreads();
            prefix = sh_prefix;
            remaining = sh_remaining;
            pmask |= 255u << shift;
            __syncthreads();
        }
    }
    // Keep: key > threshold, or key == threshold among the first `remaining` in token order.
    const uint32_t thr = prefix;
    int eq_seen = 0, kept_seen = 0;
    for (int64_t i0 = 0; i0 < len; i0 += kThreads) {
        const int64_t i = i0 + tid;
        int is_eq = 0, keep = 0;
        if (i < len) {
            if (r >= len) {
                keep = 1;
            } else if (r > 0) {
                const uint32_t k = orderable(priority[b + i]);
                keep = k > thr;
                is_eq = k == thr;
            }
        }
        int eq_total;
        const int eq_rank = block_excl_scan(is_eq, eq_total, scan_buf);
        if (is_eq && eq_seen + eq_rank < remaining) keep = 1;
        int kept_total;
        const int kept_rank = block_excl_scan(keep, kept_total, scan_buf);
        if (i < len) {
            if (mask) mask[b + i] = (uint8_t)keep;
            if (keep) sel[sel_base + kept_seen + kept_rank] = (int32_t)(b + i);
        }
        eq_seen += eq_total;
        kept_seen += kept_total;
    }
}

// Keys held in registers (len <= kSelectThreads * kRegKeys): one read of the
// priorities, the passes work on registers.
static __device__ __noinline__ void select_segment_regs(const float* priority, int64_t b, int64_t len, int64_t r,
                                                 int64_t sel_base, uint8_t* mask, int32_t* sel) {
    constexpr int kThreads = kSelectThreads;
    __shared__ int hist[256];
    __shared__ int scan_buf[33];
    __shared__ uint32_t sh_prefix;
    __shared__ int sh_remaining;
    const int tid = threadIdx.x;
    uint32_t key[kRegKeys];
#pragma unroll
    for (int u = 0; u < kRegKeys; ++u) {
        const int64_t i = (int64_t)u * kThreads + tid;
        key[u] = i < len ? orderable(priority[b + i]) : 0u;
    }
    uint32_t prefix = 0, pmask = 0;
    int remaining = (int)r;
    if (r > 0 && r < len) {
        for (int shift = 24; shift >= 0; shift -= 8) {
            for (int i = tid; i < 256; i += kThreads) hist[i] = 0;
            __syncthreads();
#pragma unroll
            for (int u = 0; u < kRegKeys; ++u) {
                const int64_t i = (int64_t)u * kThreads + tid;
                if (i < len && (key[u] & pmask) == prefix) atomicAdd(&hist[(key[u] >> shift) & 255u], 1);
            }
            __syncthreads();
            if (tid < 32) {
                const int top = 255 - 8 * tid;
                int local = 0;
#pragma unroll
                for (int i = 0; i < 8; ++i) local += hist[top - i];
                int inc = local;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int n = __shfl_up_sync(0xFFFFFFFFu, inc, o);
                    if (tid >= o) inc += n;
                }
                const int excl = inc - local;
                if (excl < remaining && remaining <= inc) {
                    int above = excl, d = top;
                    for (int i = 0; i < 8; ++i) {
                        d = top - i;
                        if (above + hist[d] >= remaining) break;
                        above += hist[d];
                    }
                    sh_prefix = prefix | ((uint32_t)d << shift);
                    sh_remaining = remaining - above;
                }
            }
            __syncthreads();
            prefix = sh_prefix;
            remaining = sh_remaining;
            pmask |= 255u << shift;
            __syncthreads();
        }
    }
    const uint32_t thr = prefix;
    int eq_seen = 0, kept_seen = 0;
#pragma unroll
    for (int u = 0; u < kRegKeys; ++u) {
        const int64_t i0 = (int64_t)u * kThreads;
        if (i0 >= len) break;  // uniform
        const int64_t i = i0 + tid;
        int is_eq = 0, keep = 0;
        if (i < len) {
            if (r >= len) {
                keep = 1;
            } else if (r > 0) {
                keep = key[u] > thr;
                is_eq = key[u] == thr;
            }
        }
        int eq_total;
        const int eq_rank = block_excl_scan(is_eq, eq_total, scan_buf);
        if (is_eq && eq_seen + eq_rank < remaining) keep = 1;
        int kept_total;
        const int kept_rank = block_excl_scan(keep, kept_total, scan_buf);
        if (i < len) {
            if (mask) mask[b + i] = (uint8_t)keep;
            if (keep) sel[sel_base + kept_seen + kept_rank] = (int32_t)(b + i);
        }
        eq_seen += eq_total;
        kept_seen += kept_total;
    }
}

__device__ __forceinline__ void select_segment(const float* priority, int64_t b, int64_t len, int64_t r,
                                               int64_t sel_base, uint8_t* mask, int32_t* sel) {
    if (len <= (int64_t)kSelectThreads * kRegKeys) select_segment_regs(priority, b, len, r, sel_base, mask, sel);
    else select_segment_global(priority, b, len, r, sel_base, mask, sel);
}
}  // namespace sel
}  // namespace lookme
