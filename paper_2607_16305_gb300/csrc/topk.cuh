// Warp-level top-k + softmax of one token's level-2 logits (Sec. "Level-2:
// scene-primitive retrieval": I = top-k of the logits, weights = softmax over
// the selected), shared by the level-2 kernels.
#pragma once

#include "common.cuh"

namespace lookme {
namespace k3 {

// What a lane holds after a top-k: lane j < top_k the j-th selected primitive
// and its softmax weight, other lanes p = -1.
struct TopkLane {
    int p;
    float w;
};

// Inverse of orderable(): the float whose order key is u.
__device__ __forceinline__ float from_orderable(uint32_t u) {
    return __uint_as_float((u & 0x80000000u) ? (u & 0x7FFFFFFFu) : ~u);
}

// Top-k of z[0], z[zs], ..., z[(P-1) zs] by one warp (larger z first, lower
// index on ties) and the
// softmax over the selected logits; writes prim/weight of token t (nothing
// when prim_out is null).
__device__ __forceinline__ TopkLane topk_token(const float* z, int64_t P, int top_k, int lane, int64_t t,
                                           int32_t* prim_out, float* weight_out, int zs = 1) {
    // Each lane keeps the best untaken element of its slice p = lane + 32 i.
    uint64_t taken = 0ull;
    auto local_best = [&](uint32_t& key, uint32_t& pb) {
        key = 0u;
        pb = 0xFFFFFFFFu;
        int i = 0;
        for (int64_t p = lane; p < P; p += 32, ++i) {
            if (!((taken >> i) & 1ull)) {
                const uint32_t k = orderable(z[p * zs]);
                if (pb == 0xFFFFFFFFu || k > key) {
                    key = k;
                    pb = (uint32_t)p;
                }
            }
        }
    };
    uint32_t key, pb;
    local_best(key, pb);
    float my_z[2] = {0.f, 0.f};  // output slots lane and lane + 32
    int my_p[2] = {0, 0};
    for (int kk = 0; kk < top_k; ++kk) {
        const uint32_t kmax = __reduce_max_sync(0xFFFFFFFFu, pb == 0xFFFFFFFFu ? 0u : key);
        const uint32_t pmin = __reduce_min_sync(0xFFFFFFFFu, (pb != 0xFFFFFFFFu && key == kmax) ? pb : 0xFFFFFFFFu);
        if ((kk & 31) == lane) {
            if (kk < 32) {
                my_z[0] = from_orderable(kmax);
                my_p[0] = (int)pmin;
            } else {
                my_z[1] = from_orderable(kmax);
                my_p[1] = (int)pmin;
            }
        }
        if (pmin != 0xFFFFFFFFu && (int)(pmin & 31u) == lane) {
            taken |= 1ull << (pmin >> 5);
            local_best(key, pb);
        }
    }
    const float zmax = __shfl_sync(0xFFFFFFFFu, my_z[0], 0);
    float e[2];
    float sum = 0.f;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        e[h] = (h * 32 + lane < top_k) ? expf(my_z[h] - zmax) : 0.f;
        sum += e[h];
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int j = h * 32 + lane;
        if (j < top_k && prim_out) {
            prim_out[t * top_k + j] = my_p[h];
            weight_out[t * top_k + j] = e[h] / sum;
        }
    }
    return lane < top_k ? TopkLane{my_p[0], e[0] / sum} : TopkLane{-1, 0.f};
}
// Register-resident variant for N_p <= 32 * PPL: each lane holds the order
// keys of its elements p = 32 i + lane, so a round is an unrolled scan of
// PPL registers plus two warp reductions.  Same result as topk_token.
template <int PPL>
__device__ __forceinline__ TopkLane topk_token_regs(const float* z, int64_t P, int top_k, int lane, int64_t t,
                                                int32_t* prim_out, float* weight_out, int zs = 1) {
    uint32_t key[PPL];
#pragma unroll
    for (int i = 0; i < PPL; ++i) {
        const int64_t p = (int64_t)i * 32 + lane;
        key[i] = p < P ? max(orderable(z[p * zs]), 1u) : 0u;  // 0 marks "no element"
    }
    uint32_t taken = 0u;
    float my_z[2] = {0.f, 0.f};
    int my_p[2] = {0, 0};
    for (int kk = 0; kk < top_k; ++kk) {
        uint32_t bk = 0u;
        int bi = -1;
#pragma unroll
        for (int i = 0; i < PPL; ++i) {
            if (!((taken >> i) & 1u) && key[i] > bk) {  // strict: the lowest i (lowest p) wins ties
                bk = key[i];
                bi = i;
            }
        }
        const uint32_t kmax = __reduce_max_sync(0xFFFFFFFFu, bk);
        const uint32_t pmin = __reduce_min_sync(0xFFFFFFFFu, (bi >= 0 && bk == kmax) ? (uint32_t)(bi * 32 + lane)
                                                                                     : 0xFFFFFFFFu);
        if (pmin != 0xFFFFFFFFu && (int)(pmin & 31u) == lane) taken |= 1u << (pmin >> 5);
        if ((kk & 31) == lane) {
            const float zz = pmin != 0xFFFFFFFFu ? z[(int64_t)pmin * zs] : 0.f;
            if (kk < 32) {
                my_z[0] = zz;
                my_p[0] = (int)pmin;
            } else {
                my_z[1] = zz;
                my_p[1] = (int)pmin;
            }
        }
    }
    const float zmax = __shfl_sync(0xFFFFFFFFu, my_z[0], 0);
    float e[2];
    float sum = 0.f;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        e[h] = (h * 32 + lane < top_k) ? expf(my_z[h] - zmax) : 0.f;
        sum += e[h];
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int j = h * 32 + lane;
        if (j < top_k && prim_out) {
            prim_out[t * top_k + j] = my_p[h];
            weight_out[t * top_k + j] = e[h] / sum;
        }
    }
    return lane < top_k ? TopkLane{my_p[0], e[0] / sum} : TopkLane{-1, 0.f};
}

// Sorted-list variant for top_k <= L (L = 8 or 16), N_p <= 32 * PPL.  An
// element is the 64-bit key (order key of z) << 32 | (2^32 - 1 - p): a larger
// key is a larger z, then a lower index, the order the variants above use.
// Each lane first sorts its own elements (bitonic networks, no cross-lane
// traffic) and keeps its best L in descending order; then each of the top_k
// rounds takes the warp's largest head (two warp reductions: value, then the
// lowest index among equal values) and the winning lane drops its head.  A
// round is a handful of dependent instructions around the two reductions,
// instead of a rescan of every element.
template <int L>
__device__ __forceinline__ void cas_desc(uint64_t (&a)[L], int i, int l) {
    const uint64_t x = a[i], y = a[l];
    a[i] = x > y ? x : y;
    a[l] = x > y ? y : x;
}
// a bitonic -> sorted in descending order.
template <int L>
__device__ __forceinline__ void bitonic_merge_desc(uint64_t (&a)[L]) {
#pragma unroll
    for (int j = L / 2; j > 0; j >>= 1) {
#pragma unroll
        for (int i = 0; i < L; ++i)
            if ((i ^ j) > i) cas_desc<L>(a, i, i ^ j);
    }
}
template <int L>
__device__ __forceinline__ void bitonic_sort_desc(uint64_t (&a)[L]) {
#pragma unroll
    for (int k = 2; k <= L; k <<= 1) {
#pragma unroll
        for (int j = k / 2; j > 0; j >>= 1) {
#pragma unroll
            for (int i = 0; i < L; ++i) {
                const int l = i ^ j;
                if (l > i) {
                    if ((i & k) == 0) cas_desc<L>(a, i, l);
                    else cas_desc<L>(a, l, i);
                }
            }
        }
    }
}
// a = top L of a and b (both sorted descending), sorted descending.
template <int L>
__device__ __forceinline__ void merge_top_desc(uint64_t (&a)[L], const uint64_t (&b)[L]) {
#pragma unroll
    for (int i = 0; i < L; ++i) a[i] = a[i] > b[L - 1 - i] ? a[i] : b[L - 1 - i];
    bitonic_merge_desc<L>(a);
}

template <int PPL, int L>
__device__ __forceinline__ TopkLane topk_token_pop(const float* z, int64_t P, int top_k, int lane, int64_t t,
                                               int32_t* prim_out, float* weight_out, int zs = 1) {
    constexpr int G = (PPL + L - 1) / L;  // groups of L elements per lane
    uint64_t a[L];
#pragma unroll
    for (int g = 0; g < G; ++g) {
        uint64_t b[L];
#pragma unroll
        for (int u = 0; u < L; ++u) {
            const int i = g * L + u;
            const int p = i * 32 + lane;
            b[u] = (i < PPL && p < P)
                       ? ((uint64_t)max(orderable(z[(int64_t)p * zs]), 1u) << 32) | (uint64_t)(0xFFFFFFFFu - (uint32_t)p)
                       : 0ull;
        }
        bitonic_sort_desc<L>(b);
        if (g == 0) {
#pragma unroll
            for (int u = 0; u < L; ++u) a[u] = b[u];
        } else {
            merge_top_desc<L>(a, b);
        }
    }
    uint32_t my_key = 0u, my_p = 0u;
    for (int kk = 0; kk < top_k; ++kk) {
        const uint32_t h = (uint32_t)(a[0] >> 32);
        const uint32_t kmax = __reduce_max_sync(0xFFFFFFFFu, h);
        const uint32_t pmin =
            __reduce_min_sync(0xFFFFFFFFu, (h == kmax && h != 0u) ? 0xFFFFFFFFu - (uint32_t)a[0] : 0xFFFFFFFFu);
        if (lane == kk) {
            my_key = kmax;
            my_p = pmin;
        }
        if (lane == (int)(pmin & 31u)) {  // the owner of the winner drops its head
#pragma unroll
            for (int u = 0; u + 1 < L; ++u) a[u] = a[u + 1];
            a[L - 1] = 0ull;
        }
    }
    // Softmax over the selected logits; lane j < top_k holds the j-th largest.
    const float zmax = from_orderable(__shfl_sync(0xFFFFFFFFu, my_key, 0));
    const float e = lane < top_k ? expf(from_orderable(my_key) - zmax) : 0.f;
    float sum = e;
#pragma unroll
    for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
    if (lane < top_k && prim_out) {
        prim_out[t * top_k + lane] = (int32_t)my_p;
        weight_out[t * top_k + lane] = e / sum;
    }
    return lane < top_k ? TopkLane{(int)my_p, e / sum} : TopkLane{-1, 0.f};
}

// Top-k of one token, picking the register-resident variant when N_p allows.
__device__ __forceinline__ TopkLane topk_any(const float* z, int64_t P, int top_k, int lane, int64_t t,
                                         int32_t* prim_out, float* weight_out, int zs = 1) {
    if (top_k <= 8) {
        if (P <= 64) return topk_token_pop<2, 8>(z, P, top_k, lane, t, prim_out, weight_out, zs);
        else if (P <= 256) return topk_token_pop<8, 8>(z, P, top_k, lane, t, prim_out, weight_out, zs);
        else if (P <= 512) return topk_token_pop<16, 8>(z, P, top_k, lane, t, prim_out, weight_out, zs);
        else if (P <= 1024) return topk_token_pop<32, 8>(z, P, top_k, lane, t, prim_out, weight_out, zs);
        return topk_token(z, P, top_k, lane, t, prim_out, weight_out, zs);
    }
    if (top_k <= 16 && P <= 1024) {
        if (P <= 512) return topk_token_pop<16, 16>(z, P, top_k, lane, t, prim_out, weight_out, zs);
        return topk_token_pop<32, 16>(z, P, top_k, lane, t, prim_out, weight_out, zs);
    }
    if (P <= 32) return topk_token_regs<1>(z, P, top_k, lane, t, prim_out, weight_out, zs);
    if (P <= 64) return topk_token_regs<2>(z, P, top_k, lane, t, prim_out, weight_out, zs);
    if (P <= 128) return topk_token_regs<4>(z, P, top_k, lane, t, prim_out, weight_out, zs);
    if (P <= 256) return topk_token_regs<8>(z, P, top_k, lane, t, prim_out, weight_out, zs);
    if (P <= 512) return topk_token_regs<16>(z, P, top_k, lane, t, prim_out, weight_out, zs);
    if (P <= 1024) return topk_token_regs<32>(z, P, top_k, lane, t, prim_out, weight_out, zs);
    return topk_token(z, P, top_k, lane, t, prim_out, weight_out, zs);
}

}  // namespace k3
}  // namespace lookme
