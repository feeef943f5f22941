// Pieces of the tcgen05 level-2 scoring (Sec. "Level-2: scene-primitive
// retrieval") shared by the level-2 kernel and the fused step kernel: the
// shared-memory geometry of the key ring, the MMA descriptors of the
// token-atom x key-tile product, the k-block MMA issue, the top-k variant
// choice and the L2 row prefetch.
#pragma once

#include <algorithm>

#include "common.cuh"
#include "sm100.cuh"
#include "topk.cuh"

namespace lookme {

namespace k3tc {
constexpr int BK = 64;                   // bf16 elements per 128-byte swizzled row
constexpr int kSubRows = 128;            // key rows per sub-block
constexpr int kNTile = 256;              // key rows per MMA (N)
constexpr int kTok = kTokensPerItem;     // token rows of the A atom
constexpr int kSubBytes = kSubRows * 128;  // one 128 x 64 key sub-block: 16 KiB
constexpr int kAtomBytes = 1024;         // 8 token rows x 128 bytes per k-block
constexpr int kZStride = 9;              // logits z[p][j] at p * 9 + j: conflict-free both ways
constexpr int kGroupWarps = 8;           // epilogue warps per item group (one token each)
constexpr int kEpiWarps = 2 * kGroupWarps;
constexpr int kBuildWarp = 2 + kEpiWarps;
constexpr int kThreads = (3 + kEpiWarps) * 32;
constexpr int kMaxStages = 14;           // ring slots (barrier arrays)
constexpr int kBSlots = 3;               // token tiles
constexpr int kISlots = 4;               // item metadata (scene, count, token ids)
constexpr int kSeq = 4;                  // item indices passed from the producer to the token-tile warp
constexpr uint64_t kTimeoutNs = 1000000000ull;
constexpr int kSmemLimit = 227 * 1024;

struct Geometry {
    int nkb;              // 64-wide k-blocks of d_k
    int ntile;            // 128-row sub-block rows of N_p
    int nnt;              // N-tiles (256 rows; the last may hold one sub-block)
    int spi;              // sub-blocks per item (ntile x nkb)
    int group;            // sub-blocks per ring slot (one bulk copy): 4, 2 or 1
    int gshift;           // log2(group)
    int slot_bytes;       // group x 16 KiB
    int n_stages;         // ring slots
    int chunks;           // bulk copies per item
    int row_bytes;        // d_k * 2
    int b_bytes;          // one token tile (nkb x 1 KiB)
    int tmem_cols;        // two D buffers
    int zbytes;           // logits of one item (per epilogue group)
    int off_b, off_z, off_bar, off_meta;
    int smem;             // bytes requested, including 1 KiB of alignment slack
};

inline Geometry geometry(int64_t P, int dk) {
    Geometry g;
    g.nkb = (dk + BK - 1) / BK;
    g.ntile = (int)((P + kSubRows - 1) / kSubRows);
    g.nnt = (g.ntile + 1) / 2;
    g.spi = g.ntile * g.nkb;
    g.row_bytes = dk * 2;
    g.b_bytes = g.nkb * kAtomBytes;
    const int nmax = (int)std::min<int64_t>(kNTile, (P + 15) / 16 * 16);
    int cols = 32;
    while (cols < 2 * nmax) cols <<= 1;
    g.tmem_cols = cols;
    g.zbytes = ((int)P * kZStride * 4 + 15) / 16 * 16;  // per epilogue group
    const int fixed = kBSlots * g.b_bytes + 2 * g.zbytes + 1024 /*bar+meta*/ + 1024 /*align*/;
    // The largest copies that leave at least two ring slots; a two-sub-block
    // N-tile unit must fit in one slot, and units start at even sub-blocks.
    g.gshift = 2;
    while (g.gshift > 0 && (kSmemLimit - fixed) / ((kSubBytes << g.gshift)) < 2) --g.gshift;
    while (g.gshift > 0 && (1 << g.gshift) > g.spi) --g.gshift;
    g.group = 1 << g.gshift;
    g.slot_bytes = g.group * kSubBytes;
    g.chunks = (g.spi + g.group - 1) / g.group;
    g.n_stages = (kSmemLimit - fixed) / g.slot_bytes;
    if (g.n_stages > kMaxStages) g.n_stages = kMaxStages;
    g.off_b = g.n_stages * g.slot_bytes;
    g.off_z = g.off_b + kBSlots * g.b_bytes;
    g.off_bar = g.off_z + 2 * g.zbytes;
    g.off_meta = g.off_bar + (2 * kMaxStages + 2 * kBSlots + 2 * kISlots + 4 + 2 + 1 + 2 + 2 * kSeq) * 8;
    g.smem = g.off_meta + kISlots * ((int)sizeof(WorkItem) + kTok * 4 + 4) + 16 + kSeq * 4 + kISlots * kTok * 4 + 1024;
    return g;
}

// Named barrier 1 + grp over one epilogue group, returning the OR of `v` over it.
template <int ID>
__device__ __forceinline__ bool bar_or(bool v) {
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
__device__ __forceinline__ bool group_sync_or(int grp, bool v) { return grp == 0 ? bar_or<1>(v) : bar_or<2>(v); }

// Shared-memory descriptor of a K-major, 128-byte-swizzled operand whose
// 8-row atoms are `sbo` bytes apart (0: every atom is the same 1 KiB).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr, uint32_t sbo) {
    return (ptx::sw128_kmajor_desc(saddr) & ~(0x3FFFull << 32)) | ((uint64_t)(sbo >> 4) << 32);
}

// Instruction descriptor of kind::f16, bf16 A and B, fp32 D, M = 128, N = n.
__device__ __forceinline__ uint32_t idesc_m128(int n) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
}

// The four k-steps of one 64-wide k-block of an N-tile.  live = 0 runs the
// same instructions with every MMA switched off (the warm-up call); one copy
// of the code serves both.
static __device__ __noinline__ void mma_kblock(uint32_t live, uint32_t d, uint64_t ad, uint64_t bd, uint32_t idesc,
                                        uint32_t first) {
#pragma unroll
    for (int k = 0; k < BK / 16; ++k)
        ptx::mma_bf16_if(live, d, ad + (uint64_t)(k * 2), bd + (uint64_t)(k * 2), idesc,
                         (first && k == 0) ? 0u : 1u);
}

// Top-k + softmax of one token over logits at stride kZStride; a single copy
// serves the warm-up call (prim_out == nullptr: nothing is written) and the
// real ones.  Each variant is a function of its own, so that no variant's
// registers weigh on another (one function holding them all spills).
// Each returns the lane's selected primitive and its weight (lanes < top_k, first 32).
template <int PPL, int L>
__device__ __noinline__ k3::TopkLane topk_pop_fn(const float* z, int64_t P, int top_k, int lane, int64_t t, int32_t* prim_out,
                                        float* weight_out) {
    return k3::topk_token_pop<PPL, L>(z, P, top_k, lane, t, prim_out, weight_out, kZStride);
}
template <int PPL>
__device__ __noinline__ k3::TopkLane topk_regs_fn(const float* z, int64_t P, int top_k, int lane, int64_t t,
                                         int32_t* prim_out, float* weight_out) {
    return k3::topk_token_regs<PPL>(z, P, top_k, lane, t, prim_out, weight_out, kZStride);
}
static __device__ __noinline__ k3::TopkLane topk_scan_fn(const float* z, int64_t P, int top_k, int lane, int64_t t, int32_t* prim_out,
                                         float* weight_out) {
    return k3::topk_token(z, P, top_k, lane, t, prim_out, weight_out, kZStride);
}
// The variant choice of k3::topk_any.
__device__ __forceinline__ k3::TopkLane topk_item(const float* z, int64_t P, int top_k, int lane, int64_t t,
                                         int32_t* prim_out, float* weight_out) {
    if (top_k <= 8) {
        if (P <= 64) return topk_pop_fn<2, 8>(z, P, top_k, lane, t, prim_out, weight_out);
        if (P <= 256) return topk_pop_fn<8, 8>(z, P, top_k, lane, t, prim_out, weight_out);
        if (P <= 512) return topk_pop_fn<16, 8>(z, P, top_k, lane, t, prim_out, weight_out);
        if (P <= 1024) return topk_pop_fn<32, 8>(z, P, top_k, lane, t, prim_out, weight_out);
        return topk_scan_fn(z, P, top_k, lane, t, prim_out, weight_out);
    }
    if (top_k <= 16 && P <= 1024) {
        if (P <= 512) return topk_pop_fn<16, 16>(z, P, top_k, lane, t, prim_out, weight_out);
        return topk_pop_fn<32, 16>(z, P, top_k, lane, t, prim_out, weight_out);
    }
    if (P <= 32) return topk_regs_fn<1>(z, P, top_k, lane, t, prim_out, weight_out);
    if (P <= 64) return topk_regs_fn<2>(z, P, top_k, lane, t, prim_out, weight_out);
    if (P <= 128) return topk_regs_fn<4>(z, P, top_k, lane, t, prim_out, weight_out);
    if (P <= 256) return topk_regs_fn<8>(z, P, top_k, lane, t, prim_out, weight_out);
    if (P <= 512) return topk_regs_fn<16>(z, P, top_k, lane, t, prim_out, weight_out);
    if (P <= 1024) return topk_regs_fn<32>(z, P, top_k, lane, t, prim_out, weight_out);
    return topk_scan_fn(z, P, top_k, lane, t, prim_out, weight_out);
}

// Pull one value row into L2 (128-byte lines, no register result).
__device__ __forceinline__ void prefetch_row_l2(const uint8_t* row, int64_t bytes) {
    for (int64_t o = 0; o < bytes; o += 128) asm volatile("prefetch.global.L2 [%0];" ::"l"(row + o));
}

}  // namespace k3tc

}  // namespace lookme
