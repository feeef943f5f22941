// Level-1 scene routing (Sec. "Level-1: scene retrieval"):
//   scene_t = argmax_s ( cos(q_t, e_img[s]) + b_s ).
// With no bias the query norm does not change the argmax, so the kernels
// score q_t . C_s * (1 / ||C_s||); with a bias they also multiply by
// 1 / ||q_t|| and add b_s.  The argmax is fused into the epilogue: each CTA
// reduces its tile to one packed (score, scene) key per token and merges it
// into a per-token 64-bit key with atomicMax, so scores never reach HBM.
#include <cuda.h>

#include <algorithm>

#include "common.cuh"
#include "sm100.cuh"

namespace lookme {

// ------------------------------------------------------------------- K0 prep
// One warp per token: ||q_t||_2 (fp32 accumulation of exact bf16/fp32
// squares) and reset of the token's argmax key.
template <typename T>
__global__ void __launch_bounds__(256) k0_prep(const T* q, int64_t N, int dk,
                                               float* __restrict__ qnorm, float* __restrict__ qnorm_out,
                                               unsigned long long* __restrict__ best) {
    pdl_trigger();
    pdl_wait();
    const int64_t t = (int64_t)blockIdx.x * 8 + threadIdx.x / 32;
    const int lane = threadIdx.x % 32;
    if (t >= N) return;
    const T* row = q + t * dk;
    float acc = 0.f;
    constexpr int EPV = Vec16<T>::N;
    const int nvec = dk / EPV;
    for (int v = lane; v < nvec; v += 32) {
        float f[EPV];
        Vec16<T>::unpack(reinterpret_cast<const uint4*>(row)[v], f);
#pragma unroll
        for (int i = 0; i < EPV; ++i) acc = fmaf(f[i], f[i], acc);
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, o);
    if (lane == 0) {
        const float n = sqrtf(acc);
        qnorm[t] = n;
        if (qnorm_out) qnorm_out[t] = n;
        best[t] = 0ull;
    }
}

cudaError_t launch_prep(const LaunchCtx& c, int dtype, const void* q, int64_t N, int dk, float* qnorm,
                        float* qnorm_out, unsigned long long* best) {
    if (N == 0) return cudaSuccess;
    dim3 grid((unsigned)((N + 7) / 8));
    if (dtype == LOOKME_BF16)
        return launch_pdl(k0_prep<__nv_bfloat16>, grid, dim3(256), 0, c.stream, (const __nv_bfloat16*)q, N, dk, qnorm,
                          qnorm_out, best);
    return launch_pdl(k0_prep<float>, grid, dim3(256), 0, c.stream, (const float*)q, N, dk, qnorm, qnorm_out, best);
}

// Score of token row against scene s from the raw dot product.
__device__ __forceinline__ float level1_score(float dot, float inv_cnorm_s, const float* bias, int64_t s,
                                              float inv_qnorm) {
    float score = dot * inv_cnorm_s;
    if (bias) score = fmaf(score, inv_qnorm, bias[s]);
    return score;
}

// ------------------------------------------------------- K1 on CUDA cores
// 64 x 64 output tile per CTA, 4 x 4 per thread, k-steps of 16.
template <typename T>
__global__ void __launch_bounds__(256) k1_route_simt(const T* q, const T* __restrict__ cent,
                                                     int64_t N, int64_t S, int dk,
                                                     const float* __restrict__ inv_cnorm,
                                                     const float* __restrict__ bias,
                                                     const float* qnorm,
                                                     unsigned long long* __restrict__ best) {
    __shared__ float As[16][64 + 4];
    __shared__ float Bs[16][64 + 4];
    pdl_trigger();
    pdl_wait();
    const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
    const int64_t row0 = (int64_t)blockIdx.y * 64, col0 = (int64_t)blockIdx.x * 64;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

    for (int k0 = 0; k0 < dk; k0 += 16) {
        for (int i = threadIdx.x; i < 64 * 16; i += 256) {
            const int r = i / 16, kk = i % 16, gk = k0 + kk;
            const int64_t gr = row0 + r, gc = col0 + r;
            As[kk][r] = (gr < N && gk < dk) ? to_f32(q[gr * dk + gk]) : 0.f;
            Bs[kk][r] = (gc < S && gk < dk) ? to_f32(cent[gc * dk + gk]) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < 16; ++kk) {
            float a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                a[i] = As[kk][ty * 4 + i];
                b[i] = Bs[kk][tx * 4 + i];
            }
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t r = row0 + ty * 4 + i;
        float inv_q = 1.f;
        if (bias && r < N) {
            const float n = qnorm[r];
            inv_q = n > 0.f ? 1.f / n : 0.f;
        }
        unsigned long long key = 0ull;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int64_t s = col0 + tx * 4 + j;
            if (s < S) {
                const unsigned long long k =
                    pack_argmax(level1_score(acc[i][j], inv_cnorm[s], bias, s, inv_q), (uint32_t)s);
                key = k > key ? k : key;
            }
        }
#pragma unroll
        for (int o = 8; o; o >>= 1) {
            const unsigned long long other = __shfl_xor_sync(0xFFFFFFFFu, key, o);
            key = other > key ? other : key;
        }
        if (tx == 0 && r < N && key) atomicMax(&best[r], key);
    }
}

cudaError_t launch_route_simt(const LaunchCtx& c, int dtype, const void* q, const void* cent, int64_t N,
                              int64_t S, int dk, const float* inv_cnorm, const float* bias, const float* qnorm,
                              unsigned long long* best) {
    if (N == 0) return cudaSuccess;
    dim3 grid((unsigned)((S + 63) / 64), (unsigned)((N + 63) / 64));
    if (dtype == LOOKME_BF16)
        return launch_pdl(k1_route_simt<__nv_bfloat16>, grid, dim3(256), 0, c.stream, (const __nv_bfloat16*)q,
                          (const __nv_bfloat16*)cent, N, S, dk, inv_cnorm, bias, qnorm, best);
    return launch_pdl(k1_route_simt<float>, grid, dim3(256), 0, c.stream, (const float*)q, (const float*)cent, N, S,
                      dk, inv_cnorm, bias, qnorm, best);
}

// ---------------------------------------------------- K1 on tcgen05 (bf16)
// Work units are (128-token tile (MMA M), BN-scene tile (MMA N)) pairs in
// token-tile-major order; CTA b takes the contiguous run of units
// [b u, (b + 1) u), one CTA per SM, so that every SM gets the same number of
// tiles whatever the grid of tiles (a run crosses into the next token tile
// by reloading the token tile once the previous one's MMAs and norm reads
// are done).
//   warp 0      TMA producer: each token tile of the run once (all of d_k),
//               the centroid tiles through a STAGES-deep ring of 64-wide
//               k-blocks
//   warp 1      MMA issuer (one thread): D[buf] = Q_tile * C_tile^T in TMEM,
//               two accumulator buffers so the epilogue of tile i overlaps
//               the MMAs of tile i+1
//   warps 2..9  epilogue: two warps per TMEM lane quarter, each thread one
//               token row (one TMEM lane) and half of the tile's BN columns;
//               it keeps the best (score, scene) of what it read, a strict
//               float compare in increasing scene order (ties keep the lowest
//               scene), and merges it with one atomicMax per row and half
namespace k1tc {
constexpr int BM = 128;
constexpr int BK = 64;              // bf16 elements per 128-byte swizzled row
constexpr int kEpiWarps = 8;  // two per TMEM lane quarter, each half of a tile's columns
constexpr int kThreads = 64 + 32 * kEpiWarps;
constexpr uint64_t kTimeoutNs = 1000000000ull;

__host__ __device__ constexpr int smem_bytes(int BN, int STAGES, int nkb) {
    return 1024 /*alignment slack*/ + nkb * BM * 128 + STAGES * BN * 128 + 256 /*barriers*/ +
           4 * BN * 4 /*per-tile scene constants, double-buffered*/;
}

// Named barrier 1 over the epilogue warps, returning the OR of `v`.
__device__ __forceinline__ bool epi_sync_or(bool v) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.or.pred q, 1, %2, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)v), "n"(32 * kEpiWarps)
        : "memory");
    return r != 0;
}
}  // namespace k1tc

template <int BN, int STAGES>
__global__ void __launch_bounds__(k1tc::kThreads, 1)
    k1_route_tc(const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_c,
                int64_t N, int64_t S, int dk, int units_per_cta, const float* __restrict__ inv_cnorm,
                const float* __restrict__ bias, float* __restrict__ qnorm, float* __restrict__ qnorm_out,
                unsigned long long* __restrict__ best, uint32_t* __restrict__ status) {
    using namespace k1tc;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int nkb = (dk + BK - 1) / BK;
    uint8_t* sA = smem;
    uint8_t* sB = sA + nkb * BM * 128;
    uint64_t* full = reinterpret_cast<uint64_t*>(sB + STAGES * BN * 128);
    uint64_t* empty = full + STAGES;
    uint64_t* a_full = empty + STAGES;
    uint64_t* a_empty = a_full + 1;  // the token tile's MMAs and norm reads are done
    uint64_t* t_full = a_empty + 1;  // [2]
    uint64_t* t_empty = t_full + 2;  // [2]
    uint64_t* drain = t_empty + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
    volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
    // inv ||c_s|| and bias of the current and next scene tile: [2][BN] each.
    float* s_ic = reinterpret_cast<float*>(smem + nkb * BM * 128 + STAGES * BN * 128 + 256);
    float* s_bias = s_ic + 2 * BN;

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int n_tiles = (int)((S + BN - 1) / BN);
    const int64_t n_units = (int64_t)((N + BM - 1) / BM) * n_tiles;
    const int64_t u0 = (int64_t)blockIdx.x * units_per_cta;
    const int64_t u1 = min(n_units, u0 + units_per_cta);

    if (threadIdx.x == 0) {
        ptx::prefetch_tmap(&tmap_q);
        ptx::prefetch_tmap(&tmap_c);
        for (int i = 0; i < STAGES; ++i) {
            ptx::mbar_init(&full[i], 1);
            ptx::mbar_init(&empty[i], 1);
        }
        ptx::mbar_init(a_full, 1);
        ptx::mbar_init(a_empty, 1 + kEpiWarps);  // the MMA issuer's commit and each epilogue warp
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(&t_full[i], 1);
            ptx::mbar_init(&t_empty[i], kEpiWarps);  // one arrival per epilogue warp
        }
        ptx::mbar_init(drain, 1);
        *abort = 0;
        ptx::fence_mbar_init();
    }
    pdl_trigger();
    // TMEM is allocated only after the predecessor has completed, so a CTA
    // that holds TMEM never waits on an earlier kernel.
    pdl_wait();
    if (warp == 1) ptx::tmem_alloc(tmem_slot, 2 * BN);
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0) {
        if (lane == 0 && u0 < u1) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued = 0;      // bit i: ring slot i has been written at least once
            uint32_t last_par = 0;    // bit i: parity of slot i's most recent fill
            int seg = -1;             // token tiles loaded so far - 1
            int64_t m_cur = -1;
            bool ok = true;
            for (int64_t u = u0; u < u1 && ok; ++u) {
                const int64_t m = u / n_tiles;
                const int nt = (int)(u - m * n_tiles);
                if (m != m_cur) {
                    // The previous token tile's MMAs and norm reads are done before it is overwritten.
                    if (seg >= 0 && !(ok = ptx::mbar_wait(a_empty, (uint32_t)(seg & 1), abort, kTimeoutNs))) break;
                    ++seg;
                    m_cur = m;
                    ptx::mbar_arrive_expect_tx(a_full, (uint32_t)(nkb * BM * 128));
                    for (int kb = 0; kb < nkb; ++kb)
                        ptx::tma_load_2d(sA + kb * BM * 128, &tmap_q, kb * BK, (int32_t)(m * BM), a_full);
                }
                for (int kb = 0; kb < nkb; ++kb) {
                    if (!(ok = ptx::mbar_wait(&empty[stage], phase ^ 1u, abort, kTimeoutNs))) break;
                    ptx::mbar_arrive_expect_tx(&full[stage], (uint32_t)(BN * 128));
                    ptx::tma_load_2d(sB + stage * BN * 128, &tmap_c, kb * BK, nt * BN, &full[stage]);
                    issued |= 1u << stage;
                    last_par = (last_par & ~(1u << stage)) | (phase << stage);
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            // Every copy this thread issued must have landed before the CTA exits.
            if (seg >= 0) ptx::mbar_wait_drain(a_full, (uint32_t)(seg & 1), kTimeoutNs);
            for (int i = 0; i < STAGES; ++i)
                if (issued & (1u << i)) ptx::mbar_wait_drain(&full[i], (last_par >> i) & 1u, kTimeoutNs);
        }
    } else if (warp == 1) {
        if (lane == 0 && u0 < u1) {
            constexpr uint32_t idesc = ptx::idesc_bf16_f32<BM, BN>();
            bool ok = true;
            int stage = 0;
            uint32_t phase = 0;
            int seg = -1;
            int64_t m_cur = -1;
            for (int64_t u = u0, it = 0; u < u1 && ok; ++u, ++it) {
                const int64_t m = u / n_tiles;
                if (m != m_cur) {
                    // The previous token tile is free once the MMAs issued so far complete.
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
                    if (!(ok = ptx::mbar_wait(&full[stage], phase, abort, kTimeoutNs))) break;
                    ptx::tc_fence_after();
                    const uint32_t a0 = ptx::smem_u32(sA + kb * BM * 128);
                    const uint32_t b0 = ptx::smem_u32(sB + stage * BN * 128);
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k) {
                        ptx::mma_bf16(d_tmem, ptx::sw128_kmajor_desc(a0 + k * 32), ptx::sw128_kmajor_desc(b0 + k * 32),
                                      idesc, (kb | k) != 0);
                    }
                    ptx::mma_commit(&empty[stage]);
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (ok) ptx::mma_commit(&t_full[buf]);
            }
            // All MMAs must be complete before TMEM is released and the CTA exits.
            ptx::mma_commit(drain);
            ptx::mbar_wait_drain(drain, 0, kTimeoutNs);
        }
    } else {
        // Epilogue warps 2..9: warp w owns TMEM lane quarter (w % 4) * 32 .. + 31
        // and column half (w - 2) / 4 of every tile.
        const int quarter = warp & 3;
        const int half = (warp - 2) / 4;
        constexpr int HC = BN / 2;  // columns per warp and tile
        // Scene constants of the next tile are loaded while this one is scored;
        // columns past S get NaN, which no score compare ever selects.
        const int et = threadIdx.x - 64;  // 0 .. 32 kEpiWarps - 1
        constexpr int ET = 32 * kEpiWarps;
        constexpr int PER = (BN + ET - 1) / ET;
        const float nan = __int_as_float(0x7fc00000);
        float ic_next[PER], b_next[PER];
        auto load_consts = [&](int nt) {
#pragma unroll
            for (int u = 0; u < PER; ++u) {
                const int64_t s = (int64_t)nt * BN + et + u * ET;
                const bool in = et + u * ET < BN && s < S;
                ic_next[u] = in ? __ldg(inv_cnorm + s) : nan;
                b_next[u] = (in && bias) ? __ldg(bias + s) : 0.f;
            }
        };
        auto store_consts = [&](int buf) {
#pragma unroll
            for (int u = 0; u < PER; ++u) {
                if (et + u * ET < BN) {
                    s_ic[buf * BN + et + u * ET] = ic_next[u];
                    s_bias[buf * BN + et + u * ET] = b_next[u];
                }
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
                // The finished token tile's rows, then the new tile's norms: ||q_row||_2
                // from the token tile in shared memory, every 16-byte chunk of the
                // row read once (lane-rotated to avoid bank conflicts; the swizzle
                // only permutes chunks within the row, and zero-filled columns past
                // d_k add nothing).  The unit with scene tile 0 (one CTA) stores it;
                // with a bias every warp needs it.
                if (row >= 0 && row < N && best_s >= 0 && !*abort)
                    atomicMax(&best[row], pack_argmax(best_v, (uint32_t)best_s));
                best_v = -INFINITY;
                best_s = -1;
                ++seg;
                m_cur = m;
                row = m * BM + quarter * 32 + lane;
                const bool ready = ptx::mbar_wait(a_full, (uint32_t)(seg & 1), abort, kTimeoutNs);
                const bool store = nt == 0 && half == 0;
                if (ready && (store || bias)) {
                    float ss = 0.f;
                    const int r = quarter * 32 + lane;
                    for (int kb = 0; kb < nkb; ++kb) {
#pragma unroll
                        for (int c = 0; c < 8; ++c) {
                            float f[8];
                            Vec16<__nv_bfloat16>::unpack(
                                *reinterpret_cast<const uint4*>(sA + kb * BM * 128 + r * 128 + (((c + lane) & 7) * 16)),
                                f);
#pragma unroll
                            for (int i = 0; i < 8; ++i) ss = fmaf(f[i], f[i], ss);
                        }
                    }
                    const float n = sqrtf(ss);
                    if (store && row < N) {
                        qnorm[row] = n;
                        if (qnorm_out) qnorm_out[row] = n;
                    }
                    if (bias) inv_q = n > 0.f ? 1.f / n : 0.f;
                }
                // This warp is done with the token tile.
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(a_empty);
            }
            // Warp-uniform wait (tcgen05.ld below must be executed by the whole
            // warp); the barrier also publishes this tile's constants.
            const bool ready = ptx::mbar_wait(&t_full[buf], use & 1u, abort, kTimeoutNs);
            if (k1tc::epi_sync_or(!__all_sync(0xFFFFFFFFu, ready))) break;
            ptx::tc_fence_after();
            const int c0 = half * HC;
            const float* ic = s_ic + buf * BN + c0;
            const float* bs = s_bias + buf * BN + c0;
            // The best column of this tile's half: strict > in increasing column
            // order keeps the lowest scene among equal scores.
            float tv = -INFINITY;
            int tc = -1;
#pragma unroll 1
            for (int c = 0; c < HC; c += 32) {
                uint32_t r[32];
                ptx::tmem_ld_32x32b_x32(tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(buf * BN + c0 + c),
                                        r);
                ptx::tmem_wait_ld();
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                    float score = __uint_as_float(r[j]) * ic[c + j];
                    if (bias) score = fmaf(score, inv_q, bs[c + j]);
                    if (score > tv) {
                        tv = score;
                        tc = c + j;
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
        if (row >= 0 && row < N && best_s >= 0 && !*abort) atomicMax(&best[row], pack_argmax(best_v, (uint32_t)best_s));
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem_base, 2 * BN);
    }
    if (threadIdx.x == 0 && *abort) atomicOr(status, STATUS_WAIT_TIMEOUT | STATUS_IN_ROUTE);
}

template <int BN, int STAGES>
static cudaError_t launch_route_tc_t(const LaunchCtx& c, const void* tmap_q, const void* tmap_c, int64_t N,
                                     int64_t S, int dk, const float* inv_cnorm, const float* bias, float* qnorm,
                                     float* qnorm_out, unsigned long long* best, uint32_t* status) {
    using namespace k1tc;
    const int nkb = (dk + BK - 1) / BK;
    // Keep TMEM demand per SM within its 512 columns: at most 512 / (2 BN)
    // resident CTAs, enforced through the shared-memory request.
    const int max_resident = 512 / (2 * BN);
    int smem = smem_bytes(BN, STAGES, nkb);
    // (max_resident + 1) CTAs, each with 1 KB of system shared memory, must not fit in 228 KB.
    const int floor_bytes = (228 * 1024) / (max_resident + 1) - 1024 + 1;
    if (smem < floor_bytes) smem = floor_bytes;
    const int64_t m_tiles = (N + BM - 1) / BM;
    const int64_t n_tiles = (S + BN - 1) / BN;
    // One CTA per SM, each a contiguous run of (token tile, scene tile) units.
    const int64_t units = m_tiles * n_tiles;
    int64_t grid = std::min<int64_t>(units, c.num_sms);
    const int64_t per = (units + grid - 1) / grid;
    grid = (units + per - 1) / per;
    CUtensorMap mq, mc;
    memcpy(&mq, tmap_q, sizeof(CUtensorMap));
    memcpy(&mc, tmap_c, sizeof(CUtensorMap));
    return launch_pdl(k1_route_tc<BN, STAGES>, dim3((unsigned)grid), dim3(kThreads), (size_t)smem, c.stream, mq, mc,
                      N, S, dk, (int)per, inv_cnorm, bias, qnorm, qnorm_out, best, status);
}

cudaError_t launch_route_tc(const LaunchCtx& c, const void* tmap_q, const void* const tmap_c[3], int64_t N,
                            int64_t S, int dk, const float* inv_cnorm, const float* bias, float* qnorm,
                            float* qnorm_out, unsigned long long* best, uint32_t* status) {
    if (N == 0) return cudaSuccess;
    if (dk > kRouteTcMaxDk) return cudaErrorInvalidValue;
    const int m_tiles = (int)((N + k1tc::BM - 1) / k1tc::BM);
    // Narrow scene tiles when there are few token tiles, so more CTAs share the work.
    if ((int64_t)m_tiles * ((S + 255) / 256) >= c.num_sms) {
        // Three centroid stages unless the token tile of a wide d_k leaves room for two only.
        if (k1tc::smem_bytes(256, 3, (dk + k1tc::BK - 1) / k1tc::BK) <= 227 * 1024)
            return launch_route_tc_t<256, 3>(c, tmap_q, tmap_c[2], N, S, dk, inv_cnorm, bias, qnorm, qnorm_out, best,
                                              status);
        return launch_route_tc_t<256, 2>(c, tmap_q, tmap_c[2], N, S, dk, inv_cnorm, bias, qnorm, qnorm_out, best,
                                          status);
    }
    if ((int64_t)m_tiles * ((S + 127) / 128) >= c.num_sms)
        return launch_route_tc_t<128, 4>(c, tmap_q, tmap_c[1], N, S, dk, inv_cnorm, bias, qnorm, qnorm_out, best,
                                          status);
    return launch_route_tc_t<64, 4>(c, tmap_q, tmap_c[0], N, S, dk, inv_cnorm, bias, qnorm, qnorm_out, best,
                                          status);
}

cudaError_t configure_route_kernels() {
    cudaError_t e;
    e = cudaFuncSetAttribute(k1_route_tc<256, 3>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(k1_route_tc<256, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(k1_route_tc<128, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(k1_route_tc<64, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
}

// -------------------------------------------------------- load-time kernels
// Centroid = mean of the scene's keys (Sec. "Level-1: scene retrieval",
// first equation), fp32 accumulation, stored in the table dtype.
template <typename T>
__global__ void k_centroid_mean(const T* __restrict__ keys, int64_t n, int64_t P, int dk, T* __restrict__ cent) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n * dk) return;
    const int64_t s = i / dk, d = i % dk;
    float acc = 0.f;
    for (int64_t p = 0; p < P; ++p) acc += to_f32(keys[(s * P + p) * dk + d]);
    const float m = acc / (float)P;
    if constexpr (sizeof(T) == 2)
        cent[i] = __float2bfloat16_rn(m);
    else
        cent[i] = m;
}

cudaError_t launch_centroid_mean(const LaunchCtx& c, int dtype, const void* keys, int64_t n, int64_t P, int dk,
                                 void* cent) {
    const int64_t total = n * dk;
    if (total == 0) return cudaSuccess;
    dim3 grid((unsigned)((total + 255) / 256));
    if (dtype == LOOKME_BF16)
        k_centroid_mean<__nv_bfloat16><<<grid, 256, 0, c.stream>>>((const __nv_bfloat16*)keys, n, P, dk,
                                                                   (__nv_bfloat16*)cent);
    else
        k_centroid_mean<float><<<grid, 256, 0, c.stream>>>((const float*)keys, n, P, dk, (float*)cent);
    return cudaGetLastError();
}

// 1 / ||C_s|| in double, stored as fp32 (0 for a zero centroid).
template <typename T>
__global__ void k_inv_cnorm(const T* __restrict__ cent, int64_t n, int dk, float* __restrict__ out) {
    const int64_t s = (int64_t)blockIdx.x * 8 + threadIdx.x / 32;
    const int lane = threadIdx.x % 32;
    if (s >= n) return;
    double acc = 0.0;
    for (int d = lane; d < dk; d += 32) {
        const double v = (double)to_f32(cent[s * dk + d]);
        acc += v * v;
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, o);
    if (lane == 0) out[s] = acc > 0.0 ? (float)(1.0 / sqrt(acc)) : 0.f;
}

cudaError_t launch_inv_cnorm(const LaunchCtx& c, int dtype, const void* cent, int64_t n, int dk, float* inv_cnorm) {
    if (n == 0) return cudaSuccess;
    dim3 grid((unsigned)((n + 7) / 8));
    if (dtype == LOOKME_BF16)
        k_inv_cnorm<__nv_bfloat16><<<grid, 256, 0, c.stream>>>((const __nv_bfloat16*)cent, n, dk, inv_cnorm);
    else
        k_inv_cnorm<float><<<grid, 256, 0, c.stream>>>((const float*)cent, n, dk, inv_cnorm);
    return cudaGetLastError();
}

}  // namespace lookme
