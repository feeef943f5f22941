// Dense bf16 GEMM on the 5th-generation tensor cores, for the dense pieces
// around the lookup: the ranker MLP of the paper's level 2 (Sec. "Level-2:
// scene-primitive retrieval"), the projection into the embedding space (Sec.
// "Level-1", W_{v->e}), the SwiGLU-style fusion f and the propagation
// R W_p + R (Sec. "Sparse Injection"), and the router projection of the
// multi-scale retrieval (Sec. "Multi-scale image retrieval").
//
// D[M][Nn] = A[M][K] B[Nn][K]^T: A and B are row-major bf16 (B in the
// [out][in] layout of a linear layer's weight), so both are K-major operands.
// One CTA per 128 x BN output tile: a TMA producer warp streams 64-wide
// k-blocks of A and B (128-byte swizzle) through a ring; one thread issues
// tcgen05.mma (kind::f16, fp32 accumulation) into BN TMEM columns; four
// epilogue warps (one per 32-lane TMEM quarter, i.e. 32 rows) read the tile
// back 32 columns at a time and apply the epilogue.  Every mbarrier wait is
// bounded; a timeout sets the status word, drains what is in flight, frees
// TMEM and returns.
#include <cuda.h>

#include <algorithm>
#include <atomic>
#include <cstring>

#include "common.cuh"
#include "sm100.cuh"

namespace lookme {

namespace kg {
constexpr int BM = 128;
constexpr int BK = 64;
constexpr int kThreads = 192;  // producer, MMA issuer, four epilogue warps
constexpr uint64_t kTimeoutNs = 1000000000ull;

__host__ __device__ constexpr int stages_for(int BN) { return BN >= 256 ? 4 : BN >= 128 ? 5 : 6; }
__host__ __device__ constexpr int smem_bytes(int BN) {
    return 1024 /*alignment slack*/ + stages_for(BN) * (BM + BN) * 128 + 256 /*barriers*/;
}

__device__ __forceinline__ float silu(float x) { return x / (1.f + __expf(-x)); }

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t*>(&h);
}
}  // namespace kg

template <int BN>
__global__ void __launch_bounds__(kg::kThreads, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap tmap_a, const __grid_constant__ CUtensorMap tmap_b,
              const __grid_constant__ GemmArgs g) {
    using namespace kg;
    constexpr int STAGES = stages_for(BN);
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sA = smem;                              // [STAGES][BM rows][128 B]
    uint8_t* sB = sA + STAGES * BM * 128;            // [STAGES][BN rows][128 B]
    uint64_t* full = reinterpret_cast<uint64_t*>(sB + STAGES * BN * 128);
    uint64_t* empty = full + STAGES;
    uint64_t* done = empty + STAGES;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
    volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int64_t m0 = (int64_t)blockIdx.y * BM, n0 = (int64_t)blockIdx.x * BN;
    const int nkb = (int)((g.K + BK - 1) / BK);

    if (threadIdx.x == 0) {
        ptx::prefetch_tmap(&tmap_a);
        ptx::prefetch_tmap(&tmap_b);
        for (int i = 0; i < STAGES; ++i) {
            ptx::mbar_init(&full[i], 1);
            ptx::mbar_init(&empty[i], 1);
        }
        ptx::mbar_init(done, 1);
        *abort = 0;
        ptx::fence_mbar_init();
    }
    pdl_trigger();
    // TMEM only after the predecessor has completed (a CTA holding TMEM never
    // waits on an earlier kernel).
    pdl_wait();
    if (warp == 1) ptx::tmem_alloc(tmem_slot, BN);
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0, issued = 0, last_par = 0;
            for (int kb = 0; kb < nkb; ++kb) {
                if (!ptx::mbar_wait(&empty[stage], phase ^ 1u, abort, kTimeoutNs)) break;
                ptx::mbar_arrive_expect_tx(&full[stage], (uint32_t)((BM + BN) * 128));
                ptx::tma_load_2d(sA + stage * BM * 128, &tmap_a, kb * BK, (int32_t)m0, &full[stage]);
                ptx::tma_load_2d(sB + stage * BN * 128, &tmap_b, kb * BK, (int32_t)n0, &full[stage]);
                issued |= 1u << stage;
                last_par = (last_par & ~(1u << stage)) | (phase << stage);
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            // Every copy issued must land before the CTA exits.
            for (int i = 0; i < STAGES; ++i)
                if (issued & (1u << i)) ptx::mbar_wait_drain(&full[i], (last_par >> i) & 1u, kTimeoutNs);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = ptx::idesc_bf16_f32<BM, BN>();
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            for (int kb = 0; kb < nkb && ok; ++kb) {
                if (!(ok = ptx::mbar_wait(&full[stage], phase, abort, kTimeoutNs))) break;
                ptx::tc_fence_after();
                const uint32_t a0 = ptx::smem_u32(sA + stage * BM * 128);
                const uint32_t b0 = ptx::smem_u32(sB + stage * BN * 128);
#pragma unroll
                for (int k = 0; k < BK / 16; ++k)
                    ptx::mma_bf16(tmem_base, ptx::sw128_kmajor_desc(a0 + k * 32), ptx::sw128_kmajor_desc(b0 + k * 32),
                                  idesc, (kb | k) != 0);
                ptx::mma_commit(&empty[stage]);
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            // `done` completes when every MMA issued has completed (also on abort).
            ptx::mma_commit(done);
            if (!ok) ptx::mbar_wait_drain(done, 0, kTimeoutNs);
        }
    } else {
        // Epilogue: warp w reads TMEM lane quarter (w & 3), i.e. rows 32 (w & 3) ..
        const int quarter = warp & 3;
        const int64_t m = m0 + quarter * 32 + lane;
        const bool ready = ptx::mbar_wait(done, 0, abort, kTimeoutNs);
        if (__all_sync(0xFFFFFFFFu, ready) && !*abort) {
            ptx::tc_fence_after();
            const uint32_t row_taddr = tmem_base + ((uint32_t)(quarter * 32) << 16);
            const bool row_ok = m < g.M;
            const float* rb = (g.rowbias && row_ok) ? g.rowbias + (int64_t)g.rowsel[m] * g.ld_rowbias : nullptr;
            if (g.mode == EPI_SWIGLU) {
                // Columns [64 j, 64 j + 32) are gate features, [64 j + 32, 64 j + 64) the matching up features.
#pragma unroll 1
                for (int c = 0; c < BN; c += 64) {
                    uint32_t ga[32], up[32];
                    ptx::tmem_ld_32x32b_x32(row_taddr + (uint32_t)c, ga);
                    ptx::tmem_ld_32x32b_x32(row_taddr + (uint32_t)(c + 32), up);
                    ptx::tmem_wait_ld();
                    const int64_t nout = (n0 + c) / 2;  // first output feature of this pair of chunks
                    if (!row_ok || n0 + c >= g.Nn) continue;
                    __nv_bfloat16* o = reinterpret_cast<__nv_bfloat16*>(g.out) + m * g.ld_out + nout;
                    const int64_t nf = std::min<int64_t>(32, g.Nn / 2 - nout);
                    if (nf == 32) {
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            uint4 v;
                            uint32_t* w = reinterpret_cast<uint32_t*>(&v);
#pragma unroll
                            for (int e = 0; e < 4; ++e) {
                                const int j = q * 8 + 2 * e;
                                const float a0 = __uint_as_float(ga[j]) + (g.colbias ? g.colbias[n0 + c + j] : 0.f);
                                const float a1 = __uint_as_float(ga[j + 1]) + (g.colbias ? g.colbias[n0 + c + j + 1] : 0.f);
                                const float u0 = __uint_as_float(up[j]) + (g.colbias ? g.colbias[n0 + c + 32 + j] : 0.f);
                                const float u1 = __uint_as_float(up[j + 1]) + (g.colbias ? g.colbias[n0 + c + 33 + j] : 0.f);
                                w[e] = kg::pack_bf16(kg::silu(a0) * u0, kg::silu(a1) * u1);
                            }
                            reinterpret_cast<uint4*>(o)[q] = v;
                        }
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j) {
                            if (j < nf) {
                                const float a = __uint_as_float(ga[j]) + (g.colbias ? g.colbias[n0 + c + j] : 0.f);
                                const float u = __uint_as_float(up[j]) + (g.colbias ? g.colbias[n0 + c + 32 + j] : 0.f);
                                o[j] = __float2bfloat16_rn(kg::silu(a) * u);
                            }
                        }
                    }
                }
            } else {
#pragma unroll 1
                for (int c = 0; c < BN; c += 32) {
                    uint32_t r[32];
                    ptx::tmem_ld_32x32b_x32(row_taddr + (uint32_t)c, r);
                    ptx::tmem_wait_ld();
                    const int64_t n = n0 + c;
                    if (!row_ok || n >= g.Nn) continue;
                    const int nv = (int)std::min<int64_t>(32, g.Nn - n);
                    float v[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        float x = __uint_as_float(r[j]);
                        if (j < nv) {
                            if (g.colbias) x += g.colbias[n + j];
                            if (rb) x += rb[n + j];
                        }
                        v[j] = x;
                    }
                    if (g.mode == EPI_F32) {
                        float* o = reinterpret_cast<float*>(g.out) + m * g.ld_out + n;
                        if (nv == 32) {
#pragma unroll
                            for (int q = 0; q < 8; ++q)
                                reinterpret_cast<float4*>(o)[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
                        } else {
#pragma unroll
                            for (int j = 0; j < 32; ++j)
                                if (j < nv) o[j] = v[j];
                        }
                        continue;
                    }
                    // bf16 outputs
                    __nv_bfloat16* o;
                    if (g.mode == EPI_SCATTER_ADD) {
                        o = reinterpret_cast<__nv_bfloat16*>(g.out) + (int64_t)g.rowidx[m] * g.ld_out + n;
                    } else {
                        o = reinterpret_cast<__nv_bfloat16*>(g.out) + m * g.ld_out + n;
                    }
                    const __nv_bfloat16* add = nullptr;
                    if (g.mode == EPI_RESID) add = reinterpret_cast<const __nv_bfloat16*>(g.resid) + m * g.ld_resid + n;
                    if (g.mode == EPI_SCATTER_ADD) add = o;
                    if (nv == 32) {
                        uint4 a4[4];
                        if (add) {
#pragma unroll
                            for (int q = 0; q < 4; ++q) a4[q] = reinterpret_cast<const uint4*>(add)[q];
                        }
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            uint4 w4;
                            uint32_t* w = reinterpret_cast<uint32_t*>(&w4);
                            const __nv_bfloat162* ad = reinterpret_cast<const __nv_bfloat162*>(&a4[q]);
#pragma unroll
                            for (int e = 0; e < 4; ++e) {
                                float x0 = v[q * 8 + 2 * e], x1 = v[q * 8 + 2 * e + 1];
                                if (g.mode == EPI_BF16 && g.act == 1) {
                                    x0 = kg::silu(x0);
                                    x1 = kg::silu(x1);
                                }
                                if (add) {
                                    const float2 f = __bfloat1622float2(ad[e]);
                                    x0 += f.x;
                                    x1 += f.y;
                                }
                                w[e] = kg::pack_bf16(x0, x1);
                            }
                            reinterpret_cast<uint4*>(o)[q] = w4;
                        }
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j) {
                            if (j < nv) {
                                float x = v[j];
                                if (g.mode == EPI_BF16 && g.act == 1) x = kg::silu(x);
                                if (add) x += __bfloat162float(add[j]);
                                o[j] = __float2bfloat16_rn(x);
                            }
                        }
                    }
                }
            }
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem_base, BN);
    }
    if (threadIdx.x == 0 && *abort && g.status) atomicOr(g.status, STATUS_WAIT_TIMEOUT | STATUS_IN_GEMM);
}

int gemm_tile_n(int64_t M, int64_t Nn, int num_sms) {
    const int64_t mt = (M + kg::BM - 1) / kg::BM;
    if (mt * ((Nn + 255) / 256) >= num_sms) return 256;
    if (mt * ((Nn + 127) / 128) >= num_sms) return 128;
    return 64;
}

cudaError_t launch_gemm_tc(const LaunchCtx& c, const void* tmap_a, const void* tmap_b, int bn, const GemmArgs& g) {
    if (g.M == 0 || g.Nn == 0) return cudaSuccess;
    // The shared-memory opt-in, once per device (callers without a table never ran it).
    static std::atomic<uint64_t> configured{0};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const uint64_t bit = 1ull << (dev & 63);
    if (!(configured.load() & bit)) {
        if ((e = configure_gemm_kernels()) != cudaSuccess) return e;
        configured.fetch_or(bit);
    }
    CUtensorMap ma, mb;
    memcpy(&ma, tmap_a, sizeof(CUtensorMap));
    memcpy(&mb, tmap_b, sizeof(CUtensorMap));
    const dim3 grid((unsigned)((g.Nn + bn - 1) / bn), (unsigned)((g.M + kg::BM - 1) / kg::BM));
    switch (bn) {
        case 64:
            return launch_pdl(k_gemm_tc<64>, grid, dim3(kg::kThreads), (size_t)kg::smem_bytes(64), c.stream, ma, mb, g);
        case 128:
            return launch_pdl(k_gemm_tc<128>, grid, dim3(kg::kThreads), (size_t)kg::smem_bytes(128), c.stream, ma, mb,
                              g);
        case 256:
            return launch_pdl(k_gemm_tc<256>, grid, dim3(kg::kThreads), (size_t)kg::smem_bytes(256), c.stream, ma, mb,
                              g);
        default:
            return cudaErrorInvalidValue;
    }
}

cudaError_t configure_gemm_kernels() {
    cudaError_t e = cudaFuncSetAttribute(k_gemm_tc<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, kg::smem_bytes(64));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_gemm_tc<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, kg::smem_bytes(128));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_gemm_tc<256>, cudaFuncAttributeMaxDynamicSharedMemorySize, kg::smem_bytes(256));
    return e;
}

}  // namespace lookme
