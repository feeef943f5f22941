// Level 2 on the 5th-generation tensor cores (bf16 tables), Sec. "Level-2:
// scene-primitive retrieval" in its key-similarity form:
//   z_tp = q_t . K[j, p] / sqrt(d_k), I_t = top-k of z_t, w_t = softmax(z_t[I_t]).
//
// Each work item (a scene and <= 8 of its tokens) is a small grouped GEMM:
// D[j][p] = q_j . K[scene, p, :] for the item's tokens and the scene's N_p
// key rows.  The keys are the N operand, up to 256 rows per MMA (an "N-tile"),
// because a tcgen05.mma costs about the same time whatever its N: with the
// keys as N = 256 each MMA consumes 8 KiB of keys, twice what the 128-row M
// operand would.  The tokens are the M = 128 operand: one 1 KiB swizzled
// atom of 8 token rows per 64-wide k-block, with the descriptor's atom stride
// set to zero so that every 8-row group of M reads the same atom (D row r is
// token r % 8).  The fp32 accumulator D lives in TMEM, two buffers of 256
// columns.
//
// The table stores every scene's keys as the exact shared-memory image the
// MMA reads: 128-row x 64-column sub-blocks (16 KiB, 128-byte swizzle),
// ordered N-tile, then k-block, then the N-tile's one or two sub-blocks
// (which are adjacent, so an N = 256 operand is one contiguous 32 KiB), and
// zero-padded past N_p and d_k.  A scene's block is contiguous and is
// streamed with 1-D bulk copies of up to four sub-blocks: the copy engine of
// an SM spends about the same time on a 16 KiB and a 64 KiB copy, so large
// copies are what lets one CTA per SM pull its share of HBM bandwidth.
//
// One CTA per SM.  CTA b's first item is work entry b; the entries from G on
// are taken one at a time from a shared counter as CTAs progress (one item
// ahead), so the CTAs that run ahead take the last items:
//   warp 0       producer: takes the item indices, passes them to warp 18,
//                reads each item's work entry and streams the scene's key
//                block through the ring (bulk copies only)
//   warp 1       one thread issues tcgen05.mma, N-tile by N-tile, into the
//                two TMEM buffers
//   warps 2..17  epilogue, two groups of eight taking alternate items (so one
//                item's top-k overlaps the next item's read-out): TMEM ->
//                logits in shared memory (scaled), then top-k + softmax, one
//                token per warp
//   warp 18      token tiles: reads the item's token ids and copies its query
//                rows with 16-byte cp.async straight into the swizzled tile,
//                all of them in flight at once (bulk copies of a row would
//                each cost the copy engine as much time as a 64 KiB one)
// Before the grid dependency wait, the MMA issuer and the second epilogue
// group's top-k run once without effect, so their code is cached before the
// key stream starts (a first instruction fetch under the full stream costs
// microseconds; after an L2 flush the warm-up takes about 10 us).  The first
// group skips it: it reads out the CTA's first item as soon as its products
// are done, so the D buffers are not all held until the warm-up ends.
// Every wait is bounded; on a timeout the kernel drains its copies and MMAs,
// releases TMEM and reports through the status word.
#include <cuda.h>

#include <algorithm>

#include "score_tc.cuh"

namespace lookme {

__global__ void __launch_bounds__(k3tc::kThreads, 1)
    k3_score_tc(const uint8_t* __restrict__ keys_t, int64_t block_bytes, const __nv_bfloat16* q,
                int64_t P, int dk, int top_k, float scale, const WorkItem* work,
                int32_t* counters, const int32_t* item_tok, int64_t work_cap, int use_slots,
                int32_t* __restrict__ prim_out, float* __restrict__ weight_out, uint32_t* __restrict__ status,
                const int32_t* selpos, const uint8_t* __restrict__ values, int64_t vrow_bytes,
                const uint8_t* hidden0, int32_t* __restrict__ rec_t, int32_t* __restrict__ rec_row,
                float* __restrict__ rec_w,
                const __grid_constant__ k3tc::Geometry g) {
    using namespace k3tc;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* ring = smem;
    uint8_t* btile = smem + g.off_b;
    float* zs = reinterpret_cast<float*>(smem + g.off_z);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + g.off_bar);
    uint64_t* empty = full + kMaxStages;
    uint64_t* bfull = empty + kMaxStages;
    uint64_t* bempty = bfull + kBSlots;
    uint64_t* ifull = bempty + kBSlots;
    uint64_t* iempty = ifull + kISlots;
    // D buffer b ready for epilogue group q: dready[2 q + b].  Each group waits
    // only on its own pair, in the order the MMA commits to it, so no waiter is
    // ever two phases behind a barrier (the two groups share both buffers when
    // an item has several N-tiles).
    uint64_t* dready = iempty + kISlots;
    uint64_t* tempty = dready + 4;
    uint64_t* drain = tempty + 2;
    uint64_t* setup = drain + 1;      // the other barriers are initialised (thread 0)
    uint64_t* tmem_ready = setup + 1; // the TMEM address is in tmem_slot (warp 1)
    // Item j >= 1 of the CTA (item 0 is entry b) is queue entry j - 1: its index
    // is in seq[(j - 1) % kSeq], phase (j - 1) / kSeq of seqfull / seqempty.
    uint64_t* seqfull = tmem_ready + 1;
    uint64_t* seqempty = seqfull + kSeq;
    WorkItem* items = reinterpret_cast<WorkItem*>(smem + g.off_meta);
    int32_t* toks = reinterpret_cast<int32_t*>(items + kISlots);
    uint32_t* keepbits = reinterpret_cast<uint32_t*>(toks + kISlots * kTok);  // gate of the item's tokens
    uint32_t* tmem_slot = keepbits + kISlots;
    volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
    int32_t* seq = reinterpret_cast<int32_t*>(tmem_slot + 4);  // item indices; -1 ends the list
    int32_t* tpos = seq + kSeq;  // the item's tokens' kept-list slots (-1: not kept)

    const int tid = threadIdx.x, lane = tid % 32, warp = tid / 32;
    pdl_trigger();
    // Two hand-off barriers first, so that after the dependency wait no role
    // waits for another role's warm-up: only for what it actually needs.
    if (tid == 0) {
        ptx::mbar_init(setup, 1);
        ptx::mbar_init(tmem_ready, 1);
        *abort = 0;
        ptx::fence_mbar_init();
    }
    __syncthreads();
    // Warm-up while the predecessor finishes: no memory, barrier or TMEM effect
    // (the top-k in the second epilogue group only).
    if (warp == 1 && lane == 0) {
        mma_kblock(0u, 0u, 0ull, 0ull, idesc_m128(kNTile), 1u);
    } else if (warp >= 2 + kGroupWarps && warp < kBuildWarp) {
        topk_item(zs, P, top_k, lane, 0, nullptr, nullptr);
    }
    // The work list is the predecessor's output (read with plain loads: a
    // read-only/restrict qualifier would let the compiler move them above the
    // wait); TMEM is allocated only after it, so a CTA that holds TMEM never
    // waits on an earlier kernel.
    pdl_wait();
    // This CTA's first work entry, and the token-tile warp's first token ids,
    // are read together with the count (the work array holds work_cap
    // entries, the token array kTok per entry), saving dependent round trips;
    // the token ids are used only for lanes below the entry's count.
    WorkItem w0;
    w0.scene = w0.begin = w0.count = w0.slot = 0;
    int32_t tok0 = 0;
    if ((int64_t)blockIdx.x < work_cap) {
        w0 = work[blockIdx.x];
        if (warp == kBuildWarp && lane < kTok) tok0 = item_tok[(int64_t)blockIdx.x * kTok + lane];
    }
    const int n_work = counters[0];
    const int G = gridDim.x;
    // Item 0 of CTA b is work entry b; the entries from G on are taken one at
    // a time from a shared counter (reset by the bucketing kernel) as the CTA
    // progresses, so CTAs that run ahead take more of the last items.
    if (n_work <= (int)blockIdx.x) return;  // uniform for the CTA: nothing allocated yet
    if (tid == 0) {
        for (int i = 0; i < g.n_stages; ++i) {
            ptx::mbar_init(&full[i], 1);
            ptx::mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < kBSlots; ++i) {
            ptx::mbar_init(&bfull[i], 1);
            ptx::mbar_init(&bempty[i], 1);
        }
        for (int i = 0; i < kISlots; ++i) {
            ptx::mbar_init(&ifull[i], 1);
            ptx::mbar_init(&iempty[i], kGroupWarps);
        }
        for (int i = 0; i < 4; ++i) ptx::mbar_init(&dready[i], 1);
        for (int i = 0; i < 2; ++i) ptx::mbar_init(&tempty[i], kGroupWarps);
        for (int i = 0; i < kSeq; ++i) {
            ptx::mbar_init(&seqfull[i], 1);
            ptx::mbar_init(&seqempty[i], 1);
        }
        ptx::mbar_init(drain, 1);
        ptx::fence_mbar_init();
        ptx::mbar_arrive(setup);
    }
    // N-tile nt: its first sub-block, its sub-block count (1 or 2) and its N.
    auto nt_base = [&](int nt) { return nt * 2 * g.nkb; };
    auto nt_subs = [&](int nt) { return (nt == g.nnt - 1 && (g.ntile & 1)) ? 1 : 2; };
    auto nt_cols = [&](int nt) {
        const int64_t rows = P - (int64_t)nt * kNTile;
        return (int)(rows >= kNTile ? kNTile : (rows + 15) / 16 * 16);
    };
    // The producer (thread 0 initialised the barriers) starts the key stream
    // at once; the others wait for the barriers, and the MMA issuer and the
    // epilogue for the TMEM address, which warp 1 publishes.
    uint32_t tmem_base = 0;
    if (warp != 0 && warp != kBuildWarp) ptx::mbar_wait(setup, 0, abort, kTimeoutNs);
    if (warp == 1) {
        ptx::tmem_alloc(tmem_slot, g.tmem_cols);
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(tmem_ready);
    }
    if (warp >= 1 && warp < kBuildWarp) {
        ptx::mbar_wait(tmem_ready, 0, abort, kTimeoutNs);
        ptx::tc_fence_after();
        tmem_base = *tmem_slot;
    }

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        int64_t stage_seq = 0;  // copies issued
        int slot = 0;
        uint32_t phase = 0;
        bool ok = true;
        // Key blocks are read once per call: evict them first from L2, so the
        // small per-token buffers the injection re-reads stay cached.
        const uint64_t policy = ptx::l2_policy_evict_first();
        // Issues bulk copies [from, to) of item w's key block through the ring;
        // copy c holds sub-blocks [c * group, min(spi, (c + 1) * group)).
        auto issue_stages = [&](const WorkItem& w, int from, int to) {
            const uint8_t* blk = keys_t + (use_slots ? (int64_t)w.slot : (int64_t)w.scene) * block_bytes;
            for (int c = from; c < to && ok; ++c, ++stage_seq) {
                const uint32_t bytes = (uint32_t)(min(g.group, g.spi - c * g.group) * kSubBytes);
                if (lane == 0) {
                    ok = ptx::mbar_wait(&empty[slot], phase ^ 1u, abort, kTimeoutNs);
                    if (ok) {
                        ptx::mbar_arrive_expect_tx(&full[slot], bytes);
                        ptx::bulk_g2s_hint(ring + (int64_t)slot * g.slot_bytes, blk + (int64_t)c * g.slot_bytes,
                                           bytes, &full[slot], policy);
                    }
                }
                ok = __shfl_sync(0xFFFFFFFFu, (int)ok, 0) != 0;
                if (++slot == g.n_stages) {
                    slot = 0;
                    phase ^= 1u;
                }
            }
        };
        // Item i + 1's index is taken as item i's first copy goes out and passed
        // to the token-tile warp through seq (-1: no more items) before the
        // item's other copies, which may wait for ring slots that only item i's
        // token tile frees; its work entry is read before item i + 1's first copy.
        WorkItem w = w0, w_next = w0;
        for (int i = 0; ok; ++i) {
            int taken = 0;
            if (lane == 0) taken = G + atomicAdd(counters + 3, 1);
            issue_stages(w, 0, 1);
            int nxt = -1;
            if (lane == 0 && ok) {
                nxt = taken < n_work ? taken : -1;
                const int qs = i % kSeq;  // item i + 1: queue entry i
                ok = ptx::mbar_wait(&seqempty[qs], ((i / kSeq) & 1) ^ 1, abort, kTimeoutNs);
                if (ok) {
                    seq[qs] = nxt;
                    ptx::mbar_arrive(&seqfull[qs]);
                }
            }
            ok = __shfl_sync(0xFFFFFFFFu, (int)ok, 0) != 0;
            nxt = __shfl_sync(0xFFFFFFFFu, nxt, 0);
            if (ok && nxt >= 0) w_next = work[nxt];
            issue_stages(w, 1, g.chunks);
            if (!ok || nxt < 0) break;
            w = w_next;
        }
        if (!ok && lane == 0) {
            // Let every copy still in flight land before the CTA can exit.
            for (int64_t s = stage_seq - g.n_stages; s < stage_seq; ++s)
                if (s >= 0) ptx::mbar_wait_drain(&full[s % g.n_stages], (uint32_t)((s / g.n_stages) & 1), kTimeoutNs);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------- MMA
        if (lane == 0) {
            const uint32_t a_tiles = ptx::smem_u32(btile);
            int slot = 0;
            uint32_t phase = 0;
            int qn = 0;  // N-tiles issued (D buffer qn & 1)
            bool ok = true;
            for (int i = 0; ok; ++i) {
                const int bs = i % kBSlots;
                if (!(ok = ptx::mbar_wait(&bfull[bs], (i / kBSlots) & 1, abort, kTimeoutNs))) break;
                if (items[i % kISlots].count < 0) break;  // the end of the CTA's list
                ptx::tc_fence_after();
                const uint64_t ad0 = sw128_desc(a_tiles + (uint32_t)(bs * g.b_bytes), 0);
                int cur_chunk = -1;
                for (int nt = 0; nt < g.nnt && ok; ++nt, ++qn) {
                    const int buf = qn & 1;
                    if (!(ok = ptx::mbar_wait(&tempty[buf], ((qn >> 1) & 1) ^ 1, abort, kTimeoutNs))) break;
                    ptx::tc_fence_after();
                    const uint32_t d = tmem_base + (uint32_t)(buf * (g.tmem_cols >> 1));
                    const uint32_t idesc = idesc_m128(nt_cols(nt));
                    const int ns = nt_subs(nt);
                    for (int kb = 0; kb < g.nkb; ++kb) {
                        const int sb = nt_base(nt) + kb * ns;
                        const int ch = sb >> g.gshift;
                        if (ch != cur_chunk) {
                            if (cur_chunk >= 0) {
                                ptx::mma_commit(&empty[slot]);
                                if (++slot == g.n_stages) {
                                    slot = 0;
                                    phase ^= 1u;
                                }
                            }
                            if (!(ok = ptx::mbar_wait(&full[slot], phase, abort, kTimeoutNs))) break;
                            ptx::tc_fence_after();
                            cur_chunk = ch;
                        }
                        const uint32_t b_addr = ptx::smem_u32(ring + (int64_t)slot * g.slot_bytes +
                                                              (int64_t)(sb - (ch << g.gshift)) * kSubBytes);
                        mma_kblock(1u, d, ad0 + (uint64_t)(kb * (kAtomBytes >> 4)), sw128_desc(b_addr, 1024), idesc,
                                   kb == 0 ? 1u : 0u);
                    }
                    if (ok) ptx::mma_commit(&dready[(i & 1) * 2 + buf]);
                }
                if (!ok) break;
                // The item's last copy and its token tile are free once these MMAs complete.
                ptx::mma_commit(&empty[slot]);
                if (++slot == g.n_stages) {
                    slot = 0;
                    phase ^= 1u;
                }
                ptx::mma_commit(&bempty[bs]);
            }
            // All MMAs complete before TMEM is released and the CTA exits.
            ptx::mma_commit(drain);
            ptx::mbar_wait_drain(drain, 0, kTimeoutNs);
        }
    } else if (warp < kBuildWarp) {
        // -------------------------------------------------------- epilogue
        const int e = warp - 2;
        const int grp = e / kGroupWarps;  // takes items grp, grp + 2, ...
        const int eg = e % kGroupWarps;   // token of the top-k, column slice of the read-out
        const int quarter = warp & 3;     // TMEM lanes this warp may access
        float* zg = zs + grp * (g.zbytes / 4);
        for (int i = grp;; i += 2) {
            const int ms = i % kISlots;
            bool ok = __all_sync(0xFFFFFFFFu, ptx::mbar_wait(&ifull[ms], (i / kISlots) & 1, abort, kTimeoutNs));
            // Also orders this item's logit writes after the group's top-k of its previous item.
            if (k3tc::group_sync_or(grp, !ok || *abort)) break;
            if (items[ms].count < 0) break;  // the end of the CTA's list (uniform)
            const int nb = min(items[ms].count, kTok);
            for (int nt = 0; nt < g.nnt; ++nt) {
                const int qn = i * g.nnt + nt, buf = qn & 1;
                // Earlier N-tiles of this group on buffer buf: per earlier item of the
                // group, those nt' with the same buffer; in this item, every second nt' < nt.
                const int m = i >> 1;
                const int per_item = (g.nnt & 1) ? (g.nnt + (((buf ^ grp) & 1) ? -1 : 1)) / 2 : g.nnt / 2;
                const uint32_t par = (uint32_t)(m * per_item + (nt >> 1)) & 1u;
                ok = __all_sync(0xFFFFFFFFu, ptx::mbar_wait(&dready[grp * 2 + buf], par, abort, kTimeoutNs));
                const int ncols = nt_cols(nt);
                // Warp eg reads columns [32 eg, 32 eg + 32) of its lanes; lane j < 8 of any
                // quarter holds token j (D row r is token r % 8).
                const int c0 = eg * 32;
                if (ok && c0 < ncols) {
                    ptx::tc_fence_after();
                    const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16) +
                                           (uint32_t)(buf * (g.tmem_cols >> 1) + c0);
                    const int64_t p0 = (int64_t)nt * kNTile + c0;
                    if (c0 + 32 <= ncols) {  // one load and one wait for the warp's 32 columns
                        uint32_t r[32];
                        ptx::tmem_ld_32x32b_x32(taddr, r);
                        ptx::tmem_wait_ld();
                        if (lane < nb) {
#pragma unroll
                            for (int j = 0; j < 32; ++j)
                                if (p0 + j < P) zg[(p0 + j) * kZStride + lane] = __uint_as_float(r[j]) * scale;
                        }
                    } else {  // 16 columns (N is a multiple of 16)
                        uint32_t r[16];
                        ptx::tmem_ld_32x32b_x16(taddr, r);
                        ptx::tmem_wait_ld();
                        if (lane < nb) {
#pragma unroll
                            for (int j = 0; j < 16; ++j)
                                if (p0 + j < P) zg[(p0 + j) * kZStride + lane] = __uint_as_float(r[j]) * scale;
                        }
                    }
                }
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(&tempty[buf]);
            }
            if (k3tc::group_sync_or(grp, *abort)) break;  // all logits of the item are in shared memory
            if (eg < nb) {
                const int64_t t = toks[ms * kTok + eg];
                const k3::TopkLane r = k3tc::topk_item(zg + eg, P, top_k, lane, t, prim_out, weight_out);
                if ((keepbits[ms] >> eg) & 1u) {
                    // A kept token: its record for the injection kernel, and its value
                    // rows and hidden row (read by that kernel next) into L2 now.
                    const int64_t row = (int64_t)items[ms].scene * P + r.p;
                    if (rec_t) {
                        const int pos = tpos[ms * kTok + eg];
                        if (pos < 0) {  // a kept token without a kept-list slot: skip its record
                            if (lane == 0) atomicOr(status, STATUS_BAD_INDEX);
                        } else {
                            if (lane < top_k) {
                                rec_row[(int64_t)pos * top_k + lane] = (int32_t)row;
                                rec_w[(int64_t)pos * top_k + lane] = r.w;
                            }
                            if (lane == 0) rec_t[pos] = (int32_t)t;
                        }
                    }
                    if (r.p >= 0) k3tc::prefetch_row_l2(values + row * vrow_bytes, vrow_bytes);
                    if (hidden0 && lane == 0) k3tc::prefetch_row_l2(hidden0 + t * vrow_bytes, vrow_bytes);
                }
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&iempty[ms]);
        }
    } else {
        // ---------------------------------------------------- token tiles
        // Both tiles start zeroed; columns past d_k are never written again.
        for (int idx = lane; idx < kBSlots * g.b_bytes / 16; idx += 32)
            reinterpret_cast<uint4*>(btile)[idx] = make_uint4(0u, 0u, 0u, 0u);
        const int cpr = g.row_bytes / 16;  // 16-byte chunks per query row
        const uint8_t* qb = reinterpret_cast<const uint8_t*>(q);
        const uint32_t bt0 = ptx::smem_u32(btile);
        WorkItem w = w0;
        int32_t tok = lane < w.count ? tok0 : 0;
        int32_t kpos = (selpos && lane < w.count) ? selpos[tok] : -1;
        bool ok = true;
        // The items until the producer's -1, then two end markers (count -1):
        // one for each epilogue group, the first also read by the MMA issuer.
        int ends = 0;
        for (int i = 0; ends < 2; ++i) {
            const int ms = i % kISlots, bs = i % kBSlots;
            // The first item's slots are free by construction: its query rows are
            // loaded before this warp touches any barrier (and before the key
            // stream fills the memory system).
            if (lane == 0 && i > 0)
                ok = ptx::mbar_wait(&iempty[ms], ((i / kISlots) & 1) ^ 1, abort, kTimeoutNs) &&
                     ptx::mbar_wait(&bempty[bs], ((i / kBSlots) & 1) ^ 1, abort, kTimeoutNs);
            if (!__shfl_sync(0xFFFFFFFFu, (int)ok, 0)) break;
            if (w.count < 0) {
                if (lane == 0) {
                    items[ms] = w;
                    ptx::mbar_arrive(&ifull[ms]);
                    if (ends == 0) ptx::mbar_arrive(&bfull[bs]);
                }
                ++ends;
                continue;
            }
            const int nb = min(w.count, kTok);
            const int total = nb * cpr;
            const uint32_t bt = bt0 + (uint32_t)(bs * g.b_bytes);
            // Every query chunk of the item in flight at once, straight into the
            // swizzled tile: row j of k-block kb, 16-byte chunk c at position c ^ j.
            for (int base = 0; base < total; base += 32) {
                const int idx = base + lane;
                const int j = idx / cpr, cc = idx - j * cpr;
                const int32_t tj = __shfl_sync(0xFFFFFFFFu, tok, j & (kTok - 1));
                if (idx < total) {
                    const int kb = cc >> 3, c = cc & 7;
                    ptx::cp_async16(bt + (uint32_t)(kb * kAtomBytes + j * 128 + ((c ^ j) * 16)),
                                    qb + (int64_t)tj * g.row_bytes + cc * 16);
                }
            }
            // The next item's index (queue entry i, which the producer publishes as
            // item i's first copy goes out), its work entry and token ids: read
            // while the rows are in flight when the index is already there, else
            // once this item is published (this item never waits for the next).
            const int qs = i % kSeq;
            WorkItem wn;
            wn.scene = wn.begin = wn.slot = 0;
            wn.count = -1;
            int32_t tokn = 0;
            bool have = false;
            auto take_next = [&](bool block) {
                int nidx = -1, got = 0;
                if (lane == 0) {
                    got = block ? ptx::mbar_wait(&seqfull[qs], (i / kSeq) & 1, abort, kTimeoutNs)
                                : ptx::mbar_try_wait(&seqfull[qs], (i / kSeq) & 1);
                    if (got) {
                        nidx = seq[qs];
                        ptx::mbar_arrive(&seqempty[qs]);
                        if (nidx >= n_work) {  // not an index the producer can take: stop the CTA
                            *abort = 1;
                            got = 0;
                            nidx = -1;
                        }
                    }
                }
                got = __shfl_sync(0xFFFFFFFFu, got, 0);
                nidx = __shfl_sync(0xFFFFFFFFu, nidx, 0);
                if (got && nidx >= 0) {
                    wn = work[nidx];
                    if (lane < kTok) tokn = item_tok[(int64_t)nidx * kTok + lane];
                }
                return got != 0;
            };
            // The queue barriers are thread 0's to initialise: none is touched
            // before it has published them.
            if (i == 0 && !__all_sync(0xFFFFFFFFu, ptx::mbar_wait(setup, 0, abort, kTimeoutNs))) break;
            have = take_next(false);
            ptx::cp_async_wait_all();
            ptx::fence_proxy_async_smem();  // the tile is read by the tensor core (async proxy)
            if (lane < nb) toks[ms * kTok + lane] = tok;
            const uint32_t kbits = __ballot_sync(0xFFFFFFFFu, kpos >= 0);
            if (lane < nb) tpos[ms * kTok + lane] = kpos;
            if (lane == 0) {
                items[ms] = w;
                keepbits[ms] = kbits;
            }
            __syncwarp();
            if (lane == 0) {
                ptx::mbar_arrive(&ifull[ms]);
                ptx::mbar_arrive(&bfull[bs]);
            }
            if (!have && !take_next(true)) break;
            w = wn;
            tok = lane < w.count ? tokn : 0;
            kpos = (selpos && lane < w.count) ? selpos[tok] : -1;
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem_base, g.tmem_cols);
    }
    if (tid == 0 && *abort) atomicOr(status, STATUS_WAIT_TIMEOUT | STATUS_IN_SCORE);
}

bool score_tc_shape_supported(int64_t P, int dk) {
    const k3tc::Geometry g = k3tc::geometry(P, dk);
    return g.n_stages >= 2 && g.smem <= k3tc::kSmemLimit && g.tmem_cols <= 512 && (dk % 8) == 0 &&
           (g.ntile < 2 || g.group >= 2);
}

int64_t score_tc_block_bytes(int64_t P, int dk) {
    const k3tc::Geometry g = k3tc::geometry(P, dk);
    return (int64_t)g.spi * k3tc::kSubBytes;
}

cudaError_t launch_score_tc(const LaunchCtx& c, const void* keys_tiled, const ScoreArgs& a) {
    const k3tc::Geometry g = k3tc::geometry(a.P, a.dk);
    if (!score_tc_shape_supported(a.P, a.dk)) return cudaErrorInvalidConfiguration;
    return launch_pdl(k3_score_tc, dim3(c.num_sms), dim3(k3tc::kThreads), (size_t)g.smem, c.stream,
                      (const uint8_t*)keys_tiled, (int64_t)g.spi * k3tc::kSubBytes, (const __nv_bfloat16*)a.q, a.P,
                      a.dk, a.top_k, a.scale, a.work, a.counters, a.item_tok, a.work_cap, a.use_slots, a.prim_out,
                      a.weight_out, a.status, a.selpos, (const uint8_t*)a.values, a.vrow_bytes,
                      (const uint8_t*)a.hidden0, a.rec_t, a.rec_row, a.rec_w, g);
}

cudaError_t configure_score_tc_kernel() {
    return cudaFuncSetAttribute(k3_score_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, k3tc::kSmemLimit);
}

}  // namespace lookme
