// Eq. 1 window scores and the Section 4.2 importance I (before pooling), from
// the window queries' attention over the candidate tokens, recomputed on the
// tensor cores with the softmax statistics (m_r, Z_r) of the score kernel.
//
// Work unit: (sequence s, 128-token tile of candidates, group of up to 8 KV
// heads); the candidates are [0, L - w), or [0, L) when every position
// competes.  An item is one KV head h of a unit: S^T = K_tile Q_h^T on
// tcgen05.mma (M = 128 tokens, N = g*w query rows padded to 16, K = d) into a
// TMEM accumulator, so one epilogue thread owns one token and every query row
// of it:
//   A[r][t]   = 2^(s_rt * scale * log2(e) - m_r) / Z_r   (softmax over all visible keys)
//   G_h[q][t] = sum_j A[(q, j)][t]                       (GQA group sum, r = q * g + j)
//   P_O[h,t]  = (1/O)  sum_{q >= w-O}  G_h[q][t]
//   P_O'[h,t] = (1/O') sum_{q >= w-O'} G_h[q][t]
//   I[t]      = (1/O)  sum_{q >= w-O}  max_h G_h[q][t]
// The grid is persistent: a CTA walks units blockIdx.x, blockIdx.x + gridDim.x,
// ... and the items of its units in order.  Warp 0 streams K_h and Q_h with
// TMA into a ring of stages, warp 1 issues the MMAs into A accumulators (4 of
// N <= 128 columns, or 2 of N <= 256), and the epilogue is A groups of four
// warps (one per TMEM lane quadrant): group a takes the CTA's items a, a + A,
// ..., each thread all the query rows of its token, so every group streams
// through its own accumulator without waiting for the others.  The head maxima
// of G_h[q][t] meet in shared memory through atomicMax on the float bits
// (values are >= +0, so the integer order is the float order and the result
// does not depend on the order of the updates); the last group to finish a
// unit sums them into I (or, with several head groups per tile, writes them to
// a partial buffer that the heads kernel combines).  The raw rows go to the
// slot arrays; pooling happens in the heads kernel.
#include <cudaTypedefs.h>

#include "kvec_internal.cuh"
#include "sm100_ptx.cuh"

namespace kvec {

namespace {

constexpr int kWinThreads = 576;                      // warp 0 TMA, warp 1 MMA, warps 2..17 epilogue
constexpr int kMaxSmemWin = 232448;                   // opt-in shared memory per CTA on sm_103
constexpr int kKTileBytes = kTileT * kHeadDim * 2;    // 32 KB: two 64-column swizzled halves
constexpr int kMaxStages = 3;                         // deepest operand ring
constexpr int kWinReserveSms = 8;                     // SMs a window launch leaves to the other kernels

struct WinArgs {
    Geometry G;
    Scratch sc;
    Slot sl;
    const int* cu;                  // device cu_seqlens
    int Npad;                       // query rows padded to a multiple of 16 (MMA N)
    int kst;                        // operand stages
    int nacc;                       // accumulators = epilogue groups (4, or 2 when N > 128)
    int units;                      // (sequence, candidate tile, head group) units of the launch
    uint32_t tmem_cols;
    int fault;                      // test of the error path (kvec_set_test_fault): the first
                                    // accumulator is never signalled and its wait gives up early
};

// Limit of the epilogue's wait for the withheld accumulator under the injected fault.
constexpr uint64_t kFaultWaitNs = 20000;

struct __align__(8) WinBars {
    uint64_t full[kMaxStages], empty[kMaxStages], acc_full[4], acc_empty[4];
    uint64_t mma_done;
    uint32_t tmem_base;
    volatile int abort_flag;
    volatile int gok[4][2];     // per group: the outcome of its accumulator wait, by item parity
    int done[2];                // per unit parity: groups finished with the unit
    volatile int ready[2];      // per unit parity: the local unit index whose maxima may use the buffer
    int last[4];                // per group: 1 if it finished a unit last
};

__host__ __device__ inline size_t stage_bytes(int Npad) { return (size_t)kKTileBytes + 2 * (size_t)Npad * 128; }

// Shared memory: stages | head maxima [2][O][128] | row statistics [4 groups][2][256] | barriers.
__host__ __device__ inline size_t win_smem_bytes(int Npad, int O, int kst) {
    return 1024 + (size_t)kst * stage_bytes(Npad) + 2 * (size_t)O * kTileT * sizeof(float) +
           4 * 2 * 256 * sizeof(float) + sizeof(WinBars);
}

__device__ __forceinline__ void win_abort(WinBars* bars, int* err) {
    bars->abort_flag = 1;
    atomicExch(err, 3);
}

// Unit u -> sequence s, candidate tile jt within it, head group ng, global
// candidate tile tg; sequence s owns ceil(Lc / 128) * NG consecutive units.
struct WinUnit {
    int s, jt, ng, tg, L, Lc, row0;
};

__device__ __forceinline__ bool decode_unit(const Geometry& G, const int* cu, int u, WinUnit& w) {
    int base = 0, tbase = 0;
    for (int b = 0; b < G.batch; ++b) {
        const int c0 = __ldg(&cu[b]), c1 = __ldg(&cu[b + 1]);
        const int Lc = c1 - c0 - G.wk;
        const int nt = Lc > 0 ? (Lc + kTileT - 1) / kTileT : 0;
        if (u < base + nt * G.NG) {
            const int local = u - base;
            w.s = b;
            w.jt = local / G.NG;
            w.ng = local - w.jt * G.NG;
            w.tg = tbase + w.jt;
            w.L = c1 - c0;
            w.Lc = Lc;
            w.row0 = c0 + w.jt * kTileT;
            return true;
        }
        base += nt * G.NG;
        tbase += nt;
    }
    return false;
}

// One head of this thread's token: the group sums G_h[q] of every window row q,
// added to po (q >= w-O) and poe (q >= w-O') and folded into the head maxima
// (q >= w-O).  Rows q < qmin come before the token (it lies in the window part,
// which only later rows see): their attention to it is 0.  GG > 0 is the group
// size g known at compile time: each 32-column chunk holds 32 / GG whole
// groups and runs as straight-line code.
template <int GG>
__device__ __forceinline__ void head_rows(uint32_t taddr, const float* __restrict__ rsb, int g, int w, int qmin,
                                          float sl2, int qO, int qOe, int* maxg_col, float& po, float& poe) {
    if constexpr (GG > 0) {
        constexpr int QPC = 32 / GG, CW = QPC * GG;
        for (int qb = 0; qb < w; qb += QPC) {
            const int c0 = qb * GG;
            float v[32];
            ptx::tmem_ld32(taddr + (uint32_t)c0, v);
            ptx::tmem_wait_ld();
            float pr[CW];
#pragma unroll
            for (int i = 0; i < CW; ++i) pr[i] = ptx::ex2(fmaf(v[i], sl2, -rsb[c0 + i]));
#pragma unroll
            for (int k = 0; k < QPC; ++k) {
                float gs = 0.f;
#pragma unroll
                for (int j = 0; j < GG; ++j) gs += pr[k * GG + j];
                const int q = qb + k;
                gs = q >= qmin ? gs : 0.f;
                if (q < w) {
                    if (q >= qOe) poe += gs;
                    if (q >= qO) {
                        po += gs;
                        atomicMax(maxg_col + (q - qO) * kTileT, __float_as_int(gs));
                    }
                }
            }
        }
    } else {
        float gs = 0.f;
        int q = 0, jq = 0;
        const int c_end = w * g;
        for (int c0 = 0; c0 < c_end; c0 += 32) {
            float v[32];
            ptx::tmem_ld32(taddr + (uint32_t)c0, v);
            ptx::tmem_wait_ld();
            const int n = min(32, c_end - c0);
#pragma unroll
            for (int i = 0; i < 32; ++i) {
                if (i >= n) break;
                gs += ptx::ex2(fmaf(v[i], sl2, -rsb[c0 + i]));
                if (++jq == g) {
                    gs = q >= qmin ? gs : 0.f;
                    if (q >= qOe) poe += gs;
                    if (q >= qO) {
                        po += gs;
                        atomicMax(maxg_col + (q - qO) * kTileT, __float_as_int(gs));
                    }
                    gs = 0.f;
                    jq = 0;
                    ++q;
                }
            }
        }
    }
}

template <int GG>
__global__ void __launch_bounds__(kWinThreads, 1)
    window_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap qmap,
                  const __grid_constant__ WinArgs A) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    if (threadIdx.x == 0) {
        ptx::prefetch_tensormap(&kmap);
        ptx::prefetch_tensormap(&qmap);
        // The next launch on this stream (the next layer's row statistics) reads
        // nothing this grid writes and does not wait for it: let it be scheduled.
        asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
    }
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    // Scalars and pointers in registers: values read through a reference to the
    // parameter block would be re-read after every asm statement that clobbers memory.
    const Geometry G = A.G;
    const Scratch sc = A.sc;
    const Slot sl = A.sl;
    const int* const cu_dev = A.cu;
    const int kst = A.kst, NA = A.nacc, units = A.units, fault = A.fault;
    const uint32_t tmem_cols = A.tmem_cols;
    const int Npad = A.Npad, R = G.R;
    const size_t sbytes = stage_bytes(Npad);
    int* maxg = reinterpret_cast<int*>(smem + kst * sbytes);             // [2][O][128] float bits
    float* rsm = reinterpret_cast<float*>(maxg + 2 * G.O * kTileT);      // [4][2][256] m_r + log2 Z_r
    WinBars* bars = reinterpret_cast<WinBars*>(rsm + 4 * 2 * 256);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int u0 = blockIdx.x, ustep = gridDim.x;

    if (threadIdx.x == 32) {
        for (int i = 0; i < kst; ++i) {
            ptx::mbar_init(&bars->full[i], 1);
            ptx::mbar_init(&bars->empty[i], 1);
        }
        for (int i = 0; i < 4; ++i) {
            ptx::mbar_init(&bars->acc_full[i], 1);
            ptx::mbar_init(&bars->acc_empty[i], 4);   // one arrival per warp of the group
        }
        ptx::mbar_init(&bars->mma_done, 1);
        bars->abort_flag = 0;
        for (int i = 0; i < 2; ++i) {
            bars->done[i] = 0;
            bars->ready[i] = i;
        }
        ptx::fence_barrier_init();
    }
    for (int i = threadIdx.x; i < 2 * G.O * kTileT; i += blockDim.x) maxg[i] = 0;
    if (warp == 1) {
        ptx::tmem_alloc(&bars->tmem_base, tmem_cols);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = bars->tmem_base;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            const uint64_t policy = ptx::policy_evict_first();   // the K tiles' last use
            int it = 0;
            int fills[kMaxStages] = {0, 0, 0};
            for (int u = u0; u < units && !bars->abort_flag; u += ustep) {
                WinUnit wu;
                decode_unit(G, cu_dev, u, wu);
                const int h0 = wu.ng * G.HG, nh = min(G.HG, G.Hkv - h0);
                bool stop = false;
                for (int hh = 0; hh < nh; ++hh, ++it) {
                    const int st = it % kst, n = it / kst;
                    if (n > 0 && !ptx::mbar_wait_abortable(&bars->empty[st], (n - 1) & 1, &bars->abort_flag)) {
                        win_abort(bars, sc.err);
                        stop = true;
                        break;
                    }
                    uint8_t* sk = smem + st * sbytes;
                    uint8_t* sq = sk + kKTileBytes;
                    const int h = h0 + hh;
                    ptx::mbar_arrive_expect_tx(&bars->full[st], (uint32_t)kKTileBytes + 2u * (uint32_t)R * 128u);
                    ptx::tma_load_3d(sk, &kmap, &bars->full[st], 0, h, wu.row0, policy);
                    ptx::tma_load_3d(sk + kKTileBytes / 2, &kmap, &bars->full[st], 64, h, wu.row0, policy);
                    ptx::tma_load_4d(sq, &qmap, &bars->full[st], 0, h * G.g, 0, wu.s);
                    ptx::tma_load_4d(sq + Npad * 128, &qmap, &bars->full[st], 64, h * G.g, 0, wu.s);
                    ++fills[st];
                }
                if (stop) break;
            }
            // Drain: every issued copy lands before the CTA may exit.
            for (int st = 0; st < kst; ++st)
                if (fills[st] > 0) ptx::mbar_wait(&bars->full[st], (fills[st] - 1) & 1, 50000000ull);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = ptx::idesc_bf16_f32(128, Npad);
            int it = 0;
            bool stop = false;
            for (int u = u0; u < units && !stop; u += ustep) {
                WinUnit wu;
                decode_unit(G, cu_dev, u, wu);
                const int nh = min(G.HG, G.Hkv - wu.ng * G.HG);
                for (int hh = 0; hh < nh; ++hh, ++it) {
                    const int st = it % kst, n = it / kst;
                    const int b = it % NA, ub = it / NA;
                    // Giving up on a stage in flight is safe: the producer drains its own loads.
                    if (bars->abort_flag || !ptx::mbar_wait_abortable(&bars->full[st], n & 1, &bars->abort_flag) ||
                        (ub > 0 && !ptx::mbar_wait_abortable(&bars->acc_empty[b], (ub - 1) & 1, &bars->abort_flag))) {
                        win_abort(bars, sc.err);
                        stop = true;
                        break;
                    }
                    ptx::tc_fence_after();
                    const uint32_t sk = ptx::smem_u32(smem + st * sbytes), sq = sk + kKTileBytes;
                    const uint32_t d = tmem + (uint32_t)(b * Npad);
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) {
                        const int half = kk >> 2, kin = kk & 3;
                        const uint64_t ad = ptx::smem_desc_k_sw128(sk + half * (kKTileBytes / 2) + kin * 32);
                        const uint64_t bd = ptx::smem_desc_k_sw128(sq + half * Npad * 128 + kin * 32);
                        ptx::mma_bf16(d, ad, bd, idesc, kk > 0 ? 1u : 0u);
                    }
                    ptx::mma_commit(&bars->empty[st]);
                    if (!(fault && it == 0)) ptx::mma_commit(&bars->acc_full[b]);
                }
            }
            ptx::mma_commit(&bars->mma_done);
        }
    } else if (warp < 2 + 4 * NA) {
        // ------------------------------------------------------------ epilogue
        const int grp = (warp - 2) >> 2;                  // accumulator / item group
        const int gtid = threadIdx.x - 64 - grp * 128;    // 0 .. 127 within the group
        const int quad = warp & 3;                        // TMEM lanes 32*quad .. +31
        const int tok = quad * 32 + lane;                 // token within the tile
        const int bar_id = 1 + grp;                       // named barrier of the group (128 threads)
        const int qO = G.w - G.O, qOe = G.w - G.Oe;
        const float invO = 1.f / (float)G.O, invOe = 1.f / (float)G.Oe;
        const uint32_t tbase = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(grp * Npad);
        float* rs_g = rsm + grp * 2 * 256;
        // Row statistics come from the launch this grid is a programmatic
        // dependent of: wait for it before the first read.
        asm volatile("griddepcontrol.wait;\n" ::: "memory");
        // This thread's rows (gtid, gtid + 128) of an item's statistics.
        auto fetch = [&](int s, int h, float& a, float& b) {
            const float2* src = sc.rowstat + ((size_t)s * G.Hkv + h) * R;
            a = b = 0.f;
            if (gtid < R) {
                const float2 m = __ldcg(src + gtid);
                a = m.x + __log2f(m.y);
            }
            if (gtid + 128 < R) {
                const float2 m = __ldcg(src + gtid + 128);
                b = m.x + __log2f(m.y);
            }
        };
        int it = 0, k = 0;   // it: CTA item index; k: this group's items so far
        bool failed = false;
        for (int u = u0, ul = 0; u < units; u += ustep, ++ul) {
            WinUnit wu;
            decode_unit(G, cu_dev, u, wu);
            const int h0 = wu.ng * G.HG, nh = min(G.HG, G.Hkv - h0);
            const int t = wu.jt * kTileT + tok;                  // token within the sequence
            const int qmin = t - (wu.L - G.w);                   // > 0 only for tokens in the window part
            const int buf = ul & 1;
            int* mg = maxg + buf * G.O * kTileT;
            // The head maxima buffer of this unit parity is free once the unit two
            // before has been folded into I (bounded wait on a flag of this CTA).
            if (!failed && ul >= 2) {
                int ok = 1;
                if (lane == 0) {
                    const long long c0 = clock64();
                    while (bars->ready[buf] != ul) {
                        if (bars->abort_flag || clock64() - c0 > 600000000ll) {
                            ok = 0;
                            break;
                        }
                        __nanosleep(64);
                    }
                }
                if (!__shfl_sync(0xffffffffu, ok, 0)) {
                    if (lane == 0) win_abort(bars, sc.err);
                    failed = true;
                }
                __threadfence_block();
            }
            float pa = 0.f, pb = 0.f;
            int hh = (grp - it % NA + NA) % NA;   // the unit's first item for this group
            if (!failed && hh < nh) fetch(wu.s, h0 + hh, pa, pb);
            for (; hh < nh && !failed; hh += NA, ++k) {
                // gtid 0 waits for the accumulator and publishes the outcome to the
                // group with the statistics (one barrier per item).
                if (gtid == 0) {
                    const bool ok = !bars->abort_flag &&
                                    ptx::mbar_wait_abortable(&bars->acc_full[grp], k & 1, &bars->abort_flag,
                                                             fault && it + hh == 0 ? kFaultWaitNs : 200000000ull);
                    if (!ok) win_abort(bars, sc.err);
                    bars->gok[grp][k & 1] = ok ? 1 : 0;
                }
                float* rsb = rs_g + (k & 1) * 256;
                rsb[gtid] = pa;
                rsb[gtid + 128] = pb;
                ptx::named_bar_sync(bar_id, 128);
                if (!bars->gok[grp][k & 1]) {
                    failed = true;
                    break;
                }
                if (hh + NA < nh) fetch(wu.s, h0 + hh + NA, pa, pb);   // next item's rows, in flight
                ptx::tc_fence_after();
                float po = 0.f, poe = 0.f;
                head_rows<GG>(tbase, rsb, G.g, G.w, qmin, G.sl2, qO, qOe, mg + tok, po, poe);
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(&bars->acc_empty[grp]);
                if (t < wu.Lc) {
                    const size_t row = (size_t)wu.s * G.Hkv + h0 + hh;
                    sl.rawO[row * G.ML + t] = po * invO;
                    sl.rawOe[row * G.ML + t] = poe * invOe;
                }
            }
            it += nh;
            if (failed) break;
            // This group is done with the unit: the last of the NA groups folds the
            // head maxima into I and frees the buffer for the unit two ahead.
            ptx::named_bar_sync(bar_id, 128);
            if (gtid == 0) {
                __threadfence_block();
                bars->last[grp] = atomicAdd(&bars->done[buf], 1) == NA - 1;
                __threadfence_block();
            }
            ptx::named_bar_sync(bar_id, 128);
            if (bars->last[grp]) {
                __threadfence_block();
                if (G.NG > 1) {
                    float* wp = sl.wpart + ((size_t)wu.tg * G.NG + wu.ng) * G.O * kTileT;
                    for (int q = 0; q < G.O; ++q) wp[q * kTileT + tok] = __int_as_float(mg[q * kTileT + tok]);
                } else if (t < wu.Lc) {
                    float ip = 0.f;
                    for (int q = 0; q < G.O; ++q) ip += __int_as_float(mg[q * kTileT + tok]);
                    sl.rawI[(size_t)wu.s * G.ML + t] = ip * invO;
                }
                for (int q = 0; q < G.O; ++q) mg[q * kTileT + tok] = 0;
                ptx::named_bar_sync(bar_id, 128);
                if (gtid == 0) {
                    bars->done[buf] = 0;
                    __threadfence_block();
                    bars->ready[buf] = ul + 2;
                }
            }
        }
    }

    // ---------------------------------------------------------------- teardown
    if (warp == 1 && lane == 0) ptx::mbar_wait(&bars->mma_done, 0, 50000000ull);
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc(tmem, tmem_cols);
}

// ---------------------------------------------------------------------------
// Tile-owning variant for O <= 16 and a group size with a straight-line epilogue
// (g in {1, 2, 4, 7, 8}): a unit is T = 4 (or, with N > 128, 2) consecutive
// candidate tiles of one sequence and one head group, and epilogue group j owns
// tile j of the unit for every head.  The query block Q_h is loaded once per
// (unit, head) into its own two-slot ring and serves the T tiles of the head, so
// the K ring holds 32 KB stages only (4 in flight instead of 3 stages of K and
// Q).  A thread keeps the running maxima over heads of its token's O last-row
// group sums in registers, so the groups never synchronise; it adds its rows in
// the same order as window_kernel, and the results are the same bits.
// ---------------------------------------------------------------------------
constexpr int kTileOMax = 16;     // largest O of the tile-owning variant (register maxima)
constexpr int kMaxKStages = 6;

struct TileArgs {
    Geometry G;
    Scratch sc;
    Slot sl;
    const int* cu;
    int Npad, kst, nacc, units, fault;
};

struct __align__(8) TileBars {
    uint64_t k_full[kMaxKStages], k_empty[kMaxKStages], q_full[2], q_empty[2], acc_full[4], acc_empty[4];
    uint64_t mma_done;
    uint32_t tmem_base;
    volatile int abort_flag;
    volatile int gok[4][2];     // per group: the outcome of its accumulator wait, by item parity
};

__host__ __device__ inline size_t tile_smem_bytes(int Npad, int kst) {
    return 1024 + (size_t)kst * kKTileBytes + 2 * (size_t)Npad * 256 + 4 * 2 * 256 * sizeof(float) + sizeof(TileBars);
}

// Unit u -> sequence s, first candidate tile j0 of the unit, its tile count nt,
// head group ng, global candidate tile of j0.
struct TileUnit {
    int s, j0, nt, ng, tg0, L, Lc, row0;
};

__device__ __forceinline__ bool decode_tile_unit(const Geometry& G, const int* cu, int T, int u, TileUnit& w) {
    int base = 0, tbase = 0;
    for (int b = 0; b < G.batch; ++b) {
        const int c0 = __ldg(&cu[b]), c1 = __ldg(&cu[b + 1]);
        const int Lc = c1 - c0 - G.wk;
        const int ntile = Lc > 0 ? (Lc + kTileT - 1) / kTileT : 0;
        const int ngrp = (ntile + T - 1) / T;
        if (u < base + ngrp * G.NG) {
            const int local = u - base;
            const int tgi = local / G.NG;
            w.s = b;
            w.ng = local - tgi * G.NG;
            w.j0 = tgi * T;
            w.nt = min(T, ntile - w.j0);
            w.tg0 = tbase + w.j0;
            w.L = c1 - c0;
            w.Lc = Lc;
            w.row0 = c0 + w.j0 * kTileT;
            return true;
        }
        base += ngrp * G.NG;
        tbase += ntile;
    }
    return false;
}

// One head of this thread's token: rows [qOe, qO) add to poe only, rows [qO, w)
// to po, to poe when q >= qOe, and to the running maxima mx[q - qO] (ascending q
// in both parts, as head_rows).
template <int GG>
__device__ __forceinline__ void head_rows_tile(uint32_t taddr, const float* __restrict__ rsb, int w, int qmin,
                                               float sl2, int qO, int qOe, float* mx, float& po, float& poe) {
    constexpr int QPC = 32 / GG, CW = QPC * GG;
    for (int qb = qOe; qb < qO; qb += QPC) {
        const int c0 = qb * GG;
        float v[32];
        ptx::tmem_ld32(taddr + (uint32_t)c0, v);
        ptx::tmem_wait_ld();
        float pr[CW];
#pragma unroll
        for (int i = 0; i < CW; ++i) pr[i] = ptx::ex2(fmaf(v[i], sl2, -rsb[c0 + i]));
#pragma unroll
        for (int k = 0; k < QPC; ++k) {
            float gs = 0.f;
#pragma unroll
            for (int j = 0; j < GG; ++j) gs += pr[k * GG + j];
            const int q = qb + k;
            gs = q >= qmin ? gs : 0.f;
            if (q < qO) poe += gs;
        }
    }
#pragma unroll
    for (int c = 0; c < (kTileOMax + QPC - 1) / QPC; ++c) {
        const int qb = qO + c * QPC;
        if (qb >= w) break;
        const int c0 = qb * GG;
        float v[32];
        ptx::tmem_ld32(taddr + (uint32_t)c0, v);
        ptx::tmem_wait_ld();
        float pr[CW];
#pragma unroll
        for (int i = 0; i < CW; ++i) pr[i] = ptx::ex2(fmaf(v[i], sl2, -rsb[c0 + i]));
#pragma unroll
        for (int k = 0; k < QPC; ++k) {
            const int idx = c * QPC + k;
            if (idx < kTileOMax) {
                float gs = 0.f;
#pragma unroll
                for (int j = 0; j < GG; ++j) gs += pr[k * GG + j];
                const int q = qb + k;
                gs = q >= qmin ? gs : 0.f;
                if (q < w) {
                    if (q >= qOe) poe += gs;
                    po += gs;
                    mx[idx] = fmaxf(mx[idx], gs);
                }
            }
        }
    }
}

template <int GG>
__global__ void __launch_bounds__(kWinThreads, 1)
    window_tiles_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap qmap,
                        const __grid_constant__ TileArgs A) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    if (threadIdx.x == 0) {
        ptx::prefetch_tensormap(&kmap);
        ptx::prefetch_tensormap(&qmap);
        // The next launch on this stream (the next layer's row statistics) reads
        // nothing this grid writes and does not wait for it: let it be scheduled.
        asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
    }
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const Geometry G = A.G;
    const Scratch sc = A.sc;
    const Slot sl = A.sl;
    const int* const cu_dev = A.cu;
    const int kst = A.kst, NA = A.nacc, units = A.units, fault = A.fault;
    const int Npad = A.Npad, R = G.R;
    const int T = NA;                                        // tiles per unit = epilogue groups
    uint8_t* sK = smem;                                      // kst x 32 KB
    uint8_t* sQ = sK + (size_t)kst * kKTileBytes;            // 2 slots x Npad x 256 B
    float* rsm = reinterpret_cast<float*>(sQ + 2 * (size_t)Npad * 256);   // [4][2][256]
    TileBars* bars = reinterpret_cast<TileBars*>(rsm + 4 * 2 * 256);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int u0 = blockIdx.x, ustep = gridDim.x;

    if (threadIdx.x == 32) {
        for (int i = 0; i < kst; ++i) {
            ptx::mbar_init(&bars->k_full[i], 1);
            ptx::mbar_init(&bars->k_empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(&bars->q_full[i], 1);
            ptx::mbar_init(&bars->q_empty[i], 1);
        }
        for (int i = 0; i < 4; ++i) {
            ptx::mbar_init(&bars->acc_full[i], 1);
            ptx::mbar_init(&bars->acc_empty[i], 4);   // one arrival per warp of the group
        }
        ptx::mbar_init(&bars->mma_done, 1);
        bars->abort_flag = 0;
        ptx::fence_barrier_init();
    }
    if (warp == 1) {
        ptx::tmem_alloc(&bars->tmem_base, 512);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = bars->tmem_base;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            const uint64_t policy = ptx::policy_evict_first();   // the K tiles' last use
            int qi = 0, ki = 0;
            int kfills[kMaxKStages] = {0, 0, 0, 0, 0, 0};
            int qfills[2] = {0, 0};
            bool stop = false;
            for (int u = u0; u < units && !stop; u += ustep) {
                TileUnit tu;
                decode_tile_unit(G, cu_dev, T, u, tu);
                const int h0 = tu.ng * G.HG, nh = min(G.HG, G.Hkv - h0);
                for (int hh = 0; hh < nh && !stop; ++hh) {
                    const int h = h0 + hh;
                    const int qs = qi & 1, nq = qi >> 1;
                    if (nq > 0 && !ptx::mbar_wait_abortable(&bars->q_empty[qs], (nq - 1) & 1, &bars->abort_flag)) {
                        bars->abort_flag = 1;
                        atomicExch(sc.err, 3);
                        stop = true;
                        break;
                    }
                    if (bars->abort_flag) {
                        stop = true;
                        break;
                    }
                    uint8_t* q = sQ + (size_t)qs * Npad * 256;
                    ptx::mbar_arrive_expect_tx(&bars->q_full[qs], 2u * (uint32_t)R * 128u);
                    ptx::tma_load_4d(q, &qmap, &bars->q_full[qs], 0, h * G.g, 0, tu.s);
                    ptx::tma_load_4d(q + Npad * 128, &qmap, &bars->q_full[qs], 64, h * G.g, 0, tu.s);
                    ++qfills[qs];
                    ++qi;
                    for (int j = 0; j < tu.nt; ++j) {
                        const int st = ki % kst, nk = ki / kst;
                        if (nk > 0 && !ptx::mbar_wait_abortable(&bars->k_empty[st], (nk - 1) & 1, &bars->abort_flag)) {
                            bars->abort_flag = 1;
                            atomicExch(sc.err, 3);
                            stop = true;
                            break;
                        }
                        uint8_t* sk = sK + (size_t)st * kKTileBytes;
                        const int row = tu.row0 + j * kTileT;
                        ptx::mbar_arrive_expect_tx(&bars->k_full[st], (uint32_t)kKTileBytes);
                        ptx::tma_load_3d(sk, &kmap, &bars->k_full[st], 0, h, row, policy);
                        ptx::tma_load_3d(sk + kKTileBytes / 2, &kmap, &bars->k_full[st], 64, h, row, policy);
                        ++kfills[st];
                        ++ki;
                    }
                }
            }
            // Drain: every issued copy lands before the CTA may exit.
            for (int st = 0; st < kst; ++st)
                if (kfills[st] > 0) ptx::mbar_wait(&bars->k_full[st], (kfills[st] - 1) & 1, 50000000ull);
            for (int qs = 0; qs < 2; ++qs)
                if (qfills[qs] > 0) ptx::mbar_wait(&bars->q_full[qs], (qfills[qs] - 1) & 1, 50000000ull);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = ptx::idesc_bf16_f32(128, Npad);
            int qi = 0, ki = 0, first = 1;
            int cnt[4] = {0, 0, 0, 0};
            bool stop = false;
            for (int u = u0; u < units && !stop; u += ustep) {
                TileUnit tu;
                decode_tile_unit(G, cu_dev, T, u, tu);
                const int nh = min(G.HG, G.Hkv - tu.ng * G.HG);
                for (int hh = 0; hh < nh && !stop; ++hh) {
                    const int qs = qi & 1;
                    if (bars->abort_flag ||
                        !ptx::mbar_wait_abortable(&bars->q_full[qs], (qi >> 1) & 1, &bars->abort_flag)) {
                        bars->abort_flag = 1;
                        atomicExch(sc.err, 3);
                        stop = true;
                        break;
                    }
                    const uint32_t sq = ptx::smem_u32(sQ + (size_t)qs * Npad * 256);
                    for (int j = 0; j < tu.nt; ++j) {
                        const int st = ki % kst;
                        // Giving up on a stage in flight is safe: the producer drains its own loads.
                        if (!ptx::mbar_wait_abortable(&bars->k_full[st], (ki / kst) & 1, &bars->abort_flag) ||
                            (cnt[j] > 0 &&
                             !ptx::mbar_wait_abortable(&bars->acc_empty[j], (cnt[j] - 1) & 1, &bars->abort_flag))) {
                            bars->abort_flag = 1;
                            atomicExch(sc.err, 3);
                            stop = true;
                            break;
                        }
                        ptx::tc_fence_after();
                        const uint32_t sk = ptx::smem_u32(sK + (size_t)st * kKTileBytes);
                        const uint32_t d = tmem + (uint32_t)(j * Npad);
#pragma unroll
                        for (int kk = 0; kk < 8; ++kk) {
                            const int half = kk >> 2, kin = kk & 3;
                            const uint64_t ad = ptx::smem_desc_k_sw128(sk + half * (kKTileBytes / 2) + kin * 32);
                            const uint64_t bd = ptx::smem_desc_k_sw128(sq + half * Npad * 128 + kin * 32);
                            ptx::mma_bf16(d, ad, bd, idesc, kk > 0 ? 1u : 0u);
                        }
                        ptx::mma_commit(&bars->k_empty[st]);
                        if (!(fault && first)) ptx::mma_commit(&bars->acc_full[j]);
                        first = 0;
                        ++ki;
                        ++cnt[j];
                    }
                    ptx::mma_commit(&bars->q_empty[qs]);
                    ++qi;
                }
            }
            ptx::mma_commit(&bars->mma_done);
        }
    } else if (warp < 2 + 4 * NA) {
        // ------------------------------------------------------------ epilogue
        const int grp = (warp - 2) >> 2;                  // the tile of the unit this group owns
        const int gtid = threadIdx.x - 64 - grp * 128;
        const int quad = warp & 3;
        const int tok = quad * 32 + lane;
        const int bar_id = 1 + grp;
        const int qO = G.w - G.O, qOe = G.w - G.Oe;
        const float invO = 1.f / (float)G.O, invOe = 1.f / (float)G.Oe;
        const uint32_t tbase = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(grp * Npad);
        float* rs_g = rsm + grp * 2 * 256;
        asm volatile("griddepcontrol.wait;\n" ::: "memory");
        auto fetch = [&](int s, int h, float& a, float& b) {
            const float2* src = sc.rowstat + ((size_t)s * G.Hkv + h) * R;
            a = b = 0.f;
            if (gtid < R) {
                const float2 m = __ldcg(src + gtid);
                a = m.x + __log2f(m.y);
            }
            if (gtid + 128 < R) {
                const float2 m = __ldcg(src + gtid + 128);
                b = m.x + __log2f(m.y);
            }
        };
        int k = 0;
        bool failed = false;
        for (int u = u0; u < units && !failed; u += ustep) {
            TileUnit tu;
            decode_tile_unit(G, cu_dev, T, u, tu);
            if (grp >= tu.nt) continue;   // this group's tile is past the sequence's last
            const int h0 = tu.ng * G.HG, nh = min(G.HG, G.Hkv - h0);
            const int t = (tu.j0 + grp) * kTileT + tok;
            const int qmin = t - (tu.L - G.w);
            float mx[kTileOMax];
#pragma unroll
            for (int i = 0; i < kTileOMax; ++i) mx[i] = 0.f;
            float pa, pb;
            fetch(tu.s, h0, pa, pb);
            for (int hh = 0; hh < nh; ++hh, ++k) {
                if (gtid == 0) {
                    const bool ok = !bars->abort_flag &&
                                    ptx::mbar_wait_abortable(&bars->acc_full[grp], k & 1, &bars->abort_flag,
                                                             fault && k == 0 && grp == 0 ? kFaultWaitNs
                                                                                         : 200000000ull);
                    if (!ok) {
                        bars->abort_flag = 1;
                        atomicExch(sc.err, 3);
                    }
                    bars->gok[grp][k & 1] = ok ? 1 : 0;
                }
                float* rsb = rs_g + (k & 1) * 256;
                rsb[gtid] = pa;
                rsb[gtid + 128] = pb;
                ptx::named_bar_sync(bar_id, 128);
                if (!bars->gok[grp][k & 1]) {
                    failed = true;
                    break;
                }
                if (hh + 1 < nh) fetch(tu.s, h0 + hh + 1, pa, pb);   // the next head's rows, in flight
                ptx::tc_fence_after();
                float po = 0.f, poe = 0.f;
                head_rows_tile<GG>(tbase, rsb, G.w, qmin, G.sl2, qO, qOe, mx, po, poe);
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(&bars->acc_empty[grp]);
                if (t < tu.Lc) {
                    const size_t row = (size_t)tu.s * G.Hkv + h0 + hh;
                    sl.rawO[row * G.ML + t] = po * invO;
                    sl.rawOe[row * G.ML + t] = poe * invOe;
                }
            }
            if (failed) break;
            // I[t] = (1/O) sum over the last O rows of the maxima over the heads (or
            // this head group's maxima, combined by the heads kernel).
            if (G.NG > 1) {
                float* wp = sl.wpart + ((size_t)(tu.tg0 + grp) * G.NG + tu.ng) * G.O * kTileT;
#pragma unroll
                for (int i = 0; i < kTileOMax; ++i)
                    if (i < G.O) wp[i * kTileT + tok] = mx[i];
            } else if (t < tu.Lc) {
                float ip = 0.f;
#pragma unroll
                for (int i = 0; i < kTileOMax; ++i)
                    if (i < G.O) ip += mx[i];
                sl.rawI[(size_t)tu.s * G.ML + t] = ip * invO;
            }
        }
    }

    // ---------------------------------------------------------------- teardown
    if (warp == 1 && lane == 0) ptx::mbar_wait(&bars->mma_done, 0, 50000000ull);
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc(tmem, 512);
}

int npad_of(int R) { return (R + 15) & ~15; }

int kst_for(int Npad, int O) {
    int k = kMaxStages;
    while (k > 1 && win_smem_bytes(Npad, O, k) > (size_t)kMaxSmemWin) --k;
    return k;
}

// Units of a launch: (sequence, candidate tile, head group).
int units_of(const Geometry& g) { return g.win_tiles * g.NG; }

}  // namespace

size_t window_smem_bytes(const Geometry& g) {
    const int Npad = npad_of(g.R);
    return win_smem_bytes(Npad, g.O, kst_for(Npad, g.O));
}

cudaError_t configure_window(const Geometry& g) {
    // Per-function attribute shared by every handle: the opt-in maximum (every
    // geometry's stage count is chosen to fit it).
    (void)g;
    cudaError_t e = cudaSuccess;
    for (auto fn : {window_kernel<0>, window_kernel<1>, window_kernel<2>, window_kernel<4>, window_kernel<7>,
                    window_kernel<8>})
        if (e == cudaSuccess) e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmemWin);
    for (auto fn : {window_tiles_kernel<1>, window_tiles_kernel<2>, window_tiles_kernel<4>, window_tiles_kernel<7>,
                    window_tiles_kernel<8>})
        if (e == cudaSuccess) e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmemWin);
    return e;
}

namespace {

int tile_kst_for(int Npad) {
    int k = kMaxKStages;
    while (k > 1 && tile_smem_bytes(Npad, k) > (size_t)kMaxSmemWin) --k;
    return k;
}

// The tile variant applies to O <= 16 with a straight-line group size, when every
// 32-column TMEM load of its epilogue (chunks starting at rows w - O' and w - O)
// stays inside the 512 allocated columns.
bool tile_variant_fits(const Geometry& g) {
    if (g.O > kTileOMax || !(g.g == 1 || g.g == 2 || g.g == 4 || g.g == 7 || g.g == 8)) return false;
    const int qpc = 32 / g.g, qO = g.w - g.O, qOe = g.w - g.Oe;
    const int Npad = npad_of(g.R), nacc = Npad <= 128 ? 4 : 2;
    int maxcol = 0;
    for (int qb = qOe; qb < qO; qb += qpc) maxcol = maxcol > qb * g.g + 32 ? maxcol : qb * g.g + 32;
    for (int c = 0; c < (kTileOMax + qpc - 1) / qpc; ++c) {
        const int qb = qO + c * qpc;
        if (qb >= g.w) break;
        maxcol = maxcol > qb * g.g + 32 ? maxcol : qb * g.g + 32;
    }
    return (nacc - 1) * Npad + maxcol <= 512;
}

// Candidate tiles per unit of the tile-owning variant: one TMEM accumulator and
// epilogue group each (nacc * Npad <= 512 columns).  With the caller's
// log-sum-exp no score grid runs beside the window grids, and units of three
// tiles (more units, a shorter tail) were faster than four there (ragged batch
// of 8: 2.09 -> 1.90 ms per step), while beside the score grids they were
// slower (3.02 -> 3.06 ms); two tiles were slower in both.
int tile_unit_tiles(const Geometry& g, bool lse) { return npad_of(g.R) <= 128 ? (lse ? 3 : 4) : 2; }

// Units of the tile-owning variant: groups of T candidate tiles per sequence and head group.
int tile_units_of(const Geometry& g, const int* cu_host, int T) {
    int units = 0;
    for (int b = 0; b < g.batch; ++b) {
        const int Lc = cu_host[b + 1] - cu_host[b] - g.wk;
        const int nt = Lc > 0 ? (Lc + kTileT - 1) / kTileT : 0;
        units += (nt + T - 1) / T * g.NG;
    }
    return units;
}

cudaError_t launch_window_tiles(const ScorePlan& sp, const Geometry& g, const LayerIO& io, const Scratch& sc,
                                const Slot& sl, cudaStream_t st, bool after_own_launch) {
    TileArgs a{};
    a.G = g;
    a.sc = sc;
    a.sl = sl;
    a.cu = io.cu;
    a.Npad = npad_of(g.R);
    a.nacc = tile_unit_tiles(g, io.lse != nullptr);
    a.kst = tile_kst_for(a.Npad);
    a.units = tile_units_of(g, g.cu_host, a.nacc);
    a.fault = test_fault() == 1 ? 1 : 0;
    const size_t smem = tile_smem_bytes(a.Npad, a.kst);
    const int usable = sp.num_sms > 2 * kWinReserveSms ? sp.num_sms - kWinReserveSms : sp.num_sms;
    const int grid = a.units < usable ? a.units : usable;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kWinThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = after_own_launch ? 1 : 0;
    switch (g.g) {
        case 1: return cudaLaunchKernelEx(&cfg, window_tiles_kernel<1>, sp.kmap, sp.qmap, a);
        case 2: return cudaLaunchKernelEx(&cfg, window_tiles_kernel<2>, sp.kmap, sp.qmap, a);
        case 4: return cudaLaunchKernelEx(&cfg, window_tiles_kernel<4>, sp.kmap, sp.qmap, a);
        case 7: return cudaLaunchKernelEx(&cfg, window_tiles_kernel<7>, sp.kmap, sp.qmap, a);
        default: return cudaLaunchKernelEx(&cfg, window_tiles_kernel<8>, sp.kmap, sp.qmap, a);
    }
}

}  // namespace

int window_grid_size(const ScorePlan& sp, const Geometry& g, bool lse) {
    if (g.win_tiles == 0) return 0;
    const int usable = sp.num_sms > 2 * kWinReserveSms ? sp.num_sms - kWinReserveSms : sp.num_sms;
    if (tile_variant_fits(g) && tile_units_of(g, g.cu_host, tile_unit_tiles(g, lse)) >= usable) return usable;
    return units_of(g) < usable ? units_of(g) : usable;
}

cudaError_t launch_window(const ScorePlan& sp, const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl,
                          cudaStream_t st, bool after_own_launch) {
    if (g.win_tiles == 0) return cudaSuccess;
    // The tile-owning variant where it applies and its units still give every
    // usable SM one (it has T times fewer units than the per-tile kernel, whose
    // CTAs finish sooner when there are few tiles).
    if (tile_variant_fits(g)) {
        const int T = tile_unit_tiles(g, io.lse != nullptr);
        const int usable = sp.num_sms > 2 * kWinReserveSms ? sp.num_sms - kWinReserveSms : sp.num_sms;
        if (tile_units_of(g, g.cu_host, T) >= usable) return launch_window_tiles(sp, g, io, sc, sl, st, after_own_launch);
    }
    WinArgs a{};
    a.G = g;
    a.sc = sc;
    a.sl = sl;
    a.cu = io.cu;
    a.Npad = npad_of(g.R);
    a.kst = kst_for(a.Npad, g.O);
    a.nacc = a.Npad <= 128 ? 4 : 2;   // nacc * Npad <= 512 TMEM columns
    a.units = units_of(g);
    a.fault = test_fault() == 1 ? 1 : 0;
    a.tmem_cols = 512;   // one CTA per SM; a 32-column load past the last group's columns stays inside
    const size_t smem = win_smem_bytes(a.Npad, g.O, a.kst);
    // Persistent: at most one CTA per SM, leaving a few SMs to the selection
    // chain and the other layers' kernels.
    const int usable = sp.num_sms > 2 * kWinReserveSms ? sp.num_sms - kWinReserveSms : sp.num_sms;
    const int grid = a.units < usable ? a.units : usable;
    // after_own_launch: the previous kernel on the stream is this layer's
    // row-statistics launch and no event wait stands between them; the launch is
    // then its programmatic dependent and waits (griddepcontrol.wait) right
    // before reading the statistics.
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kWinThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = after_own_launch ? 1 : 0;
    switch (g.g) {
        case 1: return cudaLaunchKernelEx(&cfg, window_kernel<1>, sp.kmap, sp.qmap, a);
        case 2: return cudaLaunchKernelEx(&cfg, window_kernel<2>, sp.kmap, sp.qmap, a);
        case 4: return cudaLaunchKernelEx(&cfg, window_kernel<4>, sp.kmap, sp.qmap, a);
        case 7: return cudaLaunchKernelEx(&cfg, window_kernel<7>, sp.kmap, sp.qmap, a);
        case 8: return cudaLaunchKernelEx(&cfg, window_kernel<8>, sp.kmap, sp.qmap, a);
        default: return cudaLaunchKernelEx(&cfg, window_kernel<0>, sp.kmap, sp.qmap, a);
    }
}

}  // namespace kvec
