// Eq. 1 window scores and the Section 4.2 importance I (before pooling), from
// the window queries' attention over the candidate tokens, recomputed on the
// tensor cores with the softmax statistics (m_r, Z_r) of the score kernel.
//
// One CTA per (sequence s, 128-token tile of candidates, group of KV heads);
// the candidates are [0, L - w), or [0, L) when every position competes.
// For each KV head h of the group the CTA computes S^T = K_tile Q_h^T with
// tcgen05.mma (M = 128 tokens, N = g*w query rows padded to 16, K = d) into
// TMEM, so one epilogue thread owns one token and every query row of it:
//   A[r][t]   = 2^(s_rt * scale * log2(e) - m_r) / Z_r   (softmax over all visible keys)
//   G_h[q][t] = sum_j A[(q, j)][t]                       (GQA group sum, r = q * g + j)
//   P_O[h,t]  = (1/O)  sum_{q >= w-O}  G_h[q][t]
//   P_O'[h,t] = (1/O') sum_{q >= w-O'} G_h[q][t]
//   I[t]      = (1/O)  sum_{q >= w-O}  max_h G_h[q][t]
// Warp 0 streams K_h and Q_h with TMA, warp 1 issues the MMAs into one or two
// TMEM accumulators, warps 2..17 are the epilogue: four warps per TMEM lane
// quadrant, each taking a quarter of the window rows q (straight-line code per
// 32-column chunk when the group size g is a compile-time case).  The head
// maxima of G_h[q][t] stay in shared memory; when the KV heads are split over
// several CTAs each group writes its maxima to a partial buffer and the heads
// kernel combines the groups into I.  The raw rows go to the slot arrays;
// pooling happens in the heads kernel.
#include <cudaTypedefs.h>

#include "kvec_internal.cuh"
#include "sm100_ptx.cuh"

namespace kvec {

namespace {

constexpr int kWinThreads = 576;                      // warp 0 TMA, warp 1 MMA, warps 2..17 epilogue
constexpr int kEpiThreads = 512;
constexpr int kEpiWarps = kEpiThreads / 32;
constexpr int kMaxSmemWin = 232448;                   // opt-in shared memory per CTA on sm_103
constexpr int kKTileBytes = kTileT * kHeadDim * 2;    // 32 KB: two 64-column swizzled halves
constexpr int kRsRows = 288;                          // row-statistics buffer: R <= 256 plus a chunk's overrun

struct WinArgs {
    Geometry G;
    Scratch sc;
    Slot sl;
    const int* cu;                  // device cu_seqlens
    int Npad;                       // query rows padded to a multiple of 16 (MMA N)
    int kst;                        // operand stages
    int nacc;                       // TMEM accumulators (2, or 1 when 2 do not fit)
    uint32_t tmem_cols;
    int fault;                      // test of the error path (kvec_set_test_fault): the first
                                    // accumulator is never signalled and its wait gives up early
};

// Limit of the epilogue's wait for the withheld accumulator under the injected fault.
constexpr uint64_t kFaultWaitNs = 20000;

struct __align__(8) WinBars {
    uint64_t full[2], empty[2], acc_full[2], acc_empty[2];
    uint64_t mma_done;
    uint32_t tmem_base;
    volatile int abort_flag;
    volatile int epi_fail;     // set by an epilogue warp whose accumulator wait gave up
};

__host__ __device__ inline size_t stage_bytes(int Npad) { return (size_t)kKTileBytes + 2 * (size_t)Npad * 128; }

__host__ __device__ inline size_t win_smem_bytes(int Npad, int O, int kst) {
    return 1024 + (size_t)kst * stage_bytes(Npad) + kWinHeadsPerCta * kRsRows * sizeof(float) +
           (size_t)O * kTileT * sizeof(float) + kWinHeadsPerCta * 4 * kTileT * sizeof(float2) + sizeof(WinBars);
}

__device__ __forceinline__ void win_abort(WinBars* bars, int* err) {
    bars->abort_flag = 1;
    atomicExch(err, 3);
}

// One head's window rows [q_lo, q_hi) of this thread's token: adds the rows'
// group sums G_h[q] to po (q >= w-O) and poe (q >= w-O') and folds them into
// the head maxima.  Rows q < qmin come before the token (it lies in the window
// part, which only later rows see): their attention to it is 0.  GG > 0 is the
// group size g known at compile time: each 32-column chunk holds 32 / GG whole
// groups and runs as straight-line code.
template <int GG>
__device__ __forceinline__ void head_rows(uint32_t taddr, const float* __restrict__ rsb, int g, int q_lo, int q_hi,
                                          int qmin, float sl2, int qO, int qOe, float* maxg_col, bool first,
                                          float& po, float& poe) {
    if constexpr (GG > 0) {
        constexpr int QPC = 32 / GG, CW = QPC * GG;
        for (int qb = q_lo; qb < q_hi; qb += QPC) {
            const int c0 = qb * GG;
            float v[32];
            ptx::tmem_ld32(taddr + (uint32_t)c0, v);
            ptx::tmem_wait_ld();
            float pr[CW];
#pragma unroll
            for (int i = 0; i < CW; ++i) {
                pr[i] = ptx::ex2(fmaf(v[i], sl2, -rsb[c0 + i]));
            }
#pragma unroll
            for (int k = 0; k < QPC; ++k) {
                float gs = 0.f;
#pragma unroll
                for (int j = 0; j < GG; ++j) gs += pr[k * GG + j];
                const int q = qb + k;
                gs = q >= qmin ? gs : 0.f;
                if (q < q_hi) {
                    if (q >= qOe) poe += gs;
                    if (q >= qO) {
                        po += gs;
                        float* mg = maxg_col + (q - qO) * kTileT;
                        *mg = first ? gs : fmaxf(*mg, gs);
                    }
                }
            }
        }
    } else {
        float gs = 0.f;
        int q = q_lo, jq = 0;
        const int c_end = q_hi * g;
        for (int c0 = q_lo * g; c0 < c_end; c0 += 32) {
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
                        float* mg = maxg_col + (q - qO) * kTileT;
                        *mg = first ? gs : fmaxf(*mg, gs);
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
    const int kst = A.kst, nacc = A.nacc, fault = A.fault;
    const uint32_t tmem_cols = A.tmem_cols;
    const int Npad = A.Npad, R = G.R;
    const size_t sbytes = stage_bytes(Npad);
    float* rs = reinterpret_cast<float*>(smem + kst * sbytes);        // [HG][kRsRows] m_r + log2 Z_r
    float* maxg = reinterpret_cast<float*>(rs + kWinHeadsPerCta * kRsRows);   // [O][128] max over heads of G_h[q][t]
    float2* xfer = reinterpret_cast<float2*>(maxg + G.O * kTileT);      // [HG][4][128] quarters' (P_O, P_O') sums
    WinBars* bars = reinterpret_cast<WinBars*>(xfer + kWinHeadsPerCta * 4 * kTileT);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    // Work item -> (sequence, candidate tile, head group); sequence s owns
    // ceil(Lc / 128) * NG consecutive CTAs.
    auto cu = [&](int b) { return __ldg(&cu_dev[b]); };
    int s = -1, jt = 0, ng = 0, tg = 0;
    {
        int base = 0, tbase = 0;
        for (int b = 0; b < G.batch; ++b) {
            const int Lc = cu(b + 1) - cu(b) - G.wk;
            const int nt = Lc > 0 ? (Lc + kTileT - 1) / kTileT : 0;
            if ((int)blockIdx.x < base + nt * G.NG) {
                const int local = (int)blockIdx.x - base;
                s = b;
                jt = local / G.NG;
                ng = local - jt * G.NG;
                tg = tbase + jt;
                break;
            }
            base += nt * G.NG;
            tbase += nt;
        }
    }
    if (s < 0) return;   // the whole CTA, before any barrier or TMEM use
    const int L = cu(s + 1) - cu(s), Lc = L - G.wk;
    const int h0 = ng * G.HG;
    const int nh = min(G.HG, G.Hkv - h0);
    const int NB = nacc;

    if (threadIdx.x == 32) {
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(&bars->full[i], 1);
            ptx::mbar_init(&bars->empty[i], 1);
            ptx::mbar_init(&bars->acc_full[i], 1);
            ptx::mbar_init(&bars->acc_empty[i], kEpiThreads / 32);   // one arrival per epilogue warp
        }
        ptx::mbar_init(&bars->mma_done, 1);
        bars->abort_flag = 0;
        bars->epi_fail = 0;
        ptx::fence_barrier_init();
    }
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
            const int row0 = cu(s) + jt * kTileT;
            int fills[2] = {0, 0};
            for (int hh = 0; hh < nh && !bars->abort_flag; ++hh) {
                const int st = hh % kst, u = hh / kst;
                if (u > 0 && !ptx::mbar_wait_abortable(&bars->empty[st], (u - 1) & 1, &bars->abort_flag)) {
                    win_abort(bars, sc.err);
                    break;
                }
                uint8_t* sk = smem + st * sbytes;
                uint8_t* sq = sk + kKTileBytes;
                const int h = h0 + hh;
                ptx::mbar_arrive_expect_tx(&bars->full[st], (uint32_t)kKTileBytes + 2u * (uint32_t)R * 128u);
                ptx::tma_load_3d(sk, &kmap, &bars->full[st], 0, h, row0, policy);
                ptx::tma_load_3d(sk + kKTileBytes / 2, &kmap, &bars->full[st], 64, h, row0, policy);
                ptx::tma_load_4d(sq, &qmap, &bars->full[st], 0, h * G.g, 0, s);
                ptx::tma_load_4d(sq + Npad * 128, &qmap, &bars->full[st], 64, h * G.g, 0, s);
                ++fills[st];
            }
            // Drain: every issued copy lands before the CTA may exit.
            for (int st = 0; st < kst; ++st)
                if (fills[st] > 0) ptx::mbar_wait(&bars->full[st], (fills[st] - 1) & 1, 50000000ull);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = ptx::idesc_bf16_f32(128, Npad);
            for (int hh = 0; hh < nh && !bars->abort_flag; ++hh) {
                const int st = hh % kst, u = hh / kst;
                const int b = hh % NB, ub = hh / NB;
                if (!ptx::mbar_wait(&bars->full[st], u & 1) ||
                    (ub > 0 && !ptx::mbar_wait_abortable(&bars->acc_empty[b], (ub - 1) & 1, &bars->abort_flag))) {
                    win_abort(bars, sc.err);
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
                if (!(fault && hh == 0)) ptx::mma_commit(&bars->acc_full[b]);
            }
            ptx::mma_commit(&bars->mma_done);
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int e = threadIdx.x - 64;                   // 0 .. kEpiThreads - 1
        const int qt = (warp - 2) >> 2;                   // quarter of the window rows
        const int quad = warp & 3;                        // TMEM lanes 32*quad .. +31
        const int tokl = quad * 32 + lane;
        const int t = jt * kTileT + tokl;
        const int qmin = t - (L - G.w);   // > 0 only for tokens in the window part
        const int q_lo = (qt * G.w) >> 2, q_hi = ((qt + 1) * G.w) >> 2;
        const int qO = G.w - G.O, qOe = G.w - G.Oe;
        const float invO = 1.f / (float)G.O, invOe = 1.f / (float)G.Oe;
        // Row statistics of every head of the group: A = 2^(s * sl2 - (m_r + log2 Z_r)).
        // They come from the launch this grid is a programmatic dependent of: wait
        // for it here, after the set-up and the first operand loads.
        asm volatile("griddepcontrol.wait;\n" ::: "memory");
        for (int i = e; i < nh * R; i += kEpiThreads) {
            const int hh = i / R, r = i - hh * R;
            const float2 ms = __ldcg(&sc.rowstat[((size_t)s * G.Hkv + h0 + hh) * R + r]);
            rs[hh * kRsRows + r] = ms.x + __log2f(ms.y);
        }
        ptx::named_bar_sync(1, kEpiThreads);
        // The warps run through the heads independently: each waits for the
        // accumulator itself and leaves its partial sums in xfer.
        for (int hh = 0; hh < nh; ++hh) {
            const int b = hh % NB, ub = hh / NB;
            int got = 1;
            if (lane == 0)
                got = !bars->abort_flag &&
                      ptx::mbar_wait(&bars->acc_full[b], ub & 1, fault && hh == 0 ? kFaultWaitNs : 200000000ull);
            got = __shfl_sync(0xffffffffu, got, 0);
            if (!got) {
                if (lane == 0) {
                    bars->epi_fail = 1;
                    win_abort(bars, sc.err);
                }
                break;
            }
            ptx::tc_fence_after();
            const uint32_t taddr = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(b * Npad);
            float po = 0.f, poe = 0.f;
            head_rows<GG>(taddr, rs + hh * kRsRows, G.g, q_lo, q_hi, qmin, G.sl2, qO, qOe, maxg + tokl, hh == 0, po,
                          poe);
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&bars->acc_empty[b]);
            xfer[(hh * 4 + qt) * kTileT + tokl] = make_float2(po, poe);
        }
        // Every epilogue warp arrives here, failed or not; epi_fail is only written
        // before this barrier, so the branch below is uniform.
        ptx::named_bar_sync(1, kEpiThreads);
        const bool aborted = bars->epi_fail != 0;
        if (!aborted) {
            // P_O and P_O' of every head of the group: the four quarters' sums.
            for (int i = e; i < nh * kTileT; i += kEpiThreads) {
                const int hh = i >> 7, tk = i & (kTileT - 1);
                const int tt = jt * kTileT + tk;
                if (tt < Lc) {
                    float so = 0.f, soe = 0.f;
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const float2 x = xfer[(hh * 4 + k) * kTileT + tk];
                        so += x.x;
                        soe += x.y;
                    }
                    const size_t row = (size_t)s * G.Hkv + h0 + hh;
                    sl.rawO[row * G.ML + tt] = so * invO;
                    sl.rawOe[row * G.ML + tt] = soe * invOe;
                }
            }
        }
        if (!aborted) {
            // I[t] = (1/O) sum over q >= w - O of the maxima over every KV head.  With
            // the heads in one CTA it is complete here; otherwise each group leaves its
            // maxima and the heads kernel takes the maximum over the groups.
            const int n_el = G.O * kTileT;
            if (G.NG > 1) {
                float* wp = sl.wpart + ((size_t)tg * G.NG + ng) * n_el;
                for (int i = e; i < n_el; i += kEpiThreads) wp[i] = maxg[i];
            } else if (e < kTileT && jt * kTileT + e < Lc) {
                float ip = 0.f;
                for (int qi = 0; qi < G.O; ++qi) ip += maxg[qi * kTileT + e];
                sl.rawI[(size_t)s * G.ML + jt * kTileT + e] = ip * invO;
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

int npad_of(int R) { return (R + 15) & ~15; }

int kst_for(int Npad, int O) { return win_smem_bytes(Npad, O, 2) <= (size_t)kMaxSmemWin ? 2 : 1; }

}  // namespace

size_t window_smem_bytes(const Geometry& g) {
    const int Npad = npad_of(g.R);
    return win_smem_bytes(Npad, g.O, kst_for(Npad, g.O));
}

cudaError_t configure_window(const Geometry& g) {
    // Per-function attribute shared by every handle: the largest supported geometry.
    size_t need = 0;
    for (int R = 16; R <= 256; R += 16) {
        const size_t b = win_smem_bytes(R, kMaxObsWindow, kst_for(R, kMaxObsWindow));
        if (b > need) need = b;
    }
    (void)g;
    cudaError_t e = cudaSuccess;
    for (auto fn : {window_kernel<0>, window_kernel<1>, window_kernel<2>, window_kernel<4>, window_kernel<7>,
                    window_kernel<8>})
        if (e == cudaSuccess) e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)need);
    return e;
}

cudaError_t launch_window(const ScorePlan& sp, const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl,
                          cudaStream_t st, bool after_own_launch) {
    if (g.win_tiles == 0) return cudaSuccess;
    WinArgs a{};
    a.G = g;
    a.sc = sc;
    a.sl = sl;
    a.cu = io.cu;
    a.Npad = npad_of(g.R);
    a.kst = kst_for(a.Npad, g.O);
    a.nacc = 2 * a.Npad + 32 <= 512 ? 2 : 1;
    a.fault = test_fault() == 1 ? 1 : 0;
    uint32_t need = a.nacc == 2 ? (uint32_t)(2 * a.Npad + 32) : 512u, cols = 32;
    while (cols < need) cols <<= 1;
    a.tmem_cols = cols;
    const size_t smem = win_smem_bytes(a.Npad, g.O, a.kst);
    const int grid = g.win_tiles * g.NG;
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
