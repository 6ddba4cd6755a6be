// Softmax statistics of the window queries' attention over every visible key
// (the denominators of the attention A that Eq. 1 averages): for each query
// row r of KV head h, the row max m_r of s = <q_r, k_t> * scale (log2 units)
// and Z_r = sum_t 2^(s_rt - m_r), causal on the window part.
//
// Persistent, warp-specialised, one CTA per SM; CTAs claim chunks of
// consecutive work items (sequence s, KV head h, 128-token tile j)
// from a per-launch counter, so a CTA that starts late (its SM held by other
// kernels) takes fewer chunks instead of delaying the launch:
//   warp 0      TMA producer: the KV head's g*w query rows (once per (s,h)) and
//               a ring of 128-token K tiles, both 128-byte swizzled;
//   warp 1      one thread issues tcgen05.mma (M = 128 query rows per M-block,
//               N = 128 tokens, K = 128 = d) into TMEM accumulators;
//   warps 2..17 epilogue: groups of warps, one per TMEM accumulator, each
//               taking every NB-th item; one thread per query row and all
//               128 columns of the item: tcgen05.ld of its logits, their sum
//               of 2^(s - max), merged online into the thread's running
//               (max, sum) of the CTA's contiguous segment of (s, h).
// At the end of a segment (a run of one (s, h) inside a chunk) the groups merge
// in shared memory and the CTA writes one (max, sum) partial per row, keyed by
// the segment's first item; rowstat_kernel then merges the partials of a (s, h)
// into (m_r, Z_r).  The segments are fixed by the chunk boundaries, not by which
// CTA claimed a chunk, so the results do not depend on the schedule.
// The window kernel recomputes the logits with these statistics.
#include <cudaTypedefs.h>

#include "kvec_internal.cuh"
#include "sm100_ptx.cuh"

namespace kvec {

namespace {

constexpr int kKStages = 4;                           // deepest K ring (fewer when shared memory is short)
constexpr int kMaxSmem = 232448;                      // opt-in shared memory per CTA on sm_103
constexpr int kKStageBytes = kTileT * kHeadDim * 2;   // 32 KB: two 64-column swizzled halves
constexpr int kKHalfBytes = kTileT * 128;             // 16 KB
constexpr uint32_t kTmemCols = 512;

// Position of work item i: sequence s, KV head h, tile j.  Items are ordered
// (s, h, j); sequence s owns ntiles(s) * Hkv consecutive items.  A CTA walks its
// items in order, so the walker decodes once and then steps, reading the
// sequence offsets (device memory) only when the sequence changes.
struct ItemWalker {
    const int* cu;
    int batch, Hkv;
    int s, h, j, ibase, ntiles;   // ibase: first item of (s, h)
    int row0, L;                  // cu[s], L_s

    __device__ __forceinline__ void enter_sequence() {
        row0 = __ldg(&cu[s]);
        L = __ldg(&cu[s + 1]) - row0;
        ntiles = tiles_of(L);
    }
    __device__ __forceinline__ void init(const int* cu_, int batch_, int Hkv_, int i) {
        cu = cu_;
        batch = batch_;
        Hkv = Hkv_;
        int base = 0;
        for (s = 0; s < batch; ++s) {
            enter_sequence();
            if (i < base + ntiles * Hkv) break;
            base += ntiles * Hkv;
        }
        const int local = i - base;
        h = local / ntiles;
        j = local - h * ntiles;
        ibase = base + h * ntiles;
    }
    __device__ __forceinline__ bool last_of_head() const { return j + 1 == ntiles; }
    __device__ __forceinline__ void next() {
        if (++j < ntiles) return;
        j = 0;
        ibase += ntiles;
        if (++h < Hkv) return;
        h = 0;
        if (++s < batch) enter_sequence();
    }
};

constexpr int kScoreReserveSms = 8;      // SMs a score launch leaves to the other kernels
constexpr int kChunkLarge = 12;          // (sequence, head, tile) items per claim when there are enough
constexpr int kChunkSmall = 8;           // items per claim otherwise
constexpr int kChunkSlots = 4;           // claimed chunks in flight inside a CTA

struct ScoreArgs {
    Geometry G;
    const int* cu;                 // device cu_seqlens
    Scratch sc;
    int W;        // total work items
    int kst;      // K ring depth
    int* claim;   // the launch's chunk counter, zero before the launch
    int chunk;    // items per claim
};

constexpr int kEpiWarps = 16;
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kScoreThreads = 64 + kEpiThreads;

struct __align__(8) Barriers {
    uint64_t k_full[kKStages], k_empty[kKStages];
    uint64_t q_full, q_empty;
    uint64_t acc_full[4], acc_empty[4];
    uint64_t c_full[kChunkSlots], c_empty[kChunkSlots];
    uint64_t mma_done;
    uint32_t tmem_base;
    volatile int abort_flag;
    volatile int chunk[kChunkSlots];   // claimed chunk (-1: no more work)
    volatile int cur_chunk[2];         // the epilogue's current chunk (-2: gave up), double-buffered
    float2 xf[512];            // a segment's (max, sum) per epilogue group and row, merged at its end
};

__device__ __forceinline__ void raise_abort(Barriers* bars, int* err) {
    bars->abort_flag = 1;
    atomicExch(err, 3);
}

// MB: 128-row M-blocks per KV head (R <= 128 * MB).  The 16 epilogue warps form
// NB = 4 / MB groups of 4 * MB warps, one group per TMEM accumulator.
template <int MB>
__global__ void __launch_bounds__(kScoreThreads, 1)
    score_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap qmap,
                 const __grid_constant__ ScoreArgs A) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    // 1024-byte alignment for the swizzled operand tiles.
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    // Scalars and pointers in registers: values read through a reference to the
    // parameter block would be re-read after every asm statement that clobbers memory.
    const Geometry G = A.G;
    const Scratch sc = A.sc;
    const int W = A.W, kst = A.kst;
    const int chunk_items = A.chunk;
    const int nchunks = (W + chunk_items - 1) / chunk_items;
    int* const claim = A.claim;
    const int* const cu_dev = A.cu;
    const int Rpad = 128 * MB, R = G.R;
    uint8_t* sQ = smem;                                   // 2 halves x Rpad rows x 128 B
    uint8_t* sK = sQ + 2 * Rpad * 128;                    // kst x 32 KB
    Barriers* bars = reinterpret_cast<Barriers*>(sK + kst * kKStageBytes);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int NB = 4 / MB;                             // TMEM accumulator buffers

    if (warp == 0 && lane == 0) {
        ptx::prefetch_tensormap(&kmap);
        ptx::prefetch_tensormap(&qmap);
        // The next launch on this stream (the next layer's statistics) reads
        // nothing this grid writes: let it be scheduled as SMs free up.
        asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
    }
    if (threadIdx.x == 32) {
        for (int s = 0; s < kst; ++s) {
            ptx::mbar_init(&bars->k_full[s], 1);
            ptx::mbar_init(&bars->k_empty[s], 1);
        }
        ptx::mbar_init(&bars->q_full, 1);
        ptx::mbar_init(&bars->q_empty, 1);
        for (int b = 0; b < 4; ++b) {
            ptx::mbar_init(&bars->acc_full[b], 1);
            ptx::mbar_init(&bars->acc_empty[b], 4 * MB);  // one arrival per warp of the group
        }
        for (int c = 0; c < kChunkSlots; ++c) {
            ptx::mbar_init(&bars->c_full[c], 1);
            ptx::mbar_init(&bars->c_empty[c], 2);         // the MMA issuer and the epilogue's leader
        }
        ptx::mbar_init(&bars->mma_done, 1);
        bars->abort_flag = 0;
        ptx::fence_barrier_init();
    }
    if (warp == 1) {
        ptx::tmem_alloc(&bars->tmem_base, kTmemCols);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = bars->tmem_base;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            const uint64_t policy = ptx::policy_evict_normal();   // the window kernel reads K again
            int qloads = 0, issued = 0, it = 0, di = 0;
            for (;;) {
                // Claim a chunk and hand it to the MMA issuer and the epilogue.
                const int c = bars->abort_flag ? nchunks : atomicAdd(claim, 1);
                const int ds = di % kChunkSlots, nd = di / kChunkSlots;
                if (nd > 0 && !ptx::mbar_wait(&bars->c_empty[ds], (nd - 1) & 1)) {
                    raise_abort(bars, sc.err);
                    break;
                }
                bars->chunk[ds] = c < nchunks ? c : -1;
                ptx::mbar_arrive(&bars->c_full[ds]);
                ++di;
                if (c >= nchunks) break;
                const int i0 = c * chunk_items, i1 = min(W, i0 + chunk_items);
                int prev_sh = -1;   // the query rows are loaded again at every chunk's start
                ItemWalker p;
                p.init(cu_dev, G.batch, G.Hkv, i0);
                bool stop = false;
                for (int i = i0; i < i1; ++i, ++it, p.next()) {
                    const int sh = p.s * G.Hkv + p.h;
                    if (sh != prev_sh) {
                        if (qloads > 0 && !ptx::mbar_wait(&bars->q_empty, (qloads - 1) & 1)) {
                            stop = true;
                            break;
                        }
                        ptx::mbar_arrive_expect_tx(&bars->q_full, 2u * R * 128u);
                        ptx::tma_load_4d(sQ, &qmap, &bars->q_full, 0, p.h * G.g, 0, p.s);
                        ptx::tma_load_4d(sQ + Rpad * 128, &qmap, &bars->q_full, 64, p.h * G.g, 0, p.s);
                        ++qloads;
                        prev_sh = sh;
                    }
                    const int st = it % kst, n = it / kst;
                    if (n > 0 && !ptx::mbar_wait(&bars->k_empty[st], (n - 1) & 1)) {
                        stop = true;
                        break;
                    }
                    uint8_t* dst = sK + st * kKStageBytes;
                    const int row = p.row0 + p.j * kTileT;
                    ptx::mbar_arrive_expect_tx(&bars->k_full[st], (uint32_t)kKStageBytes);
                    ptx::tma_load_3d(dst, &kmap, &bars->k_full[st], 0, p.h, row, policy);
                    ptx::tma_load_3d(dst + kKHalfBytes, &kmap, &bars->k_full[st], 64, p.h, row, policy);
                    ++issued;
                }
                if (stop) {
                    raise_abort(bars, sc.err);
                    break;
                }
            }
            // Drain: every issued copy lands before the CTA may exit (stage st was
            // filled ceil((issued - st) / kst) times).
            for (int st = 0; st < kst && st < issued; ++st) {
                const int fills = (issued - st + kst - 1) / kst;
                ptx::mbar_wait(&bars->k_full[st], (fills - 1) & 1, 50000000ull);
            }
            if (qloads > 0) ptx::mbar_wait(&bars->q_full, (qloads - 1) & 1, 50000000ull);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = ptx::idesc_bf16_f32(128, kTileT);
            const uint32_t sQa = ptx::smem_u32(sQ), sKa = ptx::smem_u32(sK);
            int qk = 0, it = 0, di = 0;
            bool stop = false;
            while (!stop && !bars->abort_flag) {
                const int ds = di % kChunkSlots;
                if (!ptx::mbar_wait(&bars->c_full[ds], (di / kChunkSlots) & 1)) {
                    raise_abort(bars, sc.err);
                    break;
                }
                const int c = bars->chunk[ds];
                ptx::mbar_arrive(&bars->c_empty[ds]);
                ++di;
                if (c < 0) break;
                const int i0 = c * chunk_items, i1 = min(W, i0 + chunk_items);
                int prev_sh = -1;
                ItemWalker p;
                p.init(cu_dev, G.batch, G.Hkv, i0);
                for (int i = i0; i < i1 && !bars->abort_flag; ++i, ++it, p.next()) {
                    const int sh = p.s * G.Hkv + p.h;
                    if (sh != prev_sh) {
                        if (!ptx::mbar_wait(&bars->q_full, qk & 1)) {
                            raise_abort(bars, sc.err);
                            stop = true;
                            break;
                        }
                        ++qk;
                        prev_sh = sh;
                    }
                    const int st = it % kst, n = it / kst;
                    const int buf = it % NB, nb = it / NB;
                    if (!ptx::mbar_wait(&bars->k_full[st], n & 1) ||
                        (nb > 0 && !ptx::mbar_wait(&bars->acc_empty[buf], (nb - 1) & 1))) {
                        raise_abort(bars, sc.err);
                        stop = true;
                        break;
                    }
                    ptx::tc_fence_after();
                    const uint32_t kst = sKa + st * kKStageBytes;
                    for (int m = 0; m < MB; ++m) {
                        const uint32_t d = tmem + (uint32_t)(buf * 128 * MB + m * 128);
    #pragma unroll
                        for (int kk = 0; kk < 8; ++kk) {
                            const int half = kk >> 2, kin = kk & 3;
                            const uint64_t ad = ptx::smem_desc_k_sw128(sQa + half * Rpad * 128 + m * 16384 + kin * 32);
                            const uint64_t bd = ptx::smem_desc_k_sw128(kst + half * kKHalfBytes + kin * 32);
                            ptx::mma_bf16(d, ad, bd, idesc, kk > 0 ? 1u : 0u);
                        }
                    }
                    ptx::mma_commit(&bars->k_empty[st]);
                    ptx::mma_commit(&bars->acc_full[buf]);
                    if (i + 1 >= i1 || p.last_of_head()) ptx::mma_commit(&bars->q_empty);
                }
            }
            ptx::mma_commit(&bars->mma_done);
        }
    } else {
        // ------------------------------------------------------------ epilogue
        // NB groups of GW = 4 * MB warps; group a takes the CTA's items a, a + NB,
        // ... from its own accumulator, so the groups work on different items at
        // once (one group's TMEM loads and barrier waits overlap the others' ex2).
        // Warp k of a group reads TMEM lanes 32*(warp % 4) .. +31 (the lane
        // quadrant its warp id allows) of M-block k / 4: one thread per query row,
        // all 128 columns of the item.
        constexpr int GW = 4 * MB;
        const int ew = warp - 2;
        const int grp = ew / GW;
        const int m = (ew % GW) >> 2;
        const int quad = warp & 3;
        const int row = m * 128 + quad * 32 + lane;
        const bool vrow = row < R;
        const int q = vrow ? row / G.g : 0;
        bool aborted = false;
        float seg_m = -INFINITY, seg_z = 0.f;
        int cur_sh = -1, seg_first = 0;

        auto merge = [](float& M, float& Z, float2 o) {
            if (o.x == -INFINITY) return;
            if (o.x > M) {
                Z = Z * ptx::ex2(M - o.x) + o.y;
                M = o.x;
            } else {
                Z += o.y * ptx::ex2(o.x - M);
            }
        };
        // Every epilogue thread calls this at the same segment boundaries (aborted
        // warps included), so the named barriers always complete.  The groups'
        // partials merge here; rowstat_kernel merges the CTAs' partials of a
        // (sequence, head) into (m_r, Z_r).
        auto flush_segment = [&]() {
            bars->xf[grp * Rpad + row] = make_float2(seg_m, seg_z);
            ptx::named_bar_sync(1, kEpiThreads);
            if (grp == 0) {
                float M = seg_m, Z = seg_z;
#pragma unroll
                for (int c = 1; c < NB; ++c) merge(M, Z, bars->xf[c * Rpad + row]);
                if (vrow) sc.segpart[(size_t)seg_first * R + row] = make_float2(M, Z);
            }
            ptx::named_bar_sync(1, kEpiThreads);   // xf is free for the next segment
        };
        // 32 columns of the row, `lim` of them visible (<= 0: none).  Relative to
        // the segment's running reference seg_m, 2^(s - seg_m) sums the same mass
        // as an online max/rescale without a max pass; a chunk far above the
        // reference (sum not below 2^64) and the segment's first chunk take the
        // exact path.
        auto chunk = [&](const float* v, int lim) {
            if (lim <= 0) return;
            if (lim >= 32 && seg_m != -INFINITY) {
                float z4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int c = 0; c < 32; ++c) z4[c & 3] += ptx::ex2(fmaf(v[c], G.sl2, -seg_m));
                const float z = (z4[0] + z4[1]) + (z4[2] + z4[3]);
                if (z < 0x1p64f) {
                    seg_z += z;
                    if (seg_z >= 0x1p40f) {
                        // Keep the sum bounded: move a power of two into the reference.
                        const int k = ilogbf(seg_z);
                        seg_m += (float)k;
                        seg_z = ldexpf(seg_z, -k);
                    }
                    return;
                }
            }
            float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
            for (int c = 0; c < 32; ++c)
                if (c < lim) m4[c & 3] = fmaxf(m4[c & 3], v[c]);
            const float mu = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3])) * G.sl2;
            float z4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int c = 0; c < 32; ++c)
                if (c < lim) z4[c & 3] += ptx::ex2(fmaf(v[c], G.sl2, -mu));
            merge(seg_m, seg_z, make_float2(mu, (z4[0] + z4[1]) + (z4[2] + z4[3])));
        };

        int it = 0, di = 0;
        for (;;) {
            // The epilogue's leader takes the next claimed chunk; the barrier
            // hands it to every epilogue thread (-1: no more work, -2: gave up).
            const int ds = di % kChunkSlots;
            if (threadIdx.x == 64) {
                int c = -2;
                if (ptx::mbar_wait(&bars->c_full[ds], (di / kChunkSlots) & 1)) {
                    c = bars->chunk[ds];
                    ptx::mbar_arrive(&bars->c_empty[ds]);
                } else {
                    raise_abort(bars, sc.err);
                }
                bars->cur_chunk[di & 1] = c;
            }
            ptx::named_bar_sync(1, kEpiThreads);
            const int c = bars->cur_chunk[di & 1];
            ++di;
            if (c < 0) break;
            const int i0 = c * chunk_items, i1 = min(W, i0 + chunk_items);
            ItemWalker p;
            p.init(cu_dev, G.batch, G.Hkv, i0);
            for (int i = i0; i < i1; ++i, ++it, p.next()) {
                const int sh = p.s * G.Hkv + p.h;
                if (sh != cur_sh) {
                    if (cur_sh >= 0) flush_segment();
                    cur_sh = sh;
                    seg_m = -INFINITY;
                    seg_z = 0.f;
                    seg_first = i;
                }
                if (it % NB != grp || aborted) continue;   // another group's item (or keep walking for the barriers)
                const int nb = it / NB;
                int ok = 1;
                if (lane == 0) {
                    ok = !bars->abort_flag && ptx::mbar_wait(&bars->acc_full[grp], nb & 1);
                    if (!ok) raise_abort(bars, sc.err);
                }
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) {
                    aborted = true;
                    continue;
                }
                ptx::tc_fence_after();
                const uint32_t taddr = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(grp * 128 * MB + m * 128);
                const int L = p.L;
                const int t0 = p.j * kTileT;
                const int last = vrow ? min(L - 1, L - G.w + q) : -1;   // causal on the window part
                const int nvalid = max(0, min(kTileT, last - t0 + 1));
                // Four 32-column chunks; the next chunk's TMEM load is in flight while
                // this one is reduced.
                float va[32], vb[32];
                ptx::tmem_ld32(taddr, va);
                ptx::tmem_wait_ld();
                ptx::tmem_ld32(taddr + 32, vb);
                chunk(va, nvalid);
                ptx::tmem_wait_ld();
                ptx::tmem_ld32(taddr + 64, va);
                chunk(vb, nvalid - 32);
                ptx::tmem_wait_ld();
                ptx::tmem_ld32(taddr + 96, vb);
                chunk(va, nvalid - 64);
                ptx::tmem_wait_ld();
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(&bars->acc_empty[grp]);   // the accumulator is in registers
                chunk(vb, nvalid - 96);
            }
            if (cur_sh >= 0) flush_segment();   // a chunk's end closes its last segment
            cur_sh = -1;
        }
    }

    // ---------------------------------------------------------------- teardown
    if (warp == 1 && lane == 0) ptx::mbar_wait(&bars->mma_done, 0, 50000000ull);
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc(tmem, kTmemCols);
}

// (m_r, Z_r) of every row of (s, h) from the score kernel's segment partials:
// one at the head's first item, then one at every chunk boundary inside the
// head's range of items, merged in item order.  Grid (Hkv, batch), one thread
// per row.
__global__ void __launch_bounds__(256) rowstat_kernel(Geometry G, Scratch sc, const int* __restrict__ cu,
                                                      int chunk, int* claim, int wait_prev) {
    // The window launch that follows may start; it waits for this grid.
    if (threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
    // wait_prev: a programmatic dependent of the score launch right before it on
    // the stream, whose partials are read only after that grid has completed.
    // Otherwise the partials come through a full dependency and the stream's
    // previous kernel (if a programmatic predecessor at all) is not waited for.
    if (wait_prev) asm volatile("griddepcontrol.wait;\n" ::: "memory");
    const int h = blockIdx.x, s = blockIdx.y, r = threadIdx.x;
    // The score grid has completed: its chunk counter is free for the next launch.
    if (h == 0 && s == 0 && r == 0) *claim = 0;
    if (r >= G.R) return;
    int ib = 0;
    for (int b = 0; b < s; ++b) ib += tiles_of(__ldg(&cu[b + 1]) - __ldg(&cu[b])) * G.Hkv;
    const int nt = tiles_of(__ldg(&cu[s + 1]) - __ldg(&cu[s]));
    ib += h * nt;
    const int iend = ib + nt;
    float M = -INFINITY, Z = 0.f;
    // Segment starts: the head's first item, then every chunk boundary inside it.
    int next = ib, bnd = (ib / chunk + 1) * chunk;
    while (next < iend) {
        float2 pz[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) {
            pz[k] = make_float2(-INFINITY, 0.f);
            if (next < iend) {
                pz[k] = __ldcg(&sc.segpart[(size_t)next * G.R + r]);
                next = bnd;
                bnd += chunk;
            }
        }
#pragma unroll
        for (int k = 0; k < 16; ++k) {
            const float2 o = pz[k];
            if (o.x == -INFINITY) continue;
            if (o.x > M) {
                Z = Z * ptx::ex2(M - o.x) + o.y;
                M = o.x;
            } else {
                Z += o.y * ptx::ex2(o.x - M);
            }
        }
    }
    sc.rowstat[((size_t)s * G.Hkv + h) * G.R + r] = make_float2(M, Z);
}

// Row statistics from the caller's log-sum-exp of each window query row (the
// denominator its prefill attention already computed): row r = q * g + j of KV
// head h is query head h * g + j at window position q.  Grid (Hkv, batch).
__global__ void __launch_bounds__(256) rowstat_lse_kernel(Geometry G, Scratch sc, const float* __restrict__ lse) {
    // The window launch that follows may start; it waits for this grid before reading.
    if (threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
    const int h = blockIdx.x, s = blockIdx.y, r = threadIdx.x;
    if (r >= G.R) return;
    const int q = r / G.g, j = r - q * G.g;
    const float v = __ldg(&lse[((size_t)s * G.w + q) * G.Hq + h * G.g + j]);
    sc.rowstat[((size_t)s * G.Hkv + h) * G.R + r] = make_float2(v * 1.4426950408889634f, 1.f);
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

int mblocks(const Geometry& g) { return g.R > 128 ? 2 : 1; }

size_t smem_bytes_with(const Geometry& g, int kst) {
    const int MB = mblocks(g);
    return 1024 + 2 * (size_t)MB * 128 * 128 + (size_t)kst * kKStageBytes + sizeof(Barriers);
}

int kstages_for(const Geometry& g) {
    int kst = kKStages;
    while (kst > 2 && smem_bytes_with(g, kst) > (size_t)kMaxSmem) --kst;
    return kst;
}

size_t smem_bytes_for(const Geometry& g) { return smem_bytes_with(g, kstages_for(g)); }

}  // namespace

size_t score_smem_bytes(const Geometry& g) { return smem_bytes_for(g); }

cudaError_t configure_score(const Geometry& g) {
    // Per-function attribute shared by every handle: the largest supported geometry.
    size_t need = 0;
    for (int R = 8; R <= 256; R += 8) {
        Geometry gr = g;
        gr.R = R;
        if (smem_bytes_for(gr) > need) need = smem_bytes_for(gr);
    }
    cudaError_t e = cudaFuncSetAttribute(score_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)need);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(score_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)need);
    return e;
}

cudaError_t plan_score(const Geometry& g, const LayerIO& io, const Scratch& sc, int num_sms, ScorePlan* plan) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    CUtensorMap& kmap = plan->kmap;
    CUtensorMap& qmap = plan->qmap;
    {
        cuuint64_t dims[3] = {(cuuint64_t)kHeadDim, (cuuint64_t)g.Hkv, (cuuint64_t)g.total_tokens};
        cuuint64_t strides[2] = {(cuuint64_t)kHeadDim * 2, (cuuint64_t)g.Hkv * kHeadDim * 2};
        cuuint32_t box[3] = {64, 1, (cuuint32_t)kTileT};
        cuuint32_t es[3] = {1, 1, 1};
        if (enc(&kmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<__nv_bfloat16*>(io.k), dims, strides, box, es,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    {
        cuuint64_t dims[4] = {(cuuint64_t)kHeadDim, (cuuint64_t)g.Hq, (cuuint64_t)g.w, (cuuint64_t)g.batch};
        cuuint64_t strides[3] = {(cuuint64_t)kHeadDim * 2, (cuuint64_t)g.Hq * kHeadDim * 2,
                                 (cuuint64_t)g.w * g.Hq * kHeadDim * 2};
        cuuint32_t box[4] = {64, (cuuint32_t)g.g, (cuuint32_t)g.w, 1};
        cuuint32_t es[4] = {1, 1, 1, 1};
        if (enc(&qmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<__nv_bfloat16*>(io.q), dims, strides, box, es,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    ScoreArgs& a = *reinterpret_cast<ScoreArgs*>(plan->args);
    static_assert(sizeof(ScoreArgs) <= sizeof(plan->args), "ScorePlan::args too small");
    a = ScoreArgs{};
    a.G = g;
    a.cu = io.cu;
    a.sc = sc;
    a.W = g.total_tiles * g.Hkv;
    a.kst = kstages_for(g);
    // At most all but kScoreReserveSms SMs (the rest run the window, heads and
    // selection kernels of neighbouring layers, which cannot share an SM with a
    // score CTA) and at most one CTA per chunk.
    const int usable = num_sms > 2 * kScoreReserveSms ? num_sms - kScoreReserveSms : num_sms;
    // Chunks of kChunkLarge items when that still gives every usable SM one, else
    // of kChunkSmall (measured: larger chunks reload the query rows less often,
    // smaller ones leave fewer SMs idle on small layers).
    a.chunk = a.W / kChunkLarge >= usable ? kChunkLarge : kChunkSmall;
    const int nchunks = (a.W + a.chunk - 1) / a.chunk;
    plan->grid = nchunks < usable ? nchunks : usable;
    plan->chunk = a.chunk;
    plan->threads = kScoreThreads;
    plan->mb = mblocks(g);
    plan->smem = smem_bytes_for(g);
    plan->num_sms = num_sms;
    return cudaSuccess;
}

cudaError_t launch_rowstat(const ScorePlan& plan, const Geometry& g, const LayerIO& io, const Scratch& sc,
                           int* claim, cudaStream_t st, bool programmatic, bool after_score) {
    (void)plan;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(g.Hkv, g.batch);
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = programmatic ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, rowstat_kernel, g, sc, io.cu, plan.chunk, claim, after_score ? 1 : 0);
}

cudaError_t launch_rowstat_lse(const Geometry& g, const LayerIO& io, const Scratch& sc, cudaStream_t st,
                               bool programmatic) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(g.Hkv, g.batch);
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = programmatic ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, rowstat_lse_kernel, g, sc, io.lse);
}

cudaError_t launch_score(const ScorePlan& plan, int* claim, cudaStream_t st, bool after_own_launch) {
    ScoreArgs a = *reinterpret_cast<const ScoreArgs*>(plan.args);
    a.claim = claim;
    // after_own_launch: the previous kernel on the stream is the previous
    // layer's launch, whose results this grid does not read; the launch is then
    // its programmatic dependent and never executes griddepcontrol.wait.
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(plan.grid);
    cfg.blockDim = dim3(plan.threads);
    cfg.dynamicSmemBytes = plan.smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = after_own_launch ? 1 : 0;
    if (plan.mb == 2) return cudaLaunchKernelEx(&cfg, score_kernel<2>, plan.kmap, plan.qmap, a);
    return cudaLaunchKernelEx(&cfg, score_kernel<1>, plan.kmap, plan.qmap, a);
}

}  // namespace kvec
