// Cross-head choice, preserved tokens, coverage-adjusted top-B and the
// coverage-state update (Section 4.1, Section 4.2, Algorithm 1), plus the K/V
// gather into the budget-sized cache.
//
// Top-k is an exact block-wide MSB radix select over order-preserving uint32
// keys (11/11/10-bit digits, shared-memory histograms, block scans built from
// warp shuffles and ballots).  Ties at the threshold go to the lower position.
#include "kvec_internal.cuh"

namespace kvec {

namespace {

struct TopkShared {
    int hist[2048];
    int wsum[32];
    int bcast[4];
};

// Exclusive prefix sum over the block (blockDim.x a multiple of 32, <= 1024).
__device__ int block_exclusive_sum(int v, int* wsum, int& total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int x = v;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, off);
        if (lane >= off) x += y;
    }
    if (lane == 31) wsum[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int ws = lane < nw ? wsum[lane] : 0;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, ws, off);
            if (lane >= off) ws += y;
        }
        wsum[lane] = ws;
    }
    __syncthreads();
    const int before = warp ? wsum[warp - 1] : 0;
    total = wsum[nw - 1];
    __syncthreads();
    return before + x - v;
}

// ORs into bits[] (shared, one bit per position) the k largest keys of keys[0, n).
// Key 0 marks an ineligible position; the caller guarantees k <= #eligible.
__device__ void block_topk(const uint32_t* __restrict__ keys, int n, int k, uint32_t* bits, TopkShared& sm) {
    if (k <= 0 || n <= 0) return;
    const int tid = threadIdx.x, NT = blockDim.x;
    uint32_t prefix = 0, mask = 0;
    int kk = k;
    bool whole_bin = false;
    for (int pass = 0; pass < 3; ++pass) {
        const int sh = pass == 0 ? 21 : (pass == 1 ? 10 : 0);
        const int nb = pass == 2 ? 1024 : 2048;
        for (int i = tid; i < nb; i += NT) sm.hist[i] = 0;
        __syncthreads();
        for (int t = tid; t < n; t += NT) {
            const uint32_t u = keys[t];
            if (u != 0u && (u & mask) == prefix) atomicAdd(&sm.hist[(u >> sh) & (nb - 1)], 1);
        }
        __syncthreads();
        // Thread i owns the i-th block of bins counted from the top.
        const int bpt = (nb + NT - 1) / NT;
        const int hi = nb - tid * bpt, lo = max(hi - bpt, 0);
        int mine = 0;
        for (int b = lo; b < hi; ++b) mine += sm.hist[b];
        int total;
        const int above_me = block_exclusive_sum(mine, sm.wsum, total);
        if (hi > 0 && above_me < kk && above_me + mine >= kk) {
            int acc = above_me;
            for (int b = hi - 1; b >= lo; --b) {
                if (acc + sm.hist[b] >= kk) {
                    sm.bcast[0] = b;
                    sm.bcast[1] = acc;
                    sm.bcast[2] = sm.hist[b];
                    break;
                }
                acc += sm.hist[b];
            }
        }
        __syncthreads();
        const int D = sm.bcast[0], above = sm.bcast[1], cnt = sm.bcast[2];
        __syncthreads();
        prefix |= (uint32_t)D << sh;
        mask |= (uint32_t)(nb - 1) << sh;
        kk -= above;
        if (cnt == kk) {
            whole_bin = true;
            break;
        }
    }
    // Positions strictly above the threshold prefix are in; positions equal to it
    // are in either all together or, when equal keys exceed the need, lowest first.
    const int nchunks = (n + NT - 1) / NT;
    int taken = 0;
    for (int ch = 0; ch < nchunks; ++ch) {
        const int t = ch * NT + tid;
        const uint32_t u = t < n ? keys[t] : 0u;
        const bool above = u != 0u && (u & mask) > prefix;
        const bool eq = u != 0u && (u & mask) == prefix;
        bool sel;
        if (whole_bin) {
            sel = above || eq;
        } else {
            int tot;
            const int r = block_exclusive_sum(eq ? 1 : 0, sm.wsum, tot);
            sel = above || (eq && taken + r < kk);
            taken += tot;
        }
        const unsigned bal = __ballot_sync(0xffffffffu, sel);
        if ((tid & 31) == 0 && bal) bits[(ch * NT + (tid & ~31)) >> 5] |= bal;
    }
    __syncthreads();
}

__device__ __forceinline__ uint32_t range_bits(int word, int lo, int hi) {
    // Bits of `word` covering positions in [lo, hi).
    const int b0 = word * 32;
    const int a = max(lo - b0, 0), e = min(hi - b0, 32);
    if (e <= a) return 0u;
    const uint32_t upto = e == 32 ? 0xffffffffu : ((1u << e) - 1u);
    return upto & ~((1u << a) - 1u);
}

// Section 4.1: sigma of every head (Chan merge of chunk statistics), the delta
// lowest-sigma heads take the O' scores; then the top-K preserved tokens by P
// (Section 4.2).  Grid (Hkv, batch).
__global__ void __launch_bounds__(kSelectThreads) heads_kernel(Geometry G, LayerIO io, Scratch sc, Slot sl) {
    __shared__ TopkShared sm;
    __shared__ double sig[32];
    extern __shared__ uint32_t bits[];
    const int h = blockIdx.x, s = blockIdx.y;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int L = io.cu[s + 1] - io.cu[s];
    const int Lc = L - G.w;
    const int nch = chunks_of(Lc);
    const int stride = G.ML / kChunk + 1;
    if (warp < G.Hkv) {
        const float2* part = sl.sigpart + ((size_t)s * G.Hkv + warp) * stride;
        double cnt = 0.0, sx = 0.0;
        for (int c = lane; c < nch; c += 32) {
            const int nc = min(kChunk, Lc - c * kChunk);
            cnt += nc;
            sx += nc * (double)part[c].x;
        }
        for (int off = 16; off; off >>= 1) {
            cnt += __shfl_xor_sync(0xffffffffu, cnt, off);
            sx += __shfl_xor_sync(0xffffffffu, sx, off);
        }
        const double mean = cnt > 0.0 ? sx / cnt : 0.0;
        double m2 = 0.0;
        for (int c = lane; c < nch; c += 32) {
            const int nc = min(kChunk, Lc - c * kChunk);
            const double dm = (double)part[c].x - mean;
            m2 += (double)part[c].y + nc * dm * dm;
        }
        for (int off = 16; off; off >>= 1) m2 += __shfl_xor_sync(0xffffffffu, m2, off);
        if (lane == 0) sig[warp] = cnt >= 2.0 ? sqrt(m2 / (cnt - 1.0)) : 0.0;
    }
    for (int wd = tid; wd < G.words; wd += blockDim.x) bits[wd] = 0u;
    __syncthreads();
    int rank = 0;
    for (int o = 0; o < G.Hkv; ++o)
        if (sig[o] < sig[h] || (sig[o] == sig[h] && o < h)) ++rank;
    const int top = rank < G.delta;
    if (tid == 0) {
        sl.sigma[(size_t)s * G.Hkv + h] = (float)sig[h];
        sl.htop[(size_t)s * G.Hkv + h] = top;
    }
    if (L > G.budget && G.Kp > 0) {
        const float* P = (top ? sl.POe : sl.PO) + ((size_t)s * G.Hkv + h) * G.ML;
        uint32_t* keys = sc.keys + ((size_t)s * G.Hkv + h) * G.ML;
        for (int t = tid; t < Lc; t += blockDim.x) keys[t] = float_order_key(P[t]);
        __syncthreads();
        block_topk(keys, Lc, G.Kp, bits, sm);
    }
    uint32_t* pres = sl.pres + ((size_t)s * G.Hkv + h) * G.words;
    for (int wd = tid; wd < G.words; wd += blockDim.x) pres[wd] = bits[wd];
}

// Section 4.2: P' = P + lambda * I * (1 - n_t / (l + 1)); the preserved tokens
// stay, the rest of B - w goes to the largest P'; the last w tokens are kept.
// Writes out_idx (ascending) and folds the union of all heads into n_t once the
// last head of the sequence is done.  Grid (Hkv, batch).
__global__ void __launch_bounds__(kSelectThreads) select_kernel(Geometry G, LayerIO io, Scratch sc, Slot sl) {
    __shared__ TopkShared sm;
    __shared__ int last_head;
    extern __shared__ uint32_t bits[];
    const int h = blockIdx.x, s = blockIdx.y;
    const int tid = threadIdx.x, NT = blockDim.x;
    const int L = io.cu[s + 1] - io.cu[s];
    const int Lc = L - G.w;
    const int wordsL = (L + 31) >> 5;
    uint8_t* st = io.state + (size_t)s * G.state_stride;
    const uint32_t ell = reinterpret_cast<const uint32_t*>(st)[0];
    uint8_t* ncount = st + G.state_n_off;
    if (ell >= 255u) {  // n_t is 8-bit: a state that already saw 255 layers cannot count another
        if (tid == 0) atomicExch(sc.err, 2);
        return;
    }
    for (int wd = tid; wd < G.words; wd += NT) bits[wd] = 0u;
    __syncthreads();
    if (L > G.budget) {
        const size_t row = (size_t)s * G.Hkv + h;
        const int top = sl.htop[row];
        const float* P = (top ? sl.POe : sl.PO) + row * G.ML;
        const float* I = sl.I + (size_t)s * G.ML;
        const uint32_t* pres = sl.pres + row * G.words;
        float* Pp = sl.Pprime + row * G.ML;
        uint32_t* keys = sc.keys + row * G.ML;
        const float denom = (float)(ell + 1u);
        for (int t = tid; t < Lc; t += NT) {
            const float coverage = (float)ncount[t] / denom;
            const float pp = P[t] + G.lambda * (I[t] * (1.f - coverage));
            Pp[t] = pp;
            const bool kept = (pres[t >> 5] >> (t & 31)) & 1u;
            keys[t] = kept ? 0u : float_order_key(pp);
        }
        __syncthreads();
        block_topk(keys, Lc, G.k2, bits, sm);
        for (int wd = tid; wd < wordsL; wd += NT) bits[wd] |= pres[wd] | range_bits(wd, Lc, L);
    } else {
        for (int wd = tid; wd < wordsL; wd += NT) bits[wd] = range_bits(wd, 0, L);
    }
    __syncthreads();

    // Ascending positions: each thread owns a contiguous run of words.
    int32_t* oi = io.out_idx + ((size_t)s * G.Hkv + h) * G.budget;
    const int wpt = (wordsL + NT - 1) / NT;
    const int w_lo = min(tid * wpt, wordsL), w_hi = min(w_lo + wpt, wordsL);
    int mine = 0;
    for (int wd = w_lo; wd < w_hi; ++wd) mine += __popc(bits[wd]);
    int total;
    int pos = block_exclusive_sum(mine, sm.wsum, total);
    for (int wd = w_lo; wd < w_hi; ++wd) {
        uint32_t b = bits[wd];
        while (b) {
            const int bit = __ffs(b) - 1;
            b &= b - 1u;
            if (pos < G.budget) oi[pos] = wd * 32 + bit;
            ++pos;
        }
    }
    for (int j = total + tid; j < G.budget; j += NT) oi[j] = -1;

    // Union over heads, then the last head of the sequence updates n_t (Section 4.2).
    uint32_t* ub = sc.ubits + (size_t)s * G.words;
    for (int wd = tid; wd < wordsL; wd += NT)
        if (bits[wd]) atomicOr(&ub[wd], bits[wd]);
    __threadfence();
    __syncthreads();
    if (tid == 0) last_head = atomicAdd(&sc.ucount[s], 1u) == (unsigned)(G.Hkv - 1);
    __syncthreads();
    if (!last_head) return;
    __threadfence();
    for (int t = tid; t < L; t += NT) {
        const uint32_t wv = __ldcg(&ub[t >> 5]);
        if ((wv >> (t & 31)) & 1u) ncount[t] = (uint8_t)(ncount[t] + 1u);
    }
    __syncthreads();
    uint32_t* last_union = reinterpret_cast<uint32_t*>(st + G.state_union_off);
    for (int wd = tid; wd < G.words; wd += NT) {
        last_union[wd] = __ldcg(&ub[wd]);
        ub[wd] = 0u;
    }
    if (tid == 0) {
        reinterpret_cast<uint32_t*>(st)[0] = ell + 1u;
        reinterpret_cast<uint32_t*>(st)[1] = (uint32_t)L;
        sc.ucount[s] = 0u;
    }
}

// out_k[s,h,j,:] = K[cu[s] + idx[s,h,j], h, :] (zeros for idx = -1); the same for V.
// Grid (ceil(B/16), Hkv, batch), 256 threads: a half-warp moves one 256-byte row.
__global__ void __launch_bounds__(256) gather_kernel(Geometry G, LayerIO io) {
    const int s = blockIdx.z, h = blockIdx.y;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int row = blockIdx.x * 16 + warp * 2 + (lane >> 4), sub = lane & 15;
    if (row >= G.budget) return;
    const size_t orow = ((size_t)s * G.Hkv + h) * G.budget + row;
    const int idx = io.out_idx[orow];
    const int L = io.cu[s + 1] - io.cu[s];
    uint4 kv = make_uint4(0, 0, 0, 0), vv = make_uint4(0, 0, 0, 0);
    if (idx >= 0 && idx < L) {
        const size_t src = (((size_t)io.cu[s] + idx) * G.Hkv + h) * kHeadDim + sub * 8;
        kv = __ldg(reinterpret_cast<const uint4*>(io.k + src));
        vv = __ldg(reinterpret_cast<const uint4*>(io.v + src));
    }
    reinterpret_cast<uint4*>(io.out_k + orow * kHeadDim)[sub] = kv;
    reinterpret_cast<uint4*>(io.out_v + orow * kHeadDim)[sub] = vv;
}

}  // namespace

void launch_heads(const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl, cudaStream_t st) {
    heads_kernel<<<dim3(g.Hkv, g.batch), kSelectThreads, g.words * sizeof(uint32_t), st>>>(g, io, sc, sl);
}

void launch_select(const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl, cudaStream_t st) {
    select_kernel<<<dim3(g.Hkv, g.batch), kSelectThreads, g.words * sizeof(uint32_t), st>>>(g, io, sc, sl);
}

void launch_gather(const Geometry& g, const LayerIO& io, cudaStream_t st) {
    gather_kernel<<<dim3((g.budget + 15) / 16, g.Hkv, g.batch), 256, 0, st>>>(g, io);
}

}  // namespace kvec
