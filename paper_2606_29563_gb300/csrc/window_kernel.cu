// Eq. 1 window scores, the Section 4.2 importance I, the 1-D max-pool, and the
// per-chunk statistics of pooled P_O that the cross-head sigma needs.
//
// One CTA per (sequence, chunk of kChunk candidate positions).  It rebuilds
// normalised attention A = c_r * e[t][r] from the score kernel's token-major
// e-buffer (c_r = 2^(mu_tile - m_row - 15) / Z_row), for the chunk plus a
// pool-width halo so pooling never crosses CTAs:
//   G_h[q]   = sum_j A[h*g + j, q, t]        (GQA group sum, KV head h)
//   P_O[h,t] = (1/O)  sum_{q >= w-O}  G_h[q]
//   P_O'[h,t]= (1/O') sum_{q >= w-O'} G_h[q]
//   I[t]     = (1/O)  sum_{q >= w-O}  max_h G_h[q]
// A thread owns one (token, KV head); the HP (= next power of two >= Hkv)
// lanes of a token are adjacent, so the head max is an xor-shuffle reduction.
#include "kvec_internal.cuh"

namespace kvec {

namespace {

constexpr int kExt = kChunk + 2 * (kMaxPool / 2);  // chunk + halo on both sides
constexpr int kWindowThreads = 256;

__global__ void __launch_bounds__(kWindowThreads) window_kernel(Geometry G, LayerIO io, Scratch sc, Slot sl,
                                                                 int HP) {
    extern __shared__ float wsm[];
    int s, c, cbase;
    if (!locate_item(G.batch, blockIdx.x,
                     [&](int b) { return chunks_of(io.cu[b + 1] - io.cu[b] - G.w); }, s, c, cbase))
        return;
    const int L = io.cu[s + 1] - io.cu[s];
    const int Lc = L - G.w;
    int tbase = 0;
    for (int b = 0; b < s; ++b) tbase += tiles_of(io.cu[b + 1] - io.cu[b]);
    const int R = G.R, Hkv = G.Hkv;
    const int halo = G.pool / 2;
    const int c_lo = c * kChunk, c_hi = min(Lc, c_lo + kChunk);
    const int t_lo = max(0, c_lo - halo), t_hi = min(Lc, c_hi + halo);
    const int n_ext = t_hi - t_lo;
    const int j0 = t_lo / kTileT, j1 = (t_hi - 1) / kTileT;  // at most two tiles
    const int tid = threadIdx.x;

    float* cfac = wsm;                                   // [2][Hkv][R]
    float* rawO = cfac + 2 * Hkv * R;                    // [Hkv][kExt]
    float* rawOe = rawO + Hkv * kExt;                    // [Hkv][kExt]
    float* rawI = rawOe + Hkv * kExt;                    // [kExt]
    float* poolO = rawI + kExt;                          // [Hkv][kChunk]

    const int ncf = (j1 - j0 + 1) * Hkv * R;
    for (int i = tid; i < ncf; i += kWindowThreads) {
        const int jj = i / (Hkv * R), rem = i - jj * Hkv * R;
        const int hh = rem / R, r = rem - hh * R;
        const float2 ts = sc.tstat[((size_t)(tbase + j0 + jj) * Hkv + hh) * R + r];
        const float2 rs = sc.rowstat[((size_t)s * Hkv + hh) * R + r];
        cfac[i] = exp2f(ts.x - rs.x - kEScaleLog2) / rs.y;
    }
    __syncthreads();

    const int tokens_per_pass = kWindowThreads / HP;
    const float invO = 1.f / G.O, invOe = 1.f / G.Oe;
    for (int base = 0; base < n_ext; base += tokens_per_pass) {
        const int tl = base + tid / HP, hh = tid % HP;
        const bool act = tl < n_ext && hh < Hkv;
        const int t = t_lo + tl;
        const int jt = act ? t / kTileT : j0;
        const __half* erow =
            sc.ebuf + (((size_t)(tbase + jt) * Hkv + (act ? hh : 0)) * kTileT + (act ? t % kTileT : 0)) * R;
        const float* cf = cfac + ((jt - j0) * Hkv + (act ? hh : 0)) * R;
        float accO = 0.f, accOe = 0.f, accI = 0.f, gq = 0.f;
        int jq = 0, q = 0;
        auto finish_row = [&]() {
            if (q >= G.w - G.Oe) accOe += gq;
            if (q >= G.w - G.O) {
                accO += gq;
                float m = gq;
                for (int off = 1; off < HP; off <<= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
                accI += m;
            }
            gq = 0.f;
            jq = 0;
            ++q;
        };
        for (int v8 = 0; v8 < R / 8; ++v8) {
            uint4 raw = make_uint4(0, 0, 0, 0);
            if (act) raw = __ldcg(reinterpret_cast<const uint4*>(erow) + v8);
            const __half2* hv = reinterpret_cast<const __half2*>(&raw);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float2 f = __half22float2(hv[i]);
                gq = fmaf(cf[v8 * 8 + 2 * i], f.x, gq);
                if (++jq == G.g) finish_row();
                gq = fmaf(cf[v8 * 8 + 2 * i + 1], f.y, gq);
                if (++jq == G.g) finish_row();
            }
        }
        if (act) {
            rawO[hh * kExt + tl] = accO * invO;
            rawOe[hh * kExt + tl] = accOe * invOe;
            if (hh == 0) rawI[tl] = accI * invO;
        }
    }
    __syncthreads();

    // Max-pool over [t - halo, t + halo] restricted to the candidates [0, Lc).
    const int nc = c_hi - c_lo;
    for (int i = tid; i < nc * (Hkv + 1); i += kWindowThreads) {
        const int row = i / nc, tt = c_lo + (i - row * nc);
        const int lo = max(tt - halo, 0) - t_lo, hi = min(tt + halo, Lc - 1) - t_lo;
        if (row < Hkv) {
            float mO = rawO[row * kExt + lo], mOe = rawOe[row * kExt + lo];
            for (int x = lo + 1; x <= hi; ++x) {
                mO = fmaxf(mO, rawO[row * kExt + x]);
                mOe = fmaxf(mOe, rawOe[row * kExt + x]);
            }
            sl.PO[((size_t)s * Hkv + row) * G.ML + tt] = mO;
            sl.POe[((size_t)s * Hkv + row) * G.ML + tt] = mOe;
            poolO[row * kChunk + (tt - c_lo)] = mO;
        } else {
            float mI = rawI[lo];
            for (int x = lo + 1; x <= hi; ++x) mI = fmaxf(mI, rawI[x]);
            sl.I[(size_t)s * G.ML + tt] = mI;
        }
    }
    __syncthreads();

    // Chunk mean and sum of squared deviations of pooled P_O (merged with Chan's formula later).
    const int warp = tid >> 5, lane = tid & 31;
    const int nwarps = kWindowThreads / 32;
    const int stride = G.ML / kChunk + 1;
    for (int hh = warp; hh < Hkv; hh += nwarps) {
        float sum = 0.f;
        for (int x = lane; x < nc; x += 32) sum += poolO[hh * kChunk + x];
        for (int off = 16; off; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
        const float mean = sum / nc;
        float m2 = 0.f;
        for (int x = lane; x < nc; x += 32) {
            const float dlt = poolO[hh * kChunk + x] - mean;
            m2 = fmaf(dlt, dlt, m2);
        }
        for (int off = 16; off; off >>= 1) m2 += __shfl_xor_sync(0xffffffffu, m2, off);
        if (lane == 0) sl.sigpart[((size_t)s * Hkv + hh) * stride + c] = make_float2(mean, m2);
    }
}

}  // namespace

size_t window_smem_bytes(const Geometry& g) {
    return sizeof(float) * ((size_t)2 * g.Hkv * g.R + 2 * (size_t)g.Hkv * kExt + kExt + (size_t)g.Hkv * kChunk);
}

cudaError_t configure_window(const Geometry& g) {
    // Per-function attribute shared by every handle: size for the largest geometry
    // accepted by kvec_create (32 KV heads, 256 rows per KV head).
    Geometry widest = g;
    widest.Hkv = 32;
    widest.R = 256;
    return cudaFuncSetAttribute(window_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)window_smem_bytes(widest));
}

void launch_window(const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl, cudaStream_t st) {
    if (g.total_chunks == 0) return;
    int HP = 1;
    while (HP < g.Hkv) HP <<= 1;
    window_kernel<<<g.total_chunks, kWindowThreads, window_smem_bytes(g), st>>>(g, io, sc, sl, HP);
}

}  // namespace kvec
