// Eq. 1 window scores and the Section 4.2 importance I (before pooling).
//
// One CTA per (sequence, 32-token block of candidates).  The score kernel left
// e[tile][h][r][t] = fp16(2^15 exp(s - mu)) row-major; with the row factors
// c_r = 2^(mu_tile,r - m_r - 15) / Z_r the normalised attention is c_r * e.
// A thread owns (8-token group, KV head, subset of window rows q) and issues
// all of its 16-byte row loads before consuming them:
//   G_h[q][t] = sum_j c * e[rows (q, j) of head h][t]     (GQA group sum)
//   P_O[h,t]  = (1/O)  sum_{q >= w-O}  G_h[q][t]
//   P_O'[h,t] = (1/O') sum_{q >= w-O'} G_h[q][t]
//   I[t]      = (1/O)  sum_{q >= w-O}  max_h G_h[q][t]
// The HP (next power of two >= Hkv) lanes of a group are adjacent, so the head
// max is an xor-shuffle; row subsets are summed through shared memory.  The
// raw rows go to the slot arrays; pooling happens in the heads kernel.
#include "kvec_internal.cuh"

namespace kvec {

namespace {

constexpr int kBlockT = 32;                 // candidate tokens per CTA
constexpr int kGroups = kBlockT / 8;        // 8-token groups per CTA
constexpr int kMaxRowsPerThread = 16;       // row loads a thread keeps in flight
constexpr int kMaxWindowThreads = 512;

struct WinShape {
    int HP;       // head lanes per group
    int TPQ;      // threads per row subset: kGroups * HP rounded up to whole warps
    int QS;       // window-row subsets
    int threads;  // TPQ * QS
};

// Every warp lies inside one row subset, so all its lanes run the same q loop
// (the head-max shuffles need the whole warp).  A thread loads its rows in
// batches of kMaxRowsPerThread, all loads of a batch in flight together.
__host__ __device__ inline WinShape win_shape(int Hkv, int w, int g) {
    WinShape s{};
    s.HP = 1;
    while (s.HP < Hkv) s.HP <<= 1;
    s.TPQ = (kGroups * s.HP + 31) & ~31;
    const int qper = kMaxRowsPerThread / g > 0 ? kMaxRowsPerThread / g : 1;   // window rows per subset
    s.QS = (w + qper - 1) / qper;
    if (s.QS * s.TPQ > kMaxWindowThreads) s.QS = kMaxWindowThreads / s.TPQ > 0 ? kMaxWindowThreads / s.TPQ : 1;
    s.threads = s.TPQ * s.QS;
    return s;
}

__device__ __forceinline__ void unpack8(const uint4& raw, float* f) {
    const __half2* h = reinterpret_cast<const __half2*>(&raw);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 x = __half22float2(h[i]);
        f[2 * i] = x.x;
        f[2 * i + 1] = x.y;
    }
}

template <int HP>
__global__ void __launch_bounds__(kMaxWindowThreads) window_kernel(Geometry G, LayerIO io, Scratch sc, Slot sl) {
    extern __shared__ float wsm[];
    const WinShape ws = win_shape(G.Hkv, G.w, G.g);
    int s, blk, base;
    if (!locate_item(G.batch, blockIdx.x,
                     [&](int b) {
                         const int Lc = io.cu[b + 1] - io.cu[b] - G.w;
                         return Lc > 0 ? (Lc + kBlockT - 1) / kBlockT : 0;
                     },
                     s, blk, base))
        return;
    const int L = io.cu[s + 1] - io.cu[s];
    const int Lc = L - G.w;
    int tbase = 0;
    for (int b = 0; b < s; ++b) tbase += tiles_of(io.cu[b + 1] - io.cu[b]);
    const int R = G.R, Hkv = G.Hkv;
    const int t0 = blk * kBlockT;
    const int jt = t0 / kTileT, toff0 = t0 - jt * kTileT;
    const int tid = threadIdx.x;
    const int qper = (G.w + ws.QS - 1) / ws.QS;

    float* cfac = wsm;                                          // [Hkv][R]
    float* part = cfac + Hkv * R;                               // [QS][kBlockT][Hkv][3]

    {
        // Row factors of this tile, four loads in flight per thread.
        const int n = Hkv * R;
        for (int i0 = tid; i0 < n; i0 += 4 * blockDim.x) {
            float2 ts[4], rs[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int i = i0 + u * blockDim.x;
                if (i < n) {
                    const int hh = i / R, r = i - hh * R;
                    ts[u] = sc.tstat[((size_t)(tbase + jt) * Hkv + hh) * R + r];
                    rs[u] = sc.rowstat[((size_t)s * Hkv + hh) * R + r];
                }
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int i = i0 + u * blockDim.x;
                if (i < n) cfac[i] = exp2f(ts[u].x - rs[u].x - kEScaleLog2) / rs[u].y;
            }
        }
    }
    __syncthreads();

    // Thread role: row subset (whole warps), then group, then head lane (adjacent lanes).
    const int qs = tid / ws.TPQ;
    const int local = tid - qs * ws.TPQ;
    const int hh = local % HP;
    const int grp = local / HP;
    const int t8 = t0 + grp * 8;
    const bool act = grp < kGroups && hh < Hkv && t8 < Lc;
    const __half* ebase = sc.ebuf + ((size_t)(tbase + jt) * Hkv + (act ? hh : 0)) * R * kTileT + toff0 + grp * 8;
    const float* cf = cfac + (act ? hh : 0) * R;
    const int q_lo = min(qs * qper, G.w), q_hi = min(q_lo + qper, G.w);
    const int r_end = q_hi * G.g;

    float accO[8], accOe[8], accI[8], gsum[8];
#pragma unroll
    for (int x = 0; x < 8; ++x) accO[x] = accOe[x] = accI[x] = gsum[x] = 0.f;
    int q = q_lo, jq = 0;
    for (int r0 = q_lo * G.g; r0 < r_end; r0 += kMaxRowsPerThread) {
        const int nrows = min(kMaxRowsPerThread, r_end - r0);
        uint4 raw[kMaxRowsPerThread];
#pragma unroll
        for (int k = 0; k < kMaxRowsPerThread; ++k) {
            raw[k] = make_uint4(0, 0, 0, 0);
            if (act && k < nrows) raw[k] = __ldcg(reinterpret_cast<const uint4*>(ebase + (size_t)(r0 + k) * kTileT));
        }
#pragma unroll
        for (int k = 0; k < kMaxRowsPerThread; ++k) {
            if (k >= nrows) break;
            float f[8];
            unpack8(raw[k], f);
            const float c = cf[r0 + k];
#pragma unroll
            for (int x = 0; x < 8; ++x) gsum[x] = fmaf(c, f[x], gsum[x]);
            if (++jq == G.g) {
                if (q >= G.w - G.Oe) {
#pragma unroll
                    for (int x = 0; x < 8; ++x) accOe[x] += gsum[x];
                }
                if (q >= G.w - G.O) {
#pragma unroll
                    for (int x = 0; x < 8; ++x) {
                        float m = gsum[x];
#pragma unroll
                        for (int off = 1; off < HP; off <<= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
                        accO[x] += gsum[x];
                        accI[x] += m;
                    }
                }
#pragma unroll
                for (int x = 0; x < 8; ++x) gsum[x] = 0.f;
                jq = 0;
                ++q;
            }
        }
    }
    if (grp < kGroups && hh < Hkv) {
#pragma unroll
        for (int x = 0; x < 8; ++x) {
            float* pp = part + (((size_t)qs * kBlockT + grp * 8 + x) * Hkv + hh) * 3;
            pp[0] = accO[x];
            pp[1] = accOe[x];
            pp[2] = accI[x];
        }
    }
    __syncthreads();

    // Sum the row subsets and write the raw rows (positions of one head are consecutive).
    const float invO = 1.f / G.O, invOe = 1.f / G.Oe;
    for (int i = tid; i < kBlockT * Hkv; i += blockDim.x) {
        const int h2 = i / kBlockT, x = i - h2 * kBlockT;
        const int t = t0 + x;
        if (t >= Lc) continue;
        float o = 0.f, oe = 0.f, im = 0.f;
        for (int qq = 0; qq < ws.QS; ++qq) {
            const float* pp = part + (((size_t)qq * kBlockT + x) * Hkv + h2) * 3;
            o += pp[0];
            oe += pp[1];
            im += pp[2];
        }
        sl.rawO[((size_t)s * Hkv + h2) * G.ML + t] = o * invO;
        sl.rawOe[((size_t)s * Hkv + h2) * G.ML + t] = oe * invOe;
        if (h2 == 0) sl.rawI[(size_t)s * G.ML + t] = im * invO;
    }
}

template <int HP>
void launch_hp(const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl, cudaStream_t st) {
    const WinShape ws = win_shape(g.Hkv, g.w, g.g);
    window_kernel<HP><<<g.total_chunks, ws.threads, window_smem_bytes(g), st>>>(g, io, sc, sl);
}

template <int HP>
cudaError_t configure_hp(size_t bytes) {
    return cudaFuncSetAttribute(window_kernel<HP>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

}  // namespace

int window_blocks(int Lc) { return Lc > 0 ? (Lc + kBlockT - 1) / kBlockT : 0; }

int window_threads(const Geometry& g) { return win_shape(g.Hkv, g.w, g.g).threads; }

size_t window_smem_bytes(const Geometry& g) {
    const WinShape ws = win_shape(g.Hkv, g.w, g.g);
    return sizeof(float) * ((size_t)g.Hkv * g.R + (size_t)ws.QS * kBlockT * g.Hkv * 3);
}

cudaError_t configure_window(const Geometry& g) {
    // Per-function attributes shared by every handle: the largest geometry kvec_create accepts.
    size_t need = 0;
    for (int h = 1; h <= 32; ++h)
        for (int gg = 1; gg <= 256; ++gg) {
            Geometry t = g;
            t.Hkv = h;
            t.g = gg;
            t.w = 256 / gg;
            t.R = t.g * t.w;
            const size_t b = window_smem_bytes(t);
            if (b > need) need = b;
        }
    cudaError_t e = configure_hp<1>(need);
    if (e == cudaSuccess) e = configure_hp<2>(need);
    if (e == cudaSuccess) e = configure_hp<4>(need);
    if (e == cudaSuccess) e = configure_hp<8>(need);
    if (e == cudaSuccess) e = configure_hp<16>(need);
    if (e == cudaSuccess) e = configure_hp<32>(need);
    return e;
}

void launch_window(const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl, cudaStream_t st) {
    if (g.total_chunks == 0) return;
    const WinShape ws = win_shape(g.Hkv, g.w, g.g);
    switch (ws.HP) {
        case 1: launch_hp<1>(g, io, sc, sl, st); break;
        case 2: launch_hp<2>(g, io, sc, sl, st); break;
        case 4: launch_hp<4>(g, io, sc, sl, st); break;
        case 8: launch_hp<8>(g, io, sc, sl, st); break;
        case 16: launch_hp<16>(g, io, sc, sl, st); break;
        default: launch_hp<32>(g, io, sc, sl, st); break;
    }
}

}  // namespace kvec
