// Window-query scores against every prefix key: s = <q_obs, k_t> for the w
// observation rows of each query head (Eq. 1's A before normalisation), with the
// softmax split into per-tile partials (Section 4.1 needs A normalised over all
// visible keys, so the normalisation is finished by rowstat_kernel).
//
// One CTA per (128-token tile, KV head).  The g*w query rows of the KV head
// (r = q*g + j) form the M side of bf16 tensor-core MMAs, the tile's keys the
// N side; every accumulator row stays inside one warp, so the tile max and the
// partial sum need only quad shuffles.  The kernel writes
//   ebuf[tile][h][t][r] = fp16(2^15 * exp(s - mu_tile,r))   (token-major)
//   tstat[tile][h][r]   = (mu_tile,r in log2 units, sum_t exp(s - mu_tile,r))
#include "kvec_internal.cuh"

namespace kvec {

namespace {

constexpr int kRowBytes = 272;  // 128 bf16 + 16 B pad: conflict-free ldmatrix rows

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, int src_bytes) {
    uint32_t s = static_cast<uint32_t>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(s), "l"(gmem), "r"(src_bytes));
}

__device__ __forceinline__ void ldmatrix_x4(uint32_t* r, const void* p) {
    uint32_t a = static_cast<uint32_t>(__cvta_generic_to_shared(p));
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(a));
}

__device__ __forceinline__ void mma_bf16_16816(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__global__ void __launch_bounds__(512, 1) score_kernel(Geometry G, LayerIO io, Scratch sc) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int h = blockIdx.y;
    const int gt = blockIdx.x;
    int s, j, tbase;
    if (!locate_item(G.batch, gt, [&](int b) { return tiles_of(io.cu[b + 1] - io.cu[b]); }, s, j, tbase))
        return;
    const int L = io.cu[s + 1] - io.cu[s];
    const int t0 = j * kTileT;
    const int R = G.R;
    const int R16 = (R + 15) & ~15;
    uint8_t* sQ = smem;
    uint8_t* sK = smem + (size_t)R16 * kRowBytes;
    const int tid = threadIdx.x, nthr = blockDim.x;

    for (int i = tid; i < R16 * 16; i += nthr) {
        const int r = i >> 4, c = i & 15;
        const __nv_bfloat16* src = io.q;
        int bytes = 0;
        if (r < R) {
            const int q = r / G.g, jj = r - q * G.g;
            src = io.q + (((size_t)s * G.w + q) * G.Hq + h * G.g + jj) * kHeadDim + c * 8;
            bytes = 16;
        }
        cp_async16(sQ + r * kRowBytes + c * 16, src, bytes);
    }
    for (int i = tid; i < kTileT * 16; i += nthr) {
        const int t = i >> 4, c = i & 15;
        const __nv_bfloat16* src = io.k;
        int bytes = 0;
        if (t0 + t < L) {
            src = io.k + (((size_t)io.cu[s] + t0 + t) * G.Hkv + h) * kHeadDim + c * 8;
            bytes = 16;
        }
        cp_async16(sK + t * kRowBytes + c * 16, src, bytes);
    }
    asm volatile("cp.async.commit_group;\n");
    asm volatile("cp.async.wait_all;\n" ::: "memory");
    __syncthreads();

    const int warp = tid >> 5, lane = tid & 31;
    const int r0 = warp * 16;
    uint32_t a[8][4];
#pragma unroll
    for (int ks = 0; ks < 8; ++ks)
        ldmatrix_x4(a[ks], sQ + (r0 + (lane & 7) + ((lane >> 3) & 1) * 8) * kRowBytes + (ks * 16 + (lane >> 4) * 8) * 2);

    float acc[16][4];
#pragma unroll
    for (int n = 0; n < 16; ++n) acc[n][0] = acc[n][1] = acc[n][2] = acc[n][3] = 0.f;
#pragma unroll
    for (int np = 0; np < 8; ++np) {
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
            uint32_t b[4];
            ldmatrix_x4(b, sK + (np * 16 + (lane & 7) + (lane >> 4) * 8) * kRowBytes +
                               (ks * 16 + ((lane >> 3) & 1) * 8) * 2);
            mma_bf16_16816(acc[2 * np], a[ks], b[0], b[1]);
            mma_bf16_16816(acc[2 * np + 1], a[ks], b[2], b[3]);
        }
    }
    __syncthreads();  // Q and K tiles are dead: the e-tile reuses their shared memory

    const int gid = lane >> 2, tq = lane & 3;
    const int rA = r0 + gid, rB = rA + 8;
    // Last key visible to a row: causal for the window part (row q sits at L - w + q).
    const int lastA = rA < R ? min(L - 1, L - G.w + rA / G.g) : -1;
    const int lastB = rB < R ? min(L - 1, L - G.w + rB / G.g) : -1;
    float mA = -INFINITY, mB = -INFINITY;
#pragma unroll
    for (int n = 0; n < 16; ++n)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const int tok = t0 + n * 8 + 2 * tq + e;
            if (tok <= lastA) mA = fmaxf(mA, acc[n][e]);
            if (tok <= lastB) mB = fmaxf(mB, acc[n][2 + e]);
        }
    mA = fmaxf(mA, __shfl_xor_sync(0xffffffffu, mA, 1));
    mA = fmaxf(mA, __shfl_xor_sync(0xffffffffu, mA, 2));
    mB = fmaxf(mB, __shfl_xor_sync(0xffffffffu, mB, 1));
    mB = fmaxf(mB, __shfl_xor_sync(0xffffffffu, mB, 2));
    const float muA = mA * G.sl2, muB = mB * G.sl2;  // -inf when no key of the tile is visible
    __half* sE = reinterpret_cast<__half*>(smem);    // [kTileT][R]
    float zA = 0.f, zB = 0.f;
#pragma unroll
    for (int n = 0; n < 16; ++n)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const int tl = n * 8 + 2 * tq + e;
            const int tok = t0 + tl;
            const float eA = tok <= lastA ? exp2f(fmaf(acc[n][e], G.sl2, -muA)) : 0.f;
            const float eB = tok <= lastB ? exp2f(fmaf(acc[n][2 + e], G.sl2, -muB)) : 0.f;
            zA += eA;
            zB += eB;
            if (rA < R) sE[tl * R + rA] = __float2half_rn(eA * 32768.f);
            if (rB < R) sE[tl * R + rB] = __float2half_rn(eB * 32768.f);
        }
    zA += __shfl_xor_sync(0xffffffffu, zA, 1);
    zA += __shfl_xor_sync(0xffffffffu, zA, 2);
    zB += __shfl_xor_sync(0xffffffffu, zB, 1);
    zB += __shfl_xor_sync(0xffffffffu, zB, 2);
    float2* ts = sc.tstat + ((size_t)gt * G.Hkv + h) * R;
    if (tq == 0) {
        if (rA < R) ts[rA] = make_float2(muA, zA);
        if (rB < R) ts[rB] = make_float2(muB, zB);
    }
    __syncthreads();
    const uint4* src = reinterpret_cast<const uint4*>(sE);
    uint4* dst = reinterpret_cast<uint4*>(sc.ebuf + ((size_t)gt * G.Hkv + h) * kTileT * R);
    const int n16 = kTileT * R / 8;
    for (int i = tid; i < n16; i += nthr) dst[i] = src[i];
}

// Merges the per-tile (mu, z) partials of every window row into the row's
// softmax max and denominator.  Grid (ceil(R/32), Hkv, batch), 256 threads:
// a lane owns a row, the 8 warps stride over tiles, shared memory combines them.
__global__ void __launch_bounds__(256) rowstat_kernel(Geometry G, LayerIO io, Scratch sc) {
    __shared__ float2 part[8][32];
    const int s = blockIdx.z, h = blockIdx.y;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int r = blockIdx.x * 32 + lane;
    int tbase = 0;
    for (int b = 0; b < s; ++b) tbase += tiles_of(io.cu[b + 1] - io.cu[b]);
    const int nt = tiles_of(io.cu[s + 1] - io.cu[s]);
    float m = -INFINITY, z = 0.f;
    if (r < G.R) {
        for (int jt = warp; jt < nt; jt += 8) {
            const float2 t = sc.tstat[((size_t)(tbase + jt) * G.Hkv + h) * G.R + r];
            if (t.x == -INFINITY) continue;
            if (t.x > m) {
                z = z * exp2f(m - t.x) + t.y;
                m = t.x;
            } else {
                z += t.y * exp2f(t.x - m);
            }
        }
    }
    part[warp][lane] = make_float2(m, z);
    __syncthreads();
    if (warp == 0 && r < G.R) {
        float M = -INFINITY;
        for (int w8 = 0; w8 < 8; ++w8) M = fmaxf(M, part[w8][lane].x);
        float Z = 0.f;
        for (int w8 = 0; w8 < 8; ++w8)
            if (part[w8][lane].x != -INFINITY) Z += part[w8][lane].y * exp2f(part[w8][lane].x - M);
        sc.rowstat[((size_t)s * G.Hkv + h) * G.R + r] = make_float2(M, Z);
    }
}

}  // namespace

size_t score_smem_bytes(const Geometry& g) {
    const int R16 = (g.R + 15) & ~15;
    size_t mma = (size_t)(R16 + kTileT) * kRowBytes;
    size_t etile = (size_t)kTileT * g.R * sizeof(__half);
    return mma > etile ? mma : etile;
}

cudaError_t configure_score(const Geometry& g) {
    // The attribute is per function, shared by every handle: request the largest
    // size any supported geometry (rows per KV head <= 256) can need.
    Geometry widest = g;
    widest.R = 256;
    size_t need = score_smem_bytes(widest);
    if (score_smem_bytes(g) > need) need = score_smem_bytes(g);
    return cudaFuncSetAttribute(score_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)need);
}

void launch_score(const Geometry& g, const LayerIO& io, const Scratch& sc, cudaStream_t st) {
    const int R16 = (g.R + 15) & ~15;
    dim3 grid(g.total_tiles, g.Hkv);
    score_kernel<<<grid, (R16 / 16) * 32, score_smem_bytes(g), st>>>(g, io, sc);
}

void launch_rowstat(const Geometry& g, const LayerIO& io, const Scratch& sc, cudaStream_t st) {
    dim3 grid((g.R + 31) / 32, g.Hkv, g.batch);
    rowstat_kernel<<<grid, 256, 0, st>>>(g, io, sc);
}

}  // namespace kvec
