// Cross-head choice, preserved tokens, coverage-adjusted top-B and the
// coverage-state update (Section 4.1, Section 4.2, Algorithm 1), plus the K/V
// gather into the budget-sized cache.
//
// Top-k is an exact MSB radix select over order-preserving uint32 keys (bits
// shared by all keys skipped, 4-bit digits counted in registers, one barrier
// per digit, small threshold buckets compacted and ranked directly).  Ties at
// the threshold go to the lower position.
#include "kvec_internal.cuh"

namespace kvec {

namespace {

constexpr int kSmemKeys = 40960;   // positions whose keys fit in shared memory (160 KB)

__host__ __device__ inline bool keys_in_smem(int ML) { return ML <= kSmemKeys; }

constexpr int kSmemScores = 16448;  // row stride up to which the select kernel caches P and I in shared memory
__host__ __device__ inline bool scores_in_smem(int ML) { return ML <= kSmemScores; }

// Key rows are stored in position order in 16-byte chunks of four keys, chunk c
// at c ^ ((c >> 3) & 7): a radix-select lane reads its 16 consecutive keys as
// four 16-byte loads, and the eight lanes of a quarter-warp (64 bytes apart)
// then hit eight different 16-byte bank groups, as do eight threads storing
// eight consecutive chunks.  The permutation stays inside each group of 32
// keys, so a row of n keys takes round_up(n, 32) words (32 * words per row).
__device__ __forceinline__ int key_chunk(int t4) {   // t4 a multiple of 4
    const int c = t4 >> 2;
    return (c ^ ((c >> 3) & 7)) << 2;
}
__device__ __forceinline__ int key_index(int t) { return key_chunk(t & ~3) | (t & 3); }
__host__ __device__ inline size_t key_row_words(const Geometry& g) { return 32 * (size_t)g.words; }

constexpr int kPoolSmemBytes = 96 * 1024;     // raw-I chunk of the heads pooling kernel
constexpr int kTopkWarps = 16;                 // warps that run the radix select
constexpr int kTopkThreads = 32 * kTopkWarps;
constexpr int kTopkKPL = 16;                   // positions per lane in a warp segment (half a bits word)
constexpr int kTopkSeg = 32 * kTopkKPL;        // positions per warp segment
constexpr int kTopkBarrier = 1;                // named barrier of the select warps
constexpr int kTopkCap = 2048;                 // keys a compacted candidate list holds (4 per thread)
static_assert(kTopkKPL == 16, "two lanes share a bits word");
static_assert(kTopkCap % kTopkThreads == 0, "the compacted list is split evenly over the select threads");
constexpr int kTopkFew = 32;                   // a threshold bucket this small is ranked directly
constexpr int kTopkSampleK = 4;                // sampled threshold for k <= kTopkCap / kTopkSampleK
constexpr int kTopkSampleN = 32;               // and k <= n / kTopkSampleN (measured: slower for larger k / n)

struct TopkShared {
    int wcnt[2][kTopkWarps][16];   // per-warp digit counts, double-buffered across passes
    uint32_t wor[kTopkWarps], wand[kTopkWarps];
    int weq[kTopkWarps];
    int wsum[32];
    int fcount;
    uint32_t fkey[kTopkFew];
    int fpos[kTopkFew];
    uint32_t ckey[kTopkCap];       // compacted candidates: key and position
    int cpos[kTopkCap];
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

__device__ __forceinline__ void topk_bar() {
    asm volatile("bar.sync %0, %1;" ::"n"(kTopkBarrier), "n"(kTopkThreads) : "memory");
}

// Digit counting without divergent branches: a key adds 1 << (4 d) to a 64-bit
// accumulator of sixteen 4-bit counters (at most 15 keys per accumulator),
// which is then spread into byte counters of the even and odd digits.
__device__ __forceinline__ unsigned long long digit_nibble(uint32_t u, uint32_t mask, uint32_t prefix, int lo,
                                                           uint32_t wmask) {
    const uint32_t m = (u != 0u && (u & mask) == prefix) ? 1u : 0u;
    return (unsigned long long)m << (((u >> lo) & wmask) << 2);
}

struct DigitBytes {
    unsigned long long ev = 0ull, od = 0ull;   // byte j: count of digit 2j / 2j + 1
    __device__ __forceinline__ void add(unsigned long long nib) {
        ev += nib & 0x0F0F0F0F0F0F0F0Full;
        od += (nib >> 4) & 0x0F0F0F0F0F0F0F0Full;
    }
    // pair[j] += count(2j) | count(2j + 1) << 16
    __device__ __forceinline__ void to_pairs(uint32_t* pair) const {
#pragma unroll
        for (int j = 0; j < 8; ++j)
            pair[j] += (uint32_t)((ev >> (8 * j)) & 255ull) | ((uint32_t)((od >> (8 * j)) & 255ull) << 16);
    }
};

// Lane d < 16 receives the warp's count of digit d.
__device__ __forceinline__ int warp_digit_counts(const uint32_t* pair, int lane) {
    int mine = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        const uint32_t t = __reduce_add_sync(0xffffffffu, pair[j]);
        mine = lane == 2 * j ? (int)(t & 0xffffu) : mine;
        mine = lane == 2 * j + 1 ? (int)(t >> 16) : mine;
    }
    return mine;
}

// ORs into bits[] (shared, one bit per position) the k largest keys of a row of
// n keys (stored as key_index lays them out); every thread of the block calls it
// and the bits are complete on return.  Key 0 marks an ineligible position;
// the caller guarantees k <= #eligible.
//
// MSB radix select run by kTopkWarps warps.  Warp w owns a contiguous run of
// 512-position segments; in a segment lane l owns the 16 positions [16 l, 16 l
// + 16) (half of a bits word), which stay in registers when one segment covers
// the warp's share.  A first reduction of OR and AND over the eligible keys fixes the bits
// they all share; each pass then resolves the next (up to) 4 bits that differ:
// threads count digits in registers, warps add the counts with the hardware
// warp reduction, and after one barrier every warp scans the 16 bucket totals
// from the top to find the digit that holds the k-th key.  Once the threshold
// bucket holds at most kTopkCap keys they are compacted (key and position) so
// later passes read only them; once it holds at most kTopkFew keys one warp
// ranks them directly (larger key first, then lower position).  If more equal
// keys than that straddle the threshold they are ranked by position.
template <int NS>
__device__ __forceinline__ void block_topk_impl(const uint32_t* __restrict__ keys, int n, int k, uint32_t* bits,
                                                TopkShared& sm) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, tid = threadIdx.x;
    {
        const int nwords = (n + 31) >> 5;
        const int nseg = (n + kTopkSeg - 1) / kTopkSeg;
        const int spw = (nseg + kTopkWarps - 1) / kTopkWarps;   // segments per warp
        const int seg0 = min(warp * spw, nseg), seg1 = min(seg0 + spw, nseg);
        // This lane's 16 keys of segment sg (0 past the row): four 16-byte loads.
        // With at most NS > 0 segments per warp a lane's keys stay in registers
        // (segment seg0 + si in ureg[16 si ..]); with NS = 0 every sweep reads
        // them again, once per segment.
        auto load16 = [&](int sg, uint32_t* kv) {
            const int t0 = sg * kTopkSeg + lane * kTopkKPL;
            if (t0 + kTopkKPL <= n) {
#pragma unroll
                for (int q = 0; q < kTopkKPL / 4; ++q) {
                    const uint4 v = *reinterpret_cast<const uint4*>(keys + key_chunk(t0 + 4 * q));
                    kv[4 * q] = v.x;
                    kv[4 * q + 1] = v.y;
                    kv[4 * q + 2] = v.z;
                    kv[4 * q + 3] = v.w;
                }
            } else {
#pragma unroll
                for (int j = 0; j < kTopkKPL; ++j) kv[j] = t0 + j < n ? keys[key_index(t0 + j)] : 0u;
            }
        };
        uint32_t ureg[NS > 0 ? NS * kTopkKPL : 1];
        if constexpr (NS > 0) {
#pragma unroll
            for (int si = 0; si < NS; ++si) {
                if (seg0 + si < seg1) {
                    load16(seg0 + si, ureg + si * kTopkKPL);
                } else {
#pragma unroll
                    for (int j = 0; j < kTopkKPL; ++j) ureg[si * kTopkKPL + j] = 0u;
                }
            }
        }
        struct Keys16 {
            uint32_t v[kTopkKPL];
        };
        auto seg_keys = [&](int si, int sg) -> Keys16 {
            Keys16 r;
            if constexpr (NS > 0) {
#pragma unroll
                for (int j = 0; j < kTopkKPL; ++j) r.v[j] = ureg[si * kTopkKPL + j];
            } else {
                load16(sg, r.v);
            }
            return r;
        };
        // Segment loops: si counts the warp's segments (a constant trip count when
        // the keys are in registers, so that ureg is indexed statically).
        const int nsi = NS > 0 ? NS : seg1 - seg0;

        int cnt = 0x7fffffff;   // keys matching the prefix (unknown before the first pass)
        int mlist = -1;         // length of the compacted list, -1 while counting all keys
        if (tid == 0) sm.fcount = 0;   // read only after the next barrier
        // Sampled threshold, when k is small against the row and every warp holds
        // a segment (taken with at most 1/32 of the row selected): T, the lower edge of the 8-bit bin of two sample keys per
        // lane in which the sample's count from the top reaches about twice its
        // share of k; one compare sweep counts the keys >= T and, when there are
        // k to kTopkCap of them, a second one compacts them (in position order)
        // into the list, whose digit passes then finish the selection.  Exact:
        // the list holds every key >= T and at least k keys.  Otherwise (too few
        // or too many) the full sweeps below run as if nothing happened.
        bool listed = false;
        uint32_t gor = 0u, gand = 0xffffffffu;
        if (kTopkSampleK * k <= kTopkCap && kTopkSampleN * k <= n && nseg >= kTopkWarps) {
            int* hist = reinterpret_cast<int*>(sm.ckey);   // 256 bins; the list overwrites it later
            if (tid < 256) hist[tid] = 0;
            uint32_t s0, s1;   // this lane's samples: its first key in its first two segments (or key 8)
            {
                const Keys16 kv = seg_keys(0, seg0);
                s0 = kv.v[0];
                s1 = kv.v[8];
                if constexpr (NS >= 2) {
                    if (seg0 + 1 < seg1) s1 = ureg[kTopkKPL];
                }
            }
            uint32_t sor = s0 | s1, sand = (s0 != 0u ? s0 : 0xffffffffu) & (s1 != 0u ? s1 : 0xffffffffu);
            const int se = (s0 != 0u ? 1 : 0) + (s1 != 0u ? 1 : 0);
            const int wse = __reduce_add_sync(0xffffffffu, se);
            sor = __reduce_or_sync(0xffffffffu, sor);
            sand = __reduce_and_sync(0xffffffffu, sand);
            if (lane == 0) {
                sm.wor[warp] = sor;
                sm.wand[warp] = sand;
                sm.weq[warp] = wse;
            }
            topk_bar();
            uint32_t qor = 0u, qand = 0xffffffffu;
            int S = 0;
#pragma unroll
            for (int x = 0; x < kTopkWarps; ++x) {
                qor |= sm.wor[x];
                qand &= sm.wand[x];
                S += sm.weq[x];
            }
            // Bins: the 8 bits below the sample's highest differing bit (its
            // common bits above fixed); all sample keys equal: T is that key.
            const uint32_t qdiff = qor ^ qand;
            const int qhb = qdiff ? 31 - __clz(qdiff) : 0;
            const int qsh = max(qhb - 7, 0);
            if (qdiff) {
                if (s0 != 0u) atomicAdd(&hist[(s0 >> qsh) & 255u], 1);
                if (s1 != 0u) atomicAdd(&hist[(s1 >> qsh) & 255u], 1);
            }
            topk_bar();
            uint32_t T = qand;
            if (qdiff) {
                // Lane l holds bins 255 - 8 l .. 248 - 8 l (from the top); the bin in
                // which the count from the top reaches ks.
                const int ks = min(S, (2 * k * S + n - 1) / n + 2);
                int c8[8], csum = 0;
#pragma unroll
                for (int b = 0; b < 8; ++b) {
                    c8[b] = hist[255 - 8 * lane - b];
                    csum += c8[b];
                }
                int incl = csum;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int y = __shfl_up_sync(0xffffffffu, incl, o);
                    if (lane >= o) incl += y;
                }
                const unsigned hit = __ballot_sync(0xffffffffu, incl >= ks);
                const int hl = hit ? __ffs(hit) - 1 : 31;
                int run = __shfl_sync(0xffffffffu, incl - csum, hl);
                int bin = 248 - 8 * hl;
#pragma unroll
                for (int b = 0; b < 8; ++b) {
                    const int cb = __shfl_sync(0xffffffffu, c8[b], hl);
                    if (run < ks) {
                        run += cb;
                        bin = 255 - 8 * hl - b;
                    }
                }
                const uint32_t above = qhb >= 31 ? 0u : ~((2u << qhb) - 1u);
                T = (qand & above) | ((uint32_t)bin << qsh);
            }
            // Count the keys >= T (T > 0: eligible keys only).
            if (T != 0u) {
                int c = 0;
#pragma unroll
                for (int si = 0; si < nsi; ++si) {
                    const int sg = seg0 + si;
                    if (sg >= seg1) break;
                    const Keys16 kv = seg_keys(si, sg);
#pragma unroll
                    for (int j = 0; j < kTopkKPL; ++j) c += kv.v[j] >= T ? 1 : 0;
                }
                c = __reduce_add_sync(0xffffffffu, c);
                if (lane == 0) sm.wcnt[0][warp][0] = c;
            }
            topk_bar();
            int total = 0, off = 0;
            if (T != 0u) {
#pragma unroll
                for (int x = 0; x < kTopkWarps; ++x) {
                    const int cx = sm.wcnt[0][x][0];
                    total += cx;
                    off += x < warp ? cx : 0;
                }
            }
            if (T != 0u && total >= k && total <= kTopkCap) {
                // Compact them in position order: warp w after warps 0..w-1, a lane
                // after its segment's lower lanes and the warp's earlier segments.
#pragma unroll
                for (int si = 0; si < nsi; ++si) {
                    const int sg = seg0 + si;
                    if (sg >= seg1) break;
                    const Keys16 kv = seg_keys(si, sg);
                    int mc = 0;
#pragma unroll
                    for (int j = 0; j < kTopkKPL; ++j) mc += kv.v[j] >= T ? 1 : 0;
                    int incl = mc;
#pragma unroll
                    for (int o = 1; o < 32; o <<= 1) {
                        const int y = __shfl_up_sync(0xffffffffu, incl, o);
                        if (lane >= o) incl += y;
                    }
                    int at = off + incl - mc;
                    const int pos0 = sg * kTopkSeg + lane * kTopkKPL;
#pragma unroll
                    for (int j = 0; j < kTopkKPL; ++j) {
                        if (kv.v[j] >= T && at < kTopkCap) {
                            sm.ckey[at] = kv.v[j];
                            sm.cpos[at] = pos0 + j;
                            ++at;
                        }
                    }
                    off += __shfl_sync(0xffffffffu, incl, 31);
                }
                topk_bar();
                // The list's own shared bits start the digit passes.
                uint32_t kor = 0u, kand = 0xffffffffu;
#pragma unroll
                for (int r = 0; r < kTopkCap / kTopkThreads; ++r) {
                    const int j = tid + r * kTopkThreads;
                    if (j < total) {
                        kor |= sm.ckey[j];
                        kand &= sm.ckey[j];
                    }
                }
                kor = __reduce_or_sync(0xffffffffu, kor);
                kand = __reduce_and_sync(0xffffffffu, kand);
                if (lane == 0) {
                    sm.wor[warp] = kor;
                    sm.wand[warp] = kand;
                }
                topk_bar();
                mlist = total;
                cnt = total;
                listed = true;
            }
        }
        if (!listed) {
            // Bits shared by every eligible key.
            uint32_t kor = 0u, kand = 0xffffffffu;
#pragma unroll
            for (int si = 0; si < nsi; ++si) {
                const int sg = seg0 + si;
                if (sg >= seg1) break;
                const Keys16 kv = seg_keys(si, sg);
#pragma unroll
                for (int j = 0; j < kTopkKPL; ++j) {
                    const uint32_t v = kv.v[j];
                    kor |= v;
                    kand &= v != 0u ? v : 0xffffffffu;
                }
            }
            kor = __reduce_or_sync(0xffffffffu, kor);
            kand = __reduce_and_sync(0xffffffffu, kand);
            if (lane == 0) {
                sm.wor[warp] = kor;
                sm.wand[warp] = kand;
            }
            topk_bar();
        }
#pragma unroll
        for (int x = 0; x < kTopkWarps; ++x) {
            gor |= sm.wor[x];
            gand &= sm.wand[x];
        }
        const uint32_t gdiff = gor ^ gand;   // bits on which eligible keys differ

        uint32_t prefix = 0u, mask = 0u;
        int kk = k;
        bool whole_bin = false;
        int lo = 32;            // lowest bit resolved so far
        for (int pass = 0;; ++pass) {
            // Fix the bits below lo that every eligible key shares, then take up
            // to 4 bits down from the highest differing one.
            const uint32_t below = lo == 32 ? 0xffffffffu : ((1u << lo) - 1u);
            const uint32_t diff = gdiff & below;
            if (diff == 0u) {
                prefix |= gand & below;
                mask |= below;
                break;
            }
            const int hb = 31 - __clz(diff);
            const uint32_t fixed = below & ~((2u << hb) - 1u);   // bits (hb, lo), none when hb = 31
            prefix |= gand & fixed;
            mask |= fixed;
            lo = max(hb - 3, 0);
            const uint32_t wmask = (1u << (hb - lo + 1)) - 1u;

            int mine;   // lane d < 16: this warp's count of digit d
            if (mlist < 0) {
                uint32_t pair[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
#pragma unroll
                for (int si = 0; si < nsi; ++si) {
                    const int sg = seg0 + si;
                    if (sg >= seg1) break;
                    const Keys16 kv = seg_keys(si, sg);
                    DigitBytes db;
#pragma unroll
                    for (int j0 = 0; j0 < kTopkKPL; j0 += 15) {
                        unsigned long long nib = 0ull;
#pragma unroll
                        for (int j = j0; j < j0 + 15 && j < kTopkKPL; ++j)
                            nib += digit_nibble(kv.v[j], mask, prefix, lo, wmask);
                        db.add(nib);
                    }
                    db.to_pairs(pair);
                }
                mine = warp_digit_counts(pair, lane);
            } else {
                // At most 4 list entries per thread: a warp's count of a digit fits a byte.
                unsigned long long nib = 0ull;
#pragma unroll
                for (int r = 0; r < kTopkCap / kTopkThreads; ++r) {
                    const int j = tid + r * kTopkThreads;
                    nib += digit_nibble(j < mlist ? sm.ckey[j] : 0u, mask, prefix, lo, wmask);
                }
                DigitBytes db;
                db.add(nib);
                mine = 0;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    // quad q: bytes (digit 4q, 4q + 2) from ev, (4q + 1, 4q + 3) from od
                    const uint32_t e = (uint32_t)(db.ev >> (16 * q)) & 0xffffu, o = (uint32_t)(db.od >> (16 * q)) & 0xffffu;
                    const uint32_t quad = (e & 0xffu) | ((o & 0xffu) << 8) | ((e >> 8) << 16) | ((o >> 8) << 24);
                    const uint32_t t = __reduce_add_sync(0xffffffffu, quad);
#pragma unroll
                    for (int b = 0; b < 4; ++b) mine = lane == 4 * q + b ? (int)((t >> (8 * b)) & 0xffu) : mine;
                }
            }
            const int buf = pass & 1;
            if (lane < 16) sm.wcnt[buf][warp][lane] = mine;
            topk_bar();
            // Every warp finds the threshold digit itself (no second barrier; the
            // counts are double-buffered so the next pass cannot overwrite them early).
            int tot = 0;
            if (lane < 16) {
#pragma unroll
                for (int x = 0; x < kTopkWarps; ++x) tot += sm.wcnt[buf][x][lane];
            }
            int suf = tot;   // count of digits >= lane
#pragma unroll
            for (int off = 1; off < 16; off <<= 1) {
                const int y = __shfl_down_sync(0xffffffffu, suf, off);
                if (lane + off < 16) suf += y;
            }
            const int above_l = suf - tot;
            const unsigned hit = __ballot_sync(0xffffffffu, lane < 16 && above_l < kk && kk <= suf);
            const int D = hit ? __ffs(hit) - 1 : 0;
            const int above = __shfl_sync(0xffffffffu, above_l, D);
            cnt = __shfl_sync(0xffffffffu, tot, D);
            prefix |= (uint32_t)D << lo;
            mask |= wmask << lo;
            kk -= above;
            if (cnt == kk) {
                whole_bin = true;
                break;
            }
            if (lo == 0 || cnt <= kTopkFew) break;
            if (mlist < 0 && cnt <= kTopkCap) {
                // Compact the keys of the threshold bucket.  Warp w's share starts
                // after the bucket counts of warps 0..w-1, a lane's after the
                // matches of its segment's lower lanes and earlier segments.
                int off = 0;
                for (int x = 0; x < warp; ++x) off += sm.wcnt[buf][x][D];
#pragma unroll
                for (int si = 0; si < nsi; ++si) {
                    const int sg = seg0 + si;
                    if (sg >= seg1) break;
                    const Keys16 kv = seg_keys(si, sg);
                    int mc = 0;
#pragma unroll
                    for (int j = 0; j < kTopkKPL; ++j) {
                        const uint32_t v = kv.v[j];
                        mc += (v != 0u && (v & mask) == prefix) ? 1 : 0;
                    }
                    int incl = mc;
#pragma unroll
                    for (int o = 1; o < 32; o <<= 1) {
                        const int y = __shfl_up_sync(0xffffffffu, incl, o);
                        if (lane >= o) incl += y;
                    }
                    int at = off + incl - mc;
                    const int pos0 = sg * kTopkSeg + lane * kTopkKPL;
                    uint32_t half = 0u;   // this lane's positions above the bucket: selected for certain
#pragma unroll
                    for (int j = 0; j < kTopkKPL; ++j) {
                        const uint32_t v = kv.v[j];
                        const bool m = v != 0u && (v & mask) == prefix;
                        if (m && at < kTopkCap) {
                            sm.ckey[at] = v;
                            sm.cpos[at] = pos0 + j;
                        }
                        at += m ? 1 : 0;
                        half |= (v != 0u && (v & mask) > prefix ? 1u : 0u) << j;
                    }
                    off += __shfl_sync(0xffffffffu, incl, 31);
                    // Lanes 2m and 2m + 1 hold the low and high halves of the segment's word m.
                    const uint32_t high = __shfl_xor_sync(0xffffffffu, half, 1);
                    const int wd = sg * (kTopkSeg / 32) + (lane >> 1);
                    const uint32_t word = half | (high << 16);
                    if ((lane & 1) == 0 && wd < nwords && word) bits[wd] |= word;
                }
                mlist = cnt;
                topk_bar();
            }
        }

        const bool few = !whole_bin && cnt <= kTopkFew;
        if (few) {
            // Gather the bucket's keys with their positions.
            if (mlist >= 0) {
#pragma unroll
                for (int r = 0; r < kTopkCap / kTopkThreads; ++r) {
                    const int j = tid + r * kTopkThreads;
                    if (j < mlist && (sm.ckey[j] & mask) == prefix) {
                        const int slot = atomicAdd(&sm.fcount, 1);
                        if (slot < kTopkFew) {
                            sm.fkey[slot] = sm.ckey[j];
                            sm.fpos[slot] = sm.cpos[j];
                        }
                    }
                }
            } else {
#pragma unroll
                for (int si = 0; si < nsi; ++si) {
                    const int sg = seg0 + si;
                    if (sg >= seg1) break;
                    const Keys16 kv = seg_keys(si, sg);
                    const int pos0 = sg * kTopkSeg + lane * kTopkKPL;
#pragma unroll
                    for (int j = 0; j < kTopkKPL; ++j) {
                        const uint32_t v = kv.v[j];
                        if (v != 0u && (v & mask) == prefix) {
                            const int slot = atomicAdd(&sm.fcount, 1);
                            if (slot < kTopkFew) {
                                sm.fkey[slot] = v;
                                sm.fpos[slot] = pos0 + j;
                            }
                        }
                    }
                }
            }
        }
        const bool ties = !whole_bin && !few;
        if (mlist >= 0) {
            // The compaction sweep marked every key above its bucket; the list
            // holds that bucket in position order, a thread the four entries
            // [4 tid, 4 tid + 4).  Mark the entries above the final threshold, the
            // whole final bucket when it is taken whole, and with ties its equal
            // entries at the kk lowest positions (the few path ranks its bucket below).
            constexpr int kPer = kTopkCap / kTopkThreads;
            uint32_t v4[kPer];
            int eq = 0;
#pragma unroll
            for (int r = 0; r < kPer; ++r) {
                const int j = kPer * tid + r;
                v4[r] = j < mlist ? sm.ckey[j] : 0u;
                eq += (v4[r] != 0u && (v4[r] & mask) == prefix) ? 1 : 0;
            }
            int before = 0;   // equal entries in lower positions (ties only)
            if (ties) {
                int incl = eq;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int y = __shfl_up_sync(0xffffffffu, incl, o);
                    if (lane >= o) incl += y;
                }
                if (lane == 31) sm.weq[warp] = incl;
                topk_bar();
                for (int x = 0; x < warp; ++x) before += sm.weq[x];
                before += incl - eq;
            }
#pragma unroll
            for (int r = 0; r < kPer; ++r) {
                const int j = kPer * tid + r;
                const uint32_t um = v4[r] & mask;
                const bool isq = v4[r] != 0u && um == prefix;
                const bool sel = (v4[r] != 0u && um > prefix) || (whole_bin && isq) || (ties && isq && before < kk);
                before += isq ? 1 : 0;
                if (sel) {
                    const int pos = sm.cpos[j];
                    atomicOr(&bits[pos >> 5], 1u << (pos & 31));
                }
            }
        } else {
        if (ties) {
            // More equal keys straddle the threshold than kTopkFew: rank by position.
            int eqc = 0;
#pragma unroll
            for (int si = 0; si < nsi; ++si) {
                const int sg = seg0 + si;
                if (sg >= seg1) break;
                const Keys16 kv = seg_keys(si, sg);
#pragma unroll
                for (int j = 0; j < kTopkKPL; ++j) {
                    const uint32_t v = kv.v[j];
                    eqc += (v != 0u && (v & mask) == prefix) ? 1 : 0;
                }
            }
            eqc = __reduce_add_sync(0xffffffffu, eqc);
            if (lane == 0) sm.weq[warp] = eqc;
        }
        topk_bar();
        int base = 0;   // equal keys at lower positions (ties only)
        if (ties)
            for (int x = 0; x < warp; ++x) base += sm.weq[x];
        // Mark the keys above the threshold prefix (all of the bucket when it is
        // taken whole; with ties, the equal keys at the kk lowest positions).
#pragma unroll
        for (int si = 0; si < nsi; ++si) {
            const int sg = seg0 + si;
            if (sg >= seg1) break;
            const Keys16 kv = seg_keys(si, sg);
            uint32_t half = 0u;   // this lane's 16 positions
            if (!ties) {
#pragma unroll
                for (int j = 0; j < kTopkKPL; ++j) {
                    const uint32_t v = kv.v[j];
                    const uint32_t um = v & mask;
                    const bool sel = v != 0u && (um > prefix || (whole_bin && um == prefix));
                    half |= (sel ? 1u : 0u) << j;
                }
            } else {
                int ec = 0;
#pragma unroll
                for (int j = 0; j < kTopkKPL; ++j) {
                    const uint32_t v = kv.v[j];
                    ec += (v != 0u && (v & mask) == prefix) ? 1 : 0;
                }
                int incl = ec;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int y = __shfl_up_sync(0xffffffffu, incl, o);
                    if (lane >= o) incl += y;
                }
                int rank = base + incl - ec;
#pragma unroll
                for (int j = 0; j < kTopkKPL; ++j) {
                    const uint32_t v = kv.v[j];
                    const uint32_t um = v & mask;
                    const bool eq = v != 0u && um == prefix;
                    const bool sel = (v != 0u && um > prefix) || (eq && rank < kk);
                    rank += eq ? 1 : 0;
                    half |= (sel ? 1u : 0u) << j;
                }
                base += __shfl_sync(0xffffffffu, incl, 31);
            }
            // Lanes 2m and 2m + 1 hold the low and high halves of the segment's word m.
            const uint32_t high = __shfl_xor_sync(0xffffffffu, half, 1);
            const int wd = sg * (kTopkSeg / 32) + (lane >> 1);
            const uint32_t word = half | (high << 16);
            if ((lane & 1) == 0 && wd < nwords && word) bits[wd] |= word;
        }
        }
        if (few) {
            topk_bar();   // the sweep's plain stores are done before warp 0 adds bits
            if (warp == 0) {
                const int m = min(sm.fcount, kTopkFew);
                const uint32_t key = lane < m ? sm.fkey[lane] : 0u;
                const int pos = lane < m ? sm.fpos[lane] : 0x7fffffff;
                int rank = 0;
                for (int j = 0; j < m; ++j) {
                    const uint32_t kj = __shfl_sync(0xffffffffu, key, j);
                    const int pj = __shfl_sync(0xffffffffu, pos, j);
                    rank += (kj > key || (kj == key && pj < pos)) ? 1 : 0;
                }
                if (lane < m && rank < kk && pos < n) atomicOr(&bits[pos >> 5], 1u << (pos & 31));
            }
        }
    }
}

// NSMAX: the most 512-position segments per warp kept in registers (2 where the
// caller has the registers to spare).
template <int NSMAX = 1>
__device__ void block_topk(const uint32_t* __restrict__ keys, int n, int k, uint32_t* bits, TopkShared& sm) {
    if (k > 0 && n > 0 && (threadIdx.x >> 5) < kTopkWarps) {
        const int nseg = (n + kTopkSeg - 1) / kTopkSeg;
        if (nseg <= kTopkWarps)
            block_topk_impl<1>(keys, n, k, bits, sm);
        else if (NSMAX >= 2 && nseg <= 2 * kTopkWarps)
            block_topk_impl<NSMAX >= 2 ? 2 : 1>(keys, n, k, bits, sm);
        else
            block_topk_impl<0>(keys, n, k, bits, sm);
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

// Max-pool (width 2*halo+1, stride 1, neighbours outside [0, Lc) ignored) of
// the four positions [t4, t4+4) of a row given as the sum of `parts` partial
// rows `stride` floats apart: the raw values [t4-8, t4+12) of every part
// arrive as five float4 loads issued together.
struct Pooled4 {
    float v[4];
};

__device__ __forceinline__ Pooled4 pool4(const float* __restrict__ raw, size_t stride, int parts, int t4, int Lc,
                                         int halo, bool avg) {
    float x[20];
#pragma unroll
    for (int i = 0; i < 20; ++i) x[i] = 0.f;
    for (int pt = 0; pt < parts; ++pt) {
        const float* r = raw + pt * stride;
        float4 f[5];
#pragma unroll
        for (int b = 0; b < 5; ++b) {
            const int p = t4 - 8 + 4 * b;
            f[b] = (p >= 0 && p < Lc) ? __ldcg(reinterpret_cast<const float4*>(r + p)) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int b = 0; b < 5; ++b) {
            x[4 * b] += f[b].x;
            x[4 * b + 1] += f[b].y;
            x[4 * b + 2] += f[b].z;
            x[4 * b + 3] += f[b].w;
        }
    }
    Pooled4 out;
    if (avg) {
        // Average variant: the mean of the in-range neighbours.
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float sum = x[8 + i], cnt = 1.f;
#pragma unroll
            for (int d = 1; d <= kMaxPool / 2; ++d) {
                if (d <= halo && t4 + i - d >= 0) {
                    sum += x[8 + i - d];
                    cnt += 1.f;
                }
                if (d <= halo && t4 + i + d < Lc) {
                    sum += x[8 + i + d];
                    cnt += 1.f;
                }
            }
            out.v[i] = sum / cnt;
        }
        return out;
    }
#pragma unroll
    for (int i = 0; i < 20; ++i)
        if (t4 - 8 + i < 0 || t4 - 8 + i >= Lc) x[i] = -INFINITY;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        float m = x[8 + i];
#pragma unroll
        for (int d = 1; d <= kMaxPool / 2; ++d)
            if (d <= halo) m = fmaxf(m, fmaxf(x[8 + i - d], x[8 + i + d]));
        out.v[i] = m;
    }
    return out;
}

// Running (count, mean, sum of squared deviations); merge() is Chan et al.'s
// pairwise update, stable in fp32 (no cancellation of sum(x^2) - n*mean^2).
struct Moments {
    float n, mean, m2;
    __device__ void add(float x) {
        n += 1.f;
        const float d = x - mean;
        mean += d / n;
        m2 += d * (x - mean);
    }
    __device__ void merge(float nb, float meanb, float m2b) {
        if (nb == 0.f) return;
        if (n == 0.f) {
            n = nb;
            mean = meanb;
            m2 = m2b;
            return;
        }
        const float nt = n + nb, d = meanb - mean;
        mean += d * (nb / nt);
        m2 += m2b + d * d * (n * nb / nt);
        n = nt;
    }
};

// Sums of a and b over the block (the result is valid in thread 0).
__device__ float2 block_sum2(float a, float b, float3* red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    for (int off = 16; off; off >>= 1) {
        a += __shfl_xor_sync(0xffffffffu, a, off);
        b += __shfl_xor_sync(0xffffffffu, b, off);
    }
    if (lane == 0) red[warp] = make_float3(a, b, 0.f);
    __syncthreads();
    float2 r = make_float2(0.f, 0.f);
    if (warp == 0) {
        const float3 v = lane < nw ? red[lane] : make_float3(0.f, 0.f, 0.f);
        a = v.x;
        b = v.y;
        for (int off = 16; off; off >>= 1) {
            a += __shfl_xor_sync(0xffffffffu, a, off);
            b += __shfl_xor_sync(0xffffffffu, b, off);
        }
        r = make_float2(a, b);
    }
    __syncthreads();
    return r;
}

__device__ Moments block_moments(Moments v, float3* red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    for (int off = 16; off; off >>= 1)
        v.merge(__shfl_xor_sync(0xffffffffu, v.n, off), __shfl_xor_sync(0xffffffffu, v.mean, off),
                __shfl_xor_sync(0xffffffffu, v.m2, off));
    if (lane == 0) red[warp] = make_float3(v.n, v.mean, v.m2);
    __syncthreads();
    Moments t{0.f, 0.f, 0.f};
    if (lane < nw) t = Moments{red[lane].x, red[lane].y, red[lane].z};
    for (int off = 16; off; off >>= 1)
        t.merge(__shfl_xor_sync(0xffffffffu, t.n, off), __shfl_xor_sync(0xffffffffu, t.mean, off),
                __shfl_xor_sync(0xffffffffu, t.m2, off));
    __syncthreads();
    return t;
}

// Section 4.1, first half.  One CTA per (KV head, sequence): pool the head's
// P_O and P_O' rows and a slice of I (max-pool, inherited from SnapKV; or the
// average variant) and the head's ranking key: sigma_h = sample std of pooled
// P_O over the candidates (Welford/Chan moments in fp32), or, for the entropy
// criterion of the Section 5.4 ablation, minus the entropy of pooled P_O
// normalised over the candidates, sum(x ln x)/S - ln S with S = sum(x).
__global__ void __launch_bounds__(kSelectThreads) heads_pool_kernel(Geometry G, LayerIO io, Scratch sc, Slot sl) {
    __shared__ float3 red[32];
    extern __shared__ float mbuf[];   // raw I of a chunk, per window row (several head groups only)
    const int h = blockIdx.x, s = blockIdx.y;
    const int tid = threadIdx.x, NT = blockDim.x;
    const int L = io.cu[s + 1] - io.cu[s];
    const int Lc = L - G.wk;
    const int halo = G.pool / 2;
    const size_t row = (size_t)s * G.Hkv + h;
    // Pool P_O and P_O' of this head (four positions per thread per step) and
    // accumulate the moments of pooled P_O.
    Moments mom{0.f, 0.f, 0.f};
    float es = 0.f, exl = 0.f;   // entropy criterion: sum x, sum x ln x
    const bool avg = G.pool_avg != 0, entropy = G.head_entropy != 0;
    const float* rO = sl.rawO + row * G.ML;
    const float* rOe = sl.rawOe + row * G.ML;
    for (int t4 = 4 * tid; t4 < Lc; t4 += 4 * NT) {
        const Pooled4 a = pool4(rO, 0, 1, t4, Lc, halo, avg);
        const Pooled4 b = pool4(rOe, 0, 1, t4, Lc, halo, avg);
        *reinterpret_cast<float4*>(sl.PO + row * G.ML + t4) = make_float4(a.v[0], a.v[1], a.v[2], a.v[3]);
        *reinterpret_cast<float4*>(sl.POe + row * G.ML + t4) = make_float4(b.v[0], b.v[1], b.v[2], b.v[3]);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            if (t4 + i >= Lc) continue;
            if (entropy) {
                es += a.v[i];
                if (a.v[i] > 0.f) exl = fmaf(a.v[i], logf(a.v[i]), exl);
            } else {
                mom.add(a.v[i]);
            }
        }
    }
    // This CTA's slice of pooled I.
    {
        const int per = ((Lc + G.Hkv - 1) / G.Hkv + 3) & ~3;
        const int a0 = min(h * per, Lc), b0 = min(a0 + per, Lc);
        if (G.NG == 1) {
            const float* rI = sl.rawI + (size_t)s * G.ML;
            for (int t4 = a0 + 4 * tid; t4 < b0; t4 += 4 * NT) {
                const Pooled4 c = pool4(rI, 0, 1, t4, Lc, halo, avg);
                *reinterpret_cast<float4*>(sl.I + (size_t)s * G.ML + t4) = make_float4(c.v[0], c.v[1], c.v[2], c.v[3]);
            }
        } else {
            // The window kernel left, per group of KV heads, the maxima over the
            // group of G_h[q][t] (q >= w - O): raw I is (1/O) times the sum over q of
            // the maxima over the groups.  Built in shared memory chunk by chunk (with
            // the pool halo), each (q, t) element loaded by its own thread, then pooled.
            int tbase = 0;
            for (int b = 0; b < s; ++b) {
                const int lb = io.cu[b + 1] - io.cu[b] - G.wk;
                tbase += lb > 0 ? (lb + kTileT - 1) / kTileT : 0;
            }
            const float invO = 1.f / (float)G.O;
            const size_t n_el = (size_t)G.O * kTileT;
            const int chunk = ((kPoolSmemBytes / 4) / G.O - 2 * halo) & ~3;
            for (int c = a0; c < b0; c += chunk) {
                const int ce = min(c + chunk, b0);
                const int lo = max(c - halo, 0), hi = min(ce + halo, Lc), span = hi - lo;
                const int n = G.O * span;   // mbuf[q][span]: element index q * span + (t - lo)
                for (int base = tid; base < n; base += 8 * NT) {
                    float m[8];
#pragma unroll
                    for (int u = 0; u < 8; ++u) {
                        const int idx = base + u * NT;
                        const int q = idx / span, t = lo + idx - q * span;
                        m[u] = idx < n ? __ldcg(sl.wpart + (size_t)(tbase + (t >> 7)) * G.NG * n_el + q * kTileT + (t & 127))
                                       : 0.f;
                    }
                    for (int gg = 1; gg < G.NG; ++gg) {
#pragma unroll
                        for (int u = 0; u < 8; ++u) {
                            const int idx = base + u * NT;
                            const int q = idx / span, t = lo + idx - q * span;
                            if (idx < n)
                                m[u] = fmaxf(m[u], __ldcg(sl.wpart + ((size_t)(tbase + (t >> 7)) * G.NG + gg) * n_el +
                                                           q * kTileT + (t & 127)));
                        }
                    }
#pragma unroll
                    for (int u = 0; u < 8; ++u)
                        if (base + u * NT < n) mbuf[base + u * NT] = m[u];
                }
                __syncthreads();
                // Sum over q in place: column tt of row 0 becomes raw I (each thread owns its columns).
                for (int tt = tid; tt < span; tt += NT) {
                    float sum = 0.f;
                    for (int q = 0; q < G.O; ++q) sum += mbuf[q * span + tt];
                    mbuf[tt] = sum * invO;
                }
                __syncthreads();
                for (int t = c + tid; t < ce; t += NT) {
                    float m = mbuf[t - lo], cnt = 1.f;
                    for (int d = 1; d <= halo; ++d) {
                        if (t - d >= 0) {
                            m = avg ? m + mbuf[t - d - lo] : fmaxf(m, mbuf[t - d - lo]);
                            cnt += 1.f;
                        }
                        if (t + d < Lc) {
                            m = avg ? m + mbuf[t + d - lo] : fmaxf(m, mbuf[t + d - lo]);
                            cnt += 1.f;
                        }
                    }
                    sl.I[(size_t)s * G.ML + t] = avg ? m / cnt : m;
                }
                __syncthreads();
            }
        }
    }
    // The preserved-token kernel may be scheduled now; it waits for this grid before reading sigma.
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
    if (entropy) {
        const float2 se = block_sum2(es, exl, red);
        if (tid == 0) sl.sigma[row] = se.x > 0.f ? se.y / se.x - logf(se.x) : 0.f;
    } else {
        mom = block_moments(mom, red);
        if (tid == 0) sl.sigma[row] = Lc >= 2 ? sqrtf(fmaxf(mom.m2, 0.f) / (float)(Lc - 1)) : 0.f;
    }
}

// Section 4.1, second half, and the preserved tokens of Section 4.2.  One CTA
// per (KV head, sequence), launched after heads_pool_kernel: every CTA ranks the
// sequence's sigmas the same way, the delta lowest-sigma heads take the O'
// scores, then the top-K preserved tokens of the chosen row by radix select.
__global__ void __launch_bounds__(kSelectThreads, 2) heads_topk_kernel(Geometry G, LayerIO io, Scratch sc, Slot sl) {
    __shared__ TopkShared sm;
    __shared__ int top_flag;
    extern __shared__ __align__(16) uint32_t bits[];
    const int h = blockIdx.x, s = blockIdx.y;
    const int tid = threadIdx.x, NT = blockDim.x;
    const int L = io.cu[s + 1] - io.cu[s];
    const int Lc = L - G.wk;
    const size_t row = (size_t)s * G.Hkv + h;
    for (int wd = tid; wd < G.words; wd += NT) bits[wd] = 0u;
    // Programmatic dependent of the pooling kernel: its sigmas and pooled rows are
    // read only after that grid has completed.
    asm volatile("griddepcontrol.wait;\n" ::: "memory");
    if (tid < 32) {
        const float sigma = __ldcg(&sl.sigma[row]);
        const float so = tid < G.Hkv ? __ldcg(&sl.sigma[(size_t)s * G.Hkv + tid]) : INFINITY;
        const bool before = tid < G.Hkv && (so < sigma || (so == sigma && tid < h));
        const int rank = __popc(__ballot_sync(0xffffffffu, before));
        if (tid == 0) {
            top_flag = rank < G.delta;
            sl.htop[row] = rank < G.delta;
        }
    }
    __syncthreads();
    const int top = top_flag;
    if (L > G.budget && G.Kp > 0) {
        const float* __restrict__ P = (top ? sl.POe : sl.PO) + row * G.ML;
        uint32_t* keys = keys_in_smem(G.ML) ? bits + ((G.words + 3) & ~3) : sc.keys + row * G.ML;
        for (int b0 = 4 * tid; b0 < Lc; b0 += 16 * NT) {
            float4 pv[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int t4 = b0 + 4 * u * NT;
                pv[u] = t4 < Lc ? __ldcg(reinterpret_cast<const float4*>(P + t4)) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int t4 = b0 + 4 * u * NT;
                if (t4 < Lc) {   // positions from Lc on get key 0 (never read)
                    const float x[4] = {pv[u].x, pv[u].y, pv[u].z, pv[u].w};
                    uint32_t kq[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) kq[i] = t4 + i < Lc ? float_order_key(x[i]) : 0u;
                    *reinterpret_cast<uint4*>(keys + key_chunk(t4)) = make_uint4(kq[0], kq[1], kq[2], kq[3]);
                }
            }
        }
        __syncthreads();
        block_topk(keys, Lc, G.Kp, bits, sm);
    }
    uint32_t* pres = sl.pres + row * G.words;
    for (int wd = tid; wd < G.words; wd += NT) pres[wd] = bits[wd];
}

// Section 4.2: P' = P + lambda * I * (1 - n_t / (l + 1)); the preserved tokens
// stay, the rest of B - w goes to the largest P'; the last w tokens are kept.
// Writes the head's kept positions as bits (sl.sel); gather_kernel turns them
// into out_idx.  Grid (Hkv, batch).
//
// Coverage counts: n_t before this layer = A[t] + U_prev[t], where A is the
// count array of the previous layer (the state for lcall = 0) and U_prev the
// previous layer's union, the OR of its heads' kept bits (prev_sel; none for
// lcall = 0).  Every CTA reads them for its keys and writes the sum for its
// slice of positions to the other count array, which is the next layer's A;
// finalize_kernel folds the last union into the state.  No CTA waits for
// another, and the previous layer's selection (a programmatic dependency) is
// the only one this kernel waits for: everything after that wait is the serial
// part of a multi-layer call.
__global__ void __launch_bounds__(kSelectThreads) select_kernel(Geometry G, LayerIO io, Scratch sc, Slot sl,
                                                                 const uint32_t* prev_sel, int lcall, int ncall) {
    __shared__ TopkShared sm;
    extern __shared__ __align__(16) uint32_t bits[];
    const int h = blockIdx.x, s = blockIdx.y;
    const int tid = threadIdx.x, NT = blockDim.x;
    const int L = io.cu[s + 1] - io.cu[s];
    const int Lc = L - G.wk;
    const int wordsL = (L + 31) >> 5;
    const bool cached = scores_in_smem(G.ML) && L > G.budget;
    // Shared memory: bits[words] | preserved bits[words] | union[words] |
    // adaptive-fill candidate bits[words] | keys | P row | I row (P and I
    // 16-byte aligned for float4 stores).
    uint32_t* spres = bits + G.words;
    uint32_t* suni = spres + G.words;
    const size_t sp_off = ((size_t)4 * G.words + (keys_in_smem(G.ML) ? key_row_words(G) : 0) + 3) & ~(size_t)3;
    float* sP = reinterpret_cast<float*>(bits + sp_off);
    float* sI = sP + G.ML;
    const size_t row = (size_t)s * G.Hkv + h;
    const int top = sl.htop[row];
    const float* P = (top ? sl.POe : sl.PO) + row * G.ML;
    const float* I = sl.I + (size_t)s * G.ML;
    const uint32_t* pres = sl.pres + row * G.words;
    uint8_t* st = io.state + (size_t)s * G.state_stride;
    // This layer's scores and preserved tokens do not depend on the previous
    // layer: stage them now, overlapping the previous layer's selection.
    for (int wd = tid; wd < G.words; wd += NT) {
        bits[wd] = 0u;
        spres[wd] = __ldcg(&pres[wd]);
        suni[G.words + wd] = 0u;   // adaptive-fill candidate bits
    }
    if (cached) {
        for (int t4 = 4 * tid; t4 < Lc; t4 += 4 * NT) {
            *reinterpret_cast<float4*>(sP + t4) = __ldcg(reinterpret_cast<const float4*>(P + t4));
            *reinterpret_cast<float4*>(sI + t4) = __ldcg(reinterpret_cast<const float4*>(I + t4));
        }
    }
    // The state header changes only at the end of a call (finalize_kernel).
    // From the second layer of a call on, the previous call's finalize has
    // completed before this grid could start, so the header is read early.
    uint32_t ell0 = lcall > 0 ? __ldcg(reinterpret_cast<const uint32_t*>(st)) : 0u;
    uint8_t* nstate = st + G.state_n_off;
    uint8_t* nscr = sc.nbuf + (size_t)s * G.nlen;
    const uint8_t* nA = (lcall & 1) ? nscr : nstate;          // counts before the previous layer's union
    uint8_t* nB = (lcall & 1) ? nstate : nscr;                // counts before this layer's union
    // This CTA's slice of positions (a multiple of 32 long) for the next count array.
    const int fper = (((L + G.Hkv - 1) / G.Hkv) + 31) & ~31;
    const int f0 = min(h * fper, L), f1 = min(f0 + fper, L);
    const bool select = L > G.budget;
    __syncthreads();
    // Launched as a programmatic dependent of the previous layer's selection:
    // everything above overlaps its tail; the coverage counts are read only after
    // that grid has completed and its writes are visible.
    asm volatile("griddepcontrol.wait;\n" ::: "memory");
    if (lcall == 0) ell0 = __ldcg(reinterpret_cast<const uint32_t*>(st));
    if (ell0 + (uint32_t)ncall > 255u) {  // n_t is 8-bit: no state may count more than 255 layers
        if (tid == 0) atomicExch(sc.err, 2);  // every layer of the call refuses; the state stays as it was
        return;
    }
    const uint32_t ell = ell0 + (uint32_t)lcall;
    // One round of loads: this thread's first group of counts and the previous
    // layer's union words (the OR over its heads' kept bits).
    const int g0 = 4 * tid;
    uchar4 nv0[4];
    if (select) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int t4 = g0 + 4 * u * NT;
            if (t4 < Lc) nv0[u] = *reinterpret_cast<const uchar4*>(nA + t4);
        }
    }
    const uint32_t* prow = prev_sel ? prev_sel + (size_t)s * G.Hkv * G.words : nullptr;
    for (int wd = tid; wd < wordsL; wd += NT) {
        uint32_t u = 0u;
        if (prow) {
#pragma unroll 8
            for (int hh = 0; hh < G.Hkv; ++hh) u |= __ldcg(&prow[(size_t)hh * G.words + wd]);
        }
        suni[wd] = u;
    }
    __syncthreads();
    auto counts4 = [&](int t4, uchar4 a) {
        const uint32_t b = suni[t4 >> 5] >> (t4 & 31);
        return make_uchar4((uint8_t)(a.x + (b & 1u)), (uint8_t)(a.y + ((b >> 1) & 1u)), (uint8_t)(a.z + ((b >> 2) & 1u)),
                           (uint8_t)(a.w + ((b >> 3) & 1u)));
    };
    if (select) {
        // P' of the last layer of a call is kept for inspection (kvec_debug_scores).
        float* Pp = lcall + 1 == ncall ? sl.Pprime + row * G.ML : nullptr;
        uint32_t* keys = keys_in_smem(G.ML) ? suni + 2 * G.words : sc.keys_sel + row * G.ML;
        const float* Pr = cached ? sP : P;
        const float* Ir = cached ? sI : I;
        // coverage = n_t / (l + 1) as n_t times the rounded reciprocal: a divide
        // per position costs more than the rest of the key.
        const float inv_l1 = __frcp_rn((float)(ell + 1u));
        for (int b0 = g0; b0 < Lc; b0 += 16 * NT) {
            float4 pv[4], iv[4];
            uchar4 nv[4];
            uint32_t pw[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int t4 = b0 + 4 * u * NT;
                if (t4 < Lc) {
                    nv[u] = b0 == g0 ? nv0[u] : *reinterpret_cast<const uchar4*>(nA + t4);
                    pv[u] = *reinterpret_cast<const float4*>(Pr + t4);
                    iv[u] = *reinterpret_cast<const float4*>(Ir + t4);
                    pw[u] = spres[t4 >> 5];
                }
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int t4 = b0 + 4 * u * NT;
                if (t4 >= Lc) continue;
                const uchar4 c = counts4(t4, nv[u]);
                if (t4 >= f0 && t4 + 4 <= f1 && t4 + 4 <= Lc) *reinterpret_cast<uchar4*>(nB + t4) = c;
                const float p4[4] = {pv[u].x, pv[u].y, pv[u].z, pv[u].w};
                const float i4[4] = {iv[u].x, iv[u].y, iv[u].z, iv[u].w};
                const uint8_t n4[4] = {c.x, c.y, c.z, c.w};
                float out[4];
                uint32_t kq[4];   // positions from Lc on get key 0 (never read)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int t = t4 + i;
                    const float coverage = (float)n4[i] * inv_l1;
                    const float pp = p4[i] + G.lambda * (i4[i] * (1.f - coverage));
                    out[i] = pp;
                    const bool kept = (pw[u] >> (t & 31)) & 1u;
                    kq[i] = (t < Lc && !kept) ? float_order_key(pp) : 0u;
                }
                *reinterpret_cast<uint4*>(keys + key_chunk(t4)) = make_uint4(kq[0], kq[1], kq[2], kq[3]);
                if (Pp) *reinterpret_cast<float4*>(Pp + t4) = make_float4(out[0], out[1], out[2], out[3]);
            }
        }
        __syncthreads();
        // The next layer's selection may be scheduled now: its staging overlaps
        // this top-k, then it waits for this grid.
        asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
        block_topk<2>(keys, Lc, G.f0, bits, sm);
        if (G.ada) {
            // Head-wise adaptive fill: the head keeps its own best f0.  A head
            // can win at most extras = Hkv * (k2 - f0) slots of the joint ranking
            // over the sequence's heads, and only its best ones: it offers its
            // nC best remaining candidates (ties to the lower position), in
            // position order, as candidates h * jpool + r of the joint ranking
            // (ada_kernel), so that ties there go to the lower head, then the
            // lower position.  The preserved tokens are exactly Kp of the Lc
            // candidates, so Lc - Kp - f0 remain.
            uint32_t* cbits = suni + G.words;   // after the union words: see select_smem_bytes
            for (int wd = tid; wd < wordsL; wd += NT) {
                uint32_t a = bits[wd];
                while (a) {
                    const int t = 32 * wd + __ffs(a) - 1;
                    a &= a - 1u;
                    keys[key_index(t)] = 0u;
                }
            }
            __syncthreads();
            const int nC = min(G.jpool, Lc - G.Kp - G.f0);
            block_topk<2>(keys, Lc, nC, cbits, sm);
            uint32_t* jk = sc.jkeys + (size_t)s * G.jstride;
            int32_t* jp = sc.jpos + (size_t)s * G.jstride;
            const int wpt = (wordsL + NT - 1) / NT;
            const int w_lo = min(tid * wpt, wordsL), w_hi = min(w_lo + wpt, wordsL);
            int mine = 0;
            for (int wd = w_lo; wd < w_hi; ++wd) mine += __popc(cbits[wd]);
            int total;
            int r = block_exclusive_sum(mine, sm.wsum, total);
            for (int wd = w_lo; wd < w_hi; ++wd) {
                uint32_t c = cbits[wd];
                while (c) {
                    const int t = 32 * wd + __ffs(c) - 1;
                    c &= c - 1u;
                    const int i = h * G.jpool + r++;
                    jk[key_index(i)] = keys[key_index(t)];
                    jp[i] = t;
                }
            }
            for (int r2 = total + tid; r2 < G.jpool; r2 += NT) {
                const int i = h * G.jpool + r2;
                jk[key_index(i)] = 0u;
                jp[i] = -1;
            }
        }
        for (int wd = tid; wd < wordsL; wd += NT) bits[wd] |= spres[wd] | range_bits(wd, Lc, L);
    } else {
        // Every token is kept; the slice's counts still move to the next array.
        for (int t4 = f0 + 4 * tid; t4 < min(f1, Lc & ~3); t4 += 4 * NT)
            *reinterpret_cast<uchar4*>(nB + t4) = counts4(t4, *reinterpret_cast<const uchar4*>(nA + t4));
        for (int wd = tid; wd < wordsL; wd += NT) bits[wd] = range_bits(wd, 0, L);
    }
    // The head's kept positions, for the gather and the next layer.
    uint32_t* out_bits = sl.sel + row * G.words;
    for (int wd = tid; wd < wordsL; wd += NT) out_bits[wd] = bits[wd];
    // For the next layer only: the counts of this slice outside the candidates
    // (the kept window; positions from L on keep what the array holds).
    for (int t4 = max(f0, Lc & ~3) + 4 * tid; t4 < f1; t4 += 4 * NT) {
        if (t4 + 4 <= Lc) continue;   // written with the candidates
        const uchar4 c = counts4(t4, *reinterpret_cast<const uchar4*>(nA + t4));
        if (t4 + 4 <= L) {
            *reinterpret_cast<uchar4*>(nB + t4) = c;
        } else {
            const uint8_t c4[4] = {c.x, c.y, c.z, c.w};
            for (int i = 0; t4 + i < L; ++i) nB[t4 + i] = c4[i];
        }
    }
}

constexpr int kAdaSmemKeys = 40960;   // joint candidates staged in shared memory (160 KB)
__host__ __device__ inline bool ada_keys_in_smem(const Geometry& g) { return g.Hkv * g.jpool <= kAdaSmemKeys; }

// Head-wise adaptive fill, second step: the extras = Hkv * (k2 - f0) best of
// the candidates the sequence's heads offered (select_kernel), ranked together
// (larger P', then lower head, then lower position), join their heads' kept
// positions.  Grid (batch); a programmatic dependent of the layer's
// select_kernel.
__global__ void __launch_bounds__(kSelectThreads) ada_kernel(Geometry G, LayerIO io, Scratch sc, Slot sl, int ncall) {
    __shared__ TopkShared sm;
    const int s = blockIdx.x, tid = threadIdx.x, NT = blockDim.x;
    const int n = G.Hkv * G.jpool, nwords = (n + 31) >> 5;
    uint32_t* jb = sc.jbits + (size_t)s * (G.jstride / 32);
    // The previous layer's ada_kernel completed before this layer's selection
    // started, so the winner bits can be cleared before the wait.
    for (int wd = tid; wd < nwords; wd += NT) jb[wd] = 0u;
    // The next kernel on this stream (the next layer's selection or the
    // finalize) waits for this grid itself: let it stage now.
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
    asm volatile("griddepcontrol.wait;\n" ::: "memory");
    const int L = io.cu[s + 1] - io.cu[s];
    const uint32_t ell0 = __ldcg(reinterpret_cast<const uint32_t*>(io.state + (size_t)s * G.state_stride));
    if (L <= G.budget || ell0 + (uint32_t)ncall > 255u) return;   // all kept, or a refused call
    // The radix select sweeps the keys once per digit: stage them in shared
    // memory when they fit (the launch gave ada_smem_bytes).
    const uint32_t* keys = sc.jkeys + (size_t)s * G.jstride;
    if (ada_keys_in_smem(G)) {
        extern __shared__ __align__(16) uint32_t skeys[];
        for (int i = 4 * tid; i < 32 * nwords; i += 4 * NT)
            *reinterpret_cast<uint4*>(skeys + i) = __ldcg(reinterpret_cast<const uint4*>(keys + i));
        keys = skeys;
    }
    __syncthreads();
    block_topk(keys, n, G.extras, jb, sm);
    // A thread takes a word of winner bits and loads the 32 positions behind it
    // at once (independent 16-byte loads, not one L2 round trip per winner).
    const int32_t* jp = sc.jpos + (size_t)s * G.jstride;
    uint32_t* sel = sl.sel + (size_t)s * G.Hkv * G.words;
    for (int wd = tid; wd < nwords; wd += NT) {
        const uint32_t b = jb[wd];
        if (!b) continue;
        int4 pos[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) pos[j] = __ldcg(reinterpret_cast<const int4*>(jp + 32 * wd) + j);
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            if (!((b >> j) & 1u)) continue;
            const int4 q = pos[j >> 2];
            const int t = (j & 3) == 0 ? q.x : (j & 3) == 1 ? q.y : (j & 3) == 2 ? q.z : q.w;
            atomicOr(&sel[(size_t)((32 * wd + j) / G.jpool) * G.words + (t >> 5)], 1u << (t & 31));
        }
    }
}

// After the last layer of a call: n_t of the state = the last count array plus
// the last union (the OR of the last layer's kept bits over heads), last_union
// = that union, layers_done and seqlen updated.  Grid (batch).
__global__ void __launch_bounds__(kSelectThreads) finalize_kernel(Geometry G, LayerIO io, Scratch sc, Slot last,
                                                                   int ncall) {
    const int s = blockIdx.x, tid = threadIdx.x, NT = blockDim.x;
    asm volatile("griddepcontrol.wait;\n" ::: "memory");
    const int L = io.cu[s + 1] - io.cu[s];
    const int wordsL = (L + 31) >> 5;
    uint8_t* st = io.state + (size_t)s * G.state_stride;
    const uint32_t ell0 = reinterpret_cast<const uint32_t*>(st)[0];
    if (ell0 + (uint32_t)ncall > 255u) return;   // the select kernels reported it and wrote nothing
    const int l = ncall - 1;
    uint8_t* nstate = st + G.state_n_off;
    const uint8_t* nlast = (l & 1) ? nstate : sc.nbuf + (size_t)s * G.nlen;   // written by the last layer
    const uint32_t* srow = last.sel + (size_t)s * G.Hkv * G.words;
    uint32_t* last_union = reinterpret_cast<uint32_t*>(st + G.state_union_off);
    for (int wd = tid; wd < G.words; wd += NT) {
        uint32_t u = 0u;
        if (wd < wordsL)
            for (int hh = 0; hh < G.Hkv; ++hh) u |= __ldcg(&srow[(size_t)hh * G.words + wd]);
        last_union[wd] = u;
    }
    __syncthreads();   // the union words are read back below by other threads
    for (int t4 = 4 * tid; t4 < L; t4 += 4 * NT) {
        const uchar4 a = *reinterpret_cast<const uchar4*>(nlast + t4);
        const uint32_t b = last_union[t4 >> 5] >> (t4 & 31);
        const uint8_t c4[4] = {(uint8_t)(a.x + (b & 1u)), (uint8_t)(a.y + ((b >> 1) & 1u)),
                               (uint8_t)(a.z + ((b >> 2) & 1u)), (uint8_t)(a.w + ((b >> 3) & 1u))};
        if (t4 + 4 <= L) {
            *reinterpret_cast<uchar4*>(nstate + t4) = make_uchar4(c4[0], c4[1], c4[2], c4[3]);
        } else {
            for (int i = 0; t4 + i < L; ++i) nstate[t4 + i] = c4[i];
        }
    }
    if (tid == 0) {
        reinterpret_cast<uint32_t*>(st)[0] = ell0 + (uint32_t)ncall;
        reinterpret_cast<uint32_t*>(st)[1] = (uint32_t)L;
    }
}

// out_idx[s,h,j] = position of the j-th kept bit of (s, h) (-1 past the last),
// j < cap (the budget, or the head capacity of the adaptive fill);
// out_k[s,h,j,:] = K[cu[s] + idx, h, :] (zeros for idx = -1); the same for V.
// Grid (ceil(cap/16), Hkv, batch), 256 threads: the block finds its 16 ranks from
// a prefix count over the row's bits words, then a half-warp moves one 256-byte row.
__global__ void __launch_bounds__(256) gather_kernel(Geometry G, LayerIO io, Slot sl) {
    __shared__ int wsum[32];
    __shared__ int spos[16];
    const int s = blockIdx.z, h = blockIdx.y;
    const int tid = threadIdx.x, NT = blockDim.x;
    const int lane = tid & 31, warp = tid >> 5;
    const int L = io.cu[s + 1] - io.cu[s];
    const int wordsL = (L + 31) >> 5;
    const size_t srow = (size_t)s * G.Hkv + h;
    const uint32_t* sel = sl.sel + srow * G.words;
    const int r0 = blockIdx.x * 16;
    if (tid < 16) spos[tid] = -1;
    // Contiguous runs of words per thread, ranked by an exclusive prefix sum.
    const int wpt = (wordsL + NT - 1) / NT;
    const int w_lo = min(tid * wpt, wordsL), w_hi = min(w_lo + wpt, wordsL);
    int mine = 0;
    for (int wd = w_lo; wd < w_hi; ++wd) mine += __popc(__ldcg(&sel[wd]));
    int total;
    int rank = block_exclusive_sum(mine, wsum, total);   // its barriers also order spos's initialisation
    if (rank < r0 + 16 && rank + mine > r0) {
        for (int wd = w_lo; wd < w_hi && rank < r0 + 16; ++wd) {
            uint32_t b = __ldcg(&sel[wd]);
            while (b && rank < r0 + 16) {
                const int bit = __ffs(b) - 1;
                b &= b - 1u;
                if (rank >= r0) spos[rank - r0] = wd * 32 + bit;
                ++rank;
            }
        }
    }
    __syncthreads();
    const int rloc = warp * 2 + (lane >> 4), sub = lane & 15;
    const int j = r0 + rloc;
    if (j >= G.cap) return;
    const size_t orow = srow * G.cap + j;
    const int idx = spos[rloc];
    if (sub == 0) io.out_idx[orow] = idx;
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

size_t select_smem_bytes(const Geometry& g) {
    const size_t head = ((size_t)4 * g.words + (keys_in_smem(g.ML) ? key_row_words(g) : 0) + 3) & ~(size_t)3;
    return sizeof(uint32_t) * (head + (scores_in_smem(g.ML) ? 2 * (size_t)g.ML : 0));
}

size_t heads_smem_bytes(const Geometry& g) {
    return sizeof(uint32_t) * ((((size_t)g.words + 3) & ~(size_t)3) + (keys_in_smem(g.ML) ? key_row_words(g) : 0));
}

cudaError_t configure_select() {
    const int need = (int)(sizeof(uint32_t) * (kSmemKeys / 32 + kSmemKeys));   // bits + one key row
    // The select kernel also keeps the preserved bits and caches P and I rows
    // up to kSmemScores positions.
    const int need_sel_keys = need + (int)(sizeof(uint32_t) * (3 * (kSmemKeys / 32) + 4));
    const int need_sel_scores =
        (int)(sizeof(uint32_t) * (4 * (kSmemScores / 32) + kSmemScores + 2 * kSmemScores + 64));
    const int need_sel = need_sel_keys > need_sel_scores ? need_sel_keys : need_sel_scores;
    cudaError_t e = cudaFuncSetAttribute(heads_topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, need);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(heads_pool_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kPoolSmemBytes);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, need_sel);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(ada_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)(sizeof(uint32_t) * (kAdaSmemKeys + 32)));
    return e;
}

cudaError_t launch_heads(const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl, cudaStream_t st,
                         int priority) {
    const dim3 grid(g.Hkv, g.batch);
    cudaError_t e = launch_prio(heads_pool_kernel, grid, dim3(kSelectThreads), g.NG > 1 ? (size_t)kPoolSmemBytes : 0, st,
                                priority, false, g, io, sc, sl);
    if (e == cudaSuccess)
        e = launch_prio(heads_topk_kernel, grid, dim3(kSelectThreads), heads_smem_bytes(g), st, priority,
                        /*programmatic=*/true, g, io, sc, sl);
    return e;
}

cudaError_t launch_select(const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl, const Slot* prev,
                          cudaStream_t st, int priority, int lcall, int ncall, bool programmatic) {
    const uint32_t* prev_sel = prev ? prev->sel : nullptr;
    return launch_prio(select_kernel, dim3(g.Hkv, g.batch), dim3(kSelectThreads), select_smem_bytes(g), st, priority,
                       programmatic, g, io, sc, sl, prev_sel, lcall, ncall);
}

cudaError_t launch_finalize(const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& last, cudaStream_t st,
                            int priority, int ncall) {
    return launch_prio(finalize_kernel, dim3(g.batch), dim3(kSelectThreads), 0, st, priority, /*programmatic=*/true, g,
                       io, sc, last, ncall);
}

cudaError_t launch_ada(const Geometry& g, const LayerIO& io, const Scratch& sc, const Slot& sl, cudaStream_t st,
                       int priority, int ncall) {
    // The staged keys: 32 * ceil(n / 32) words, the extent of a key row of n keys.
    const size_t smem = ada_keys_in_smem(g) ? sizeof(uint32_t) * 32 * (((size_t)g.Hkv * g.jpool + 31) / 32) : 0;
    return launch_prio(ada_kernel, dim3(g.batch), dim3(kSelectThreads), smem, st, priority, /*programmatic=*/true, g,
                       io, sc, sl, ncall);
}

void launch_gather(const Geometry& g, const LayerIO& io, const Slot& sl, cudaStream_t st) {
    gather_kernel<<<dim3((g.cap + 15) / 16, g.Hkv, g.batch), 256, 0, st>>>(g, io, sl);
}

}  // namespace kvec
