// dpb_encode_mma.cuh -- the §2.2 encoder with the child scoring of Eq. 6 on the
// tensor cores (bf16 inputs, beam up to 16, 16 children per parent). Instantiated
// per count of inverse-coordinate sign tables (dpb_encode_mma_n*.cu).
//
// Scoring. A warp owns two tokens at a time. At level l its 16 tensor-core
// rows are the (token, beam slot) pairs and the contraction is
//     score[row][j] = sum_iota (x_token (.) phi~_parent)[iota] * gamma_j[iota],
// rows x (.) phi~_p times the universal matrix Gamma_l (Eq. 6), by mma.sync
// m16n8k16 (bf16 x bf16 -> fp32). The A operand is never staged: each lane
// builds its fragment in registers as the bf16 bits of x XOR a sign mask. The
// K order is permuted so that the lane with q4 = lane % 4 holds coordinates
// q4 + 4j of every 32-coordinate block, paired (j, j+4): the two sign bits of
// a pair sit 16 apart in the parent's sign word over the block, and one shift
// moves both to the bf16 sign positions 15 and 31. The sign word of parent p
// over block m is
//     W5[p & 31] ^ (bit m of W5[(p_lo >> 5) & 31] ? ~0 : 0) ^ XOR_k VH_k[m][chunk_k(p_hi)],
// the Walsh, block-parity and inverse-coordinate parts of parity(M[iota] & p)
// (App. A.4 Eq. 26). Gamma_l lives in shared memory in B-fragment order.
//
// Selection (global mode, readings R8-R10). Every candidate is one 64-bit
// word, |z| bits above (2^31 - 1 - index) and the sign of z, so that larger
// words come first in the order (|z| descending, index ascending). Each token
// keeps its code as a sorted list of k words in shared memory:
//   level 0  the exact top k of the d coordinates: each lane keeps its best R
//            32-bit words (|x| bf16 bits, index, sign), the warp sorts the
//            union of 32 R and takes its k-th word tau; if exactly k
//            coordinates reach tau the union's first k are the top k
//            (otherwise, and with standardisation, a bisection path);
//   level l  the distinct children ahead of the list's k-th word are merged
//            in by rank (each entrant's place = entrants ahead of it + list
//            words ahead of it); the beam is the first 8 children, read from
//            those ranks, or from a warp tournament when fewer than 8 or more
//            than 32 children enter.
// The list after the last level is the code.
#pragma once

#include <algorithm>

#include "dpb_device.cuh"
#include "dpb_internal.h"
#include "dpb_select.cuh"

namespace dpb {
namespace mmaenc {

constexpr int kMaxWarps = 20;
constexpr int kBeam = 8;

struct Args {
    const __nv_bfloat16 *x;
    int64_t T;
    const float *mu, *sigma;
    const float2 *tab;  // packed (mu, 1 / sigma), nullable
    const uint32_t *coset;  // coset scoring tables (nullable): per level, g0's block sign words, then S_j
    int32_t *idx;
    float *val, *xnorm;
    int32_t *status;
    const uint32_t *frag, *G, *VH, *DD;
    int d, nblk, levels, k, t, ecap;
    int beam;  // B <= 8: beam slots B..7 hold no parent
    float inv_sqrt_d;
};

// ---- shared-memory layout (32-bit words) ------------------------------------------

__host__ __device__ inline int block_words(int levels, int nblk, int nkc) {
    // frag [(L-1)][nblk][2][32][4], W5 [32], VH [nkc][32][32], DD [(L-1)][kDedupSlots], G [L][16]
    return (levels - 1) * nblk * 256 + 32 + nkc * 1024 + (levels - 1) * kDedupSlots + 8 * 16;
}

// 64-bit entries of the per-warp scratch buffer: the entrants of a merge, the
// lists of the bisection path, and the parents' sign words of a level
// (16 rows x nblk blocks).
__host__ __device__ inline int entrant_cap(int k, int nblk) {
    int c = 128;
    while (c < k) c <<= 1;
    return c > 8 * nblk ? c : 8 * nblk;
}

__host__ __device__ inline int warp_words(int nblk, int k) {
    // x tile [2][nblk * 16], code lists [2][k] (64-bit), scratch [ecap]
    // (64-bit), beams [2][8], duplicate bits [8], spare [8]
    return 2 * nblk * 16 + 4 * k + 2 * entrant_cap(k, nblk) + 16 + 8 + 8;
}

// ---- candidate words ------------------------------------------------------------------

__device__ __forceinline__ uint64_t cword(float z, uint32_t idx) {
    const uint32_t b = __float_as_uint(z);
    return ((uint64_t)(b & 0x7fffffffu) << 32) | ((uint64_t)(0x7fffffffu - idx) << 1) | (b >> 31);
}
__device__ __forceinline__ uint32_t cword_idx(uint64_t c) { return 0x7fffffffu - ((uint32_t)c >> 1); }
__device__ __forceinline__ float cword_z(uint64_t c) {
    return __uint_as_float((uint32_t)(c >> 32) | ((uint32_t)c << 31));
}

// Level-0 word of bf16 coordinate i (< 2^15) with bits b: the same order in 32 bits.
__device__ __forceinline__ uint32_t cword0(uint32_t b, uint32_t i) {
    return ((b & 0x7fffu) << 16) | ((0x7fffu - i) << 1) | ((b >> 15) & 1u);
}
__device__ __forceinline__ uint64_t widen0(uint32_t c) {
    const uint32_t i = 0x7fffu - ((c >> 1) & 0x7fffu);
    return ((uint64_t)((c >> 16) << 16) << 32) | ((uint64_t)(0x7fffffffu - i) << 1) | (c & 1u);
}

// ---- helpers ----------------------------------------------------------------------

__device__ __forceinline__ void mma_bf16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Parts of parent p's sign words: its Walsh word, the block-parity word
// (bit m = parity(m AND u), u = bits 5..9 of p_lo: the Walsh word of u) and
// the byte offsets into VH_k[m], packed to a word.
struct ParentOff {
    uint32_t w5;  // the Walsh word (the same for every block)
    uint32_t pq;  // the block-parity word
    uint32_t o;   // VH_0, VH_1, VH_2 byte offsets (bytes 1..3)
    uint32_t o3;  // VH_3 byte offset
};

__device__ __forceinline__ ParentOff parent_offsets(uint32_t p, int t, const uint32_t *w5) {
    ParentOff po;
    po.w5 = w5[p & 31u];  // t >= 5: bits 0..4 belong to p_lo
    po.pq = w5[((p & ((1u << t) - 1u)) >> 5) & 31u];
    const uint32_t h0 = ((p >> t) & 31u) * 4u, h1 = ((p >> (t + 5)) & 31u) * 4u;
    const uint32_t h2 = ((p >> min(t + 10, 31)) & 31u) * 4u;
    const uint32_t h3 = ((p >> min(t + 15, 31)) & 31u) * 4u;
    po.o = (h0 << 8) | (h1 << 16) | (h2 << 24);
    po.o3 = h3;
    return po;
}

// Sign word of a parent over 32-coordinate block m (bit l = 1: coordinate
// 32 m + l of phi~_p is negative).
template <int NKC>
__device__ __forceinline__ uint32_t parent_signs(const ParentOff &po, const uint32_t *vh, int m) {
    const char *V = reinterpret_cast<const char *>(vh + m * 32);
    uint32_t s = po.w5 ^ (0u - ((po.pq >> m) & 1u)) ^
                 *reinterpret_cast<const uint32_t *>(V + __byte_perm(po.o, 0, 0x4441));
    s ^= *reinterpret_cast<const uint32_t *>(V + 4096 + __byte_perm(po.o, 0, 0x4442));
    if (NKC > 2) s ^= *reinterpret_cast<const uint32_t *>(V + 8192 + __byte_perm(po.o, 0, 0x4443));
    if (NKC > 3) s ^= *reinterpret_cast<const uint32_t *>(V + 12288 + po.o3);
    return s;
}

// Coordinate i of one token's row, read back from the permuted tile.
__device__ __forceinline__ float x_at(const uint16_t *xh, int i) {
    const int m = i >> 5, l = i & 31;
    return __uint_as_float((uint32_t)xh[(m * 16 + (l & 3) * 4 + ((l >> 2) & 3)) * 2 + (l >> 4)] << 16);
}

// z = (s - mu_c) / sigma_c (§2.2 score standardisation); identity without tables.
__device__ __forceinline__ float standardise(float s, uint32_t c, const Args &a, int32_t *status) {
    return a.mu ? zscore(s, c, a.mu, a.sigma, a.tab, status) : s;
}
// The same, fixed at compile time (STD: tables are given).
template <bool STD>
__device__ __forceinline__ float stdz(float s, uint32_t c, const Args &a, int32_t *status) {
    if constexpr (STD) return zscore(s, c, a.mu, a.sigma, a.tab, status);
    return s;
}

// bf16 element e (0..7) of a 16-byte chunk.
__device__ __forceinline__ uint32_t elem16(const uint4 &v, int e) {
    const uint32_t w = (e >> 1) == 0 ? v.x : (e >> 1) == 1 ? v.y : (e >> 1) == 2 ? v.z : v.w;
    return (w >> (16 * (e & 1))) & 0xffffu;
}

__device__ __forceinline__ unsigned lanes_below() { return (1u << (threadIdx.x & 31)) - 1u; }

// Appends the lane-distributed (z, id) entries with `take` set to a shared list
// at position n; returns the new length (warp-uniform).
__device__ __forceinline__ int warp_append(float *z, uint32_t *id, int n, bool take, float zv, uint32_t iv) {
    const unsigned mb = __ballot_sync(kFull, take);
    if (take) {
        const int pos = n + __popc(mb & lanes_below());
        z[pos] = zv;
        id[pos] = iv;
    }
    return n + __popc(mb);
}

// One compare-exchange stage (size, stride) of a warp bitonic sort,
// descending, of 32 R words held R per lane (element lane * R + r).
__device__ __forceinline__ uint32_t whi(uint32_t a, uint32_t b) { return max(a, b); }
__device__ __forceinline__ uint32_t wlo(uint32_t a, uint32_t b) { return min(a, b); }
__device__ __forceinline__ uint64_t whi(uint64_t a, uint64_t b) { return a > b ? a : b; }
__device__ __forceinline__ uint64_t wlo(uint64_t a, uint64_t b) { return a > b ? b : a; }

template <int R, typename W>
__device__ __forceinline__ void sort_stage(W (&v)[R], int size, int stride) {
    const int lane = threadIdx.x & 31;
    if (stride >= R) {
        // size >= 2 stride >= 2R: r never reaches the size bit of lane R + r
        const bool keep_hi = ((lane & (stride / R)) == 0) == (((lane * R) & size) == 0);
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const W o = __shfl_xor_sync(kFull, v[r], stride / R);
            v[r] = keep_hi ? whi(v[r], o) : wlo(v[r], o);
        }
    } else {
#pragma unroll
        for (int cs = 1; cs < R; cs <<= 1) {
            if (stride == cs) {
#pragma unroll
                for (int r = 0; r < R; ++r) {
                    const int q = r ^ cs;
                    if (q > r) {
                        const bool desc = (((lane * R + r) & size) == 0);
                        const W hi = whi(v[r], v[q]), lo = wlo(v[r], v[q]);
                        v[r] = desc ? hi : lo;
                        v[q] = desc ? lo : hi;
                    }
                }
            }
        }
    }
}

// Warp bitonic sort, descending. The stages are looped, not unrolled: the
// encoder's other phases already fill the instruction caches.
template <int R, typename W>
__device__ __forceinline__ void warp_sort_desc(W (&v)[R]) {
#pragma unroll 1
    for (int size = 2; size <= 32 * R; size <<= 1)
#pragma unroll 1
        for (int stride = size / 2; stride > 0; stride >>= 1) sort_stage<R, W>(v, size, stride);
}

__device__ __forceinline__ void cas_desc(uint64_t &a, uint64_t &b) {
    const uint64_t hi = a > b ? a : b, lo = a > b ? b : a;
    a = hi;
    b = lo;
}

// The first kBeam of up to 128 distinct candidate words held 4 per lane (0 =
// none), by kBeam rounds of a warp tournament over the lanes' sorted heads.
__device__ __forceinline__ void beam_tournament(uint64_t (&c)[4], uint32_t *beam) {
    cas_desc(c[0], c[1]);
    cas_desc(c[2], c[3]);
    cas_desc(c[0], c[2]);
    cas_desc(c[1], c[3]);
    cas_desc(c[1], c[2]);
#pragma unroll 1
    for (int r = 0; r < kBeam; ++r) {
        const uint32_t hi = (uint32_t)(c[0] >> 32), lo = (uint32_t)c[0];
        const uint32_t mh = __reduce_max_sync(kFull, hi);
        const uint32_t ml = __reduce_max_sync(kFull, hi == mh ? lo : 0u);
        if (hi == mh && lo == ml && (mh | ml) != 0u) {
            beam[r] = cword_idx(c[0]);
            c[0] = c[1];
            c[1] = c[2];
            c[2] = c[3];
            c[3] = 0ull;
        }
    }
    __syncwarp();
}

// The first nb (<= 16) of up to 256 distinct candidate words held 8 per lane
// (two groups of 4, 0 = none), by nb rounds of a warp tournament over the
// heads of the lanes' two sorted groups.
__device__ __forceinline__ void beam_tournament16(uint64_t (&c)[4], uint64_t (&d)[4], uint32_t *beam, int nb) {
    cas_desc(c[0], c[1]);
    cas_desc(c[2], c[3]);
    cas_desc(c[0], c[2]);
    cas_desc(c[1], c[3]);
    cas_desc(c[1], c[2]);
    cas_desc(d[0], d[1]);
    cas_desc(d[2], d[3]);
    cas_desc(d[0], d[2]);
    cas_desc(d[1], d[3]);
    cas_desc(d[1], d[2]);
#pragma unroll 1
    for (int r = 0; r < nb; ++r) {
        const bool fc = c[0] > d[0];
        const uint64_t head = fc ? c[0] : d[0];
        const uint32_t hi = (uint32_t)(head >> 32), lo = (uint32_t)head;
        const uint32_t mh = __reduce_max_sync(kFull, hi);
        const uint32_t ml = __reduce_max_sync(kFull, hi == mh ? lo : 0u);
        if (hi == mh && lo == ml && (mh | ml) != 0u) {
            beam[r] = cword_idx(head);
            if (fc) {
                c[0] = c[1];
                c[1] = c[2];
                c[2] = c[3];
                c[3] = 0ull;
            } else {
                d[0] = d[1];
                d[1] = d[2];
                d[2] = d[3];
                d[3] = 0ull;
            }
        }
    }
    __syncwarp();
}

// The same for lanes whose R words are already sorted descending: odd lanes
// reverse theirs (a bitonic merge of size 2R wants them ascending) and the
// sort starts at size 2R.
template <int R, typename W>
__device__ __forceinline__ void warp_sort_desc_runs(W (&v)[R]) {
    if (threadIdx.x & 1) {
#pragma unroll
        for (int r = 0; r < R / 2; ++r) {
            const W t = v[r];
            v[r] = v[R - 1 - r];
            v[R - 1 - r] = t;
        }
    }
#pragma unroll 1
    for (int size = 2 * R; size <= 32 * R; size <<= 1)
#pragma unroll 1
        for (int stride = size / 2; stride > 0; stride >>= 1) sort_stage<R, W>(v, size, stride);
}

// ---- merging entrants into a code list -------------------------------------------

// Merges the m entrant words E[0..m) (each ahead of L[k-1], any order) into
// the sorted list L of k words, 32 entrants at a time: an entrant's place is
// the entrants of its chunk ahead of it plus the list words ahead of it (a
// prefix of L, found by bisection); a list word moves down by the entrants
// ahead of it; whatever lands at k or beyond drops out. When 8..32 words enter
// and `beam` is given, the first 8 entrants become the beam.
//
// 8 to 32 entrants (the usual case) take another route, free of a loop over
// the entrants (its fixed cost loses to the loop below 8): each finds its gap
// in the list by bisection (pos = list words
// ahead of it) and a histogram H of the gaps (in E, past the entrants) gives
// by prefix sums how far each list word moves (the entrants in gaps at or
// before it) and how many entrants are ahead of each entrant (those in
// earlier gaps, and those of its own gap that are larger, compared directly).
template <int KPL>
__device__ __noinline__ void merge_sorted(uint64_t *L, int k, uint64_t *E, int m, uint32_t *beam) {
    const int lane = threadIdx.x & 31;
    const int top = 1 << (31 - __clz(k));  // the largest power of 2 <= k
    if (m >= 8 && m <= 32) {
        uint32_t *H = reinterpret_cast<uint32_t *>(E + 32);  // [k] entrants per gap
        const uint64_t mine = lane < m ? E[lane] : 0ull;
        uint64_t lv[KPL];
#pragma unroll
        for (int r = 0; r < KPL; ++r) {
            const int e = lane + 32 * r;
            lv[r] = e < k ? L[e] : 0ull;
            if (e < k) H[e] = 0u;
        }
        int pos = 0;  // list words ahead of mine (< k: an entrant is ahead of L[k-1])
        for (int step = top; step > 0; step >>= 1) {
            const int np = pos + step;
            if (np <= k && L[np - 1] > mine) pos = np;
        }
        __syncwarp();
        if (lane < m) atomicAdd(&H[pos], 1u);
        __syncwarp();
        // cum[r] = entrants in gaps 0 .. lane + 32 r: how far list word lane + 32 r moves
        int cum[KPL];
        int carry = 0;
#pragma unroll
        for (int r = 0; r < KPL; ++r) {
            const int e = lane + 32 * r;
            int v = e < k ? (int)H[e] : 0;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int t = __shfl_up_sync(kFull, v, o);
                if (lane >= o) v += t;
            }
            cum[r] = carry + v;
            carry += __shfl_sync(kFull, v, 31);
        }
        // entrants ahead of mine: those of the gaps before pos ...
        int rs = 0;
        const int q = pos - 1;
#pragma unroll
        for (int r = 0; r < KPL; ++r) {
            const int v = __shfl_sync(kFull, cum[r], q & 31);
            if (q >= 0 && (q >> 5) == r) rs = v;
        }
        // ... and the larger ones of its own gap (lanes past m never match)
        unsigned same = __match_any_sync(kFull, lane < m ? pos : -1 - lane) & ~(1u << lane);
        const int rounds = (int)__reduce_max_sync(kFull, (uint32_t)__popc(same));
        for (int it = 0; it < rounds; ++it) {
            const int src = same ? __ffs(same) - 1 : lane;
            same &= same - 1u;
            const uint64_t o = __shfl_sync(kFull, mine, src);
            rs += src != lane && o > mine;
        }
        __syncwarp();
        if (lane < m && rs + pos < k) L[rs + pos] = mine;
#pragma unroll
        for (int r = 0; r < KPL; ++r) {
            const int e = lane + 32 * r;
            if (e < k && e + cum[r] < k) L[e + cum[r]] = lv[r];
        }
        if (beam && m >= kBeam && lane < m && rs < kBeam) beam[rs] = cword_idx(mine);
        __syncwarp();
        return;
    }
    for (int q0 = 0; q0 < m; q0 += 32) {
        const int mq = min(32, m - q0);
        const uint64_t mine = lane < mq ? E[q0 + lane] : 0ull;
        uint64_t lv[KPL];
        int rl[KPL];
#pragma unroll
        for (int r = 0; r < KPL; ++r) {
            const int e = lane + 32 * r;
            lv[r] = e < k ? L[e] : 0ull;
            rl[r] = 0;
        }
        int rs = 0;  // entrants of this chunk ahead of mine
        for (int i = 0; i < mq; ++i) {
            const uint64_t s = E[q0 + i];
            rs += s > mine;
#pragma unroll
            for (int r = 0; r < KPL; ++r) rl[r] += s > lv[r];
        }
        int pos = 0;  // list words ahead of mine
        for (int step = top; step > 0; step >>= 1) {
            const int np = pos + step;
            if (np <= k && L[np - 1] > mine) pos = np;
        }
        __syncwarp();
        if (lane < mq && rs + pos < k) L[rs + pos] = mine;
#pragma unroll
        for (int r = 0; r < KPL; ++r) {
            const int e = lane + 32 * r;
            if (e < k && e + rl[r] < k) L[e + rl[r]] = lv[r];
        }
        if (beam && m >= kBeam && m <= 32 && lane < mq && rs < kBeam) beam[rs] = cword_idx(mine);
        __syncwarp();
    }
}

// Gathers the candidate words c[] (4 per lane, 0 = none) that are ahead of the
// list's k-th word into E (capacity >= 128) and merges them into L. Returns
// the number of entrants.
template <int KPL>
__device__ __forceinline__ int merge_entrants(uint64_t *L, int k, uint64_t *E, const uint64_t (&c)[4],
                                              uint32_t *beam) {
    const uint64_t tau = L[k - 1];
    int m = 0;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const bool take = c[e] > tau;
        const unsigned mb = __ballot_sync(kFull, take);
        if (take) E[m + __popc(mb & lanes_below())] = c[e];
        m += __popc(mb);
    }
    __syncwarp();
    merge_sorted<KPL>(L, k, E, m, beam);
    return m;
}

// ---- level 0 ----------------------------------------------------------------------

// Fast path (no standardisation, k <= 16 R): see the header comment. `row`
// is the token's row as 16-byte chunks (8 coordinates each); this lane reads
// chunks lane + 32 j. The union's first k go to the list; coordinates that
// reach its k-th word without being among their lane's R kept words (the
// extras; only lanes whose R kept words all reach it can have them, and the
// warp rescans just those, from L1) are merged in afterwards. Returns false,
// with nothing written, when more of them arrive than the scratch holds.
template <int R, int KPL>
__device__ __forceinline__ bool level0_union(const uint4 *row, int nch, int k, uint64_t *E, int ecap, uint64_t *L,
                                             uint32_t *beam) {
    const int lane = threadIdx.x & 31;
    uint32_t top[R];
#pragma unroll
    for (int r = 0; r < R; ++r) top[r] = 0u;
#pragma unroll 1
    for (int ch = lane; ch < nch; ch += 32) {
        const uint4 v = row[ch];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            uint32_t c = cword0(elem16(v, e), (uint32_t)(8 * ch + e));
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const uint32_t hi = max(top[r], c);
                c = min(top[r], c);
                top[r] = hi;
            }
        }
    }
    const uint32_t kept_min = top[R - 1];  // every word of this lane below it was not kept
    warp_sort_desc_runs<R>(top);
    uint32_t mine = 0u;
#pragma unroll
    for (int r = 0; r < R; ++r)
        if (r == (k - 1) % R) mine = top[r];
    const uint32_t tau = __shfl_sync(kFull, mine, (k - 1) / R);
    // Extras are unkept words in [tau, kept_min): only lanes whose R kept
    // words all reach tau can have them. The warp rescans just those lanes'
    // coordinates together (a few per lane), gathering the extras into E.
    const bool flag = kept_min >= tau && kept_min != 0u;
    const unsigned fm = __ballot_sync(kFull, flag);
    const int nf = __popc(fm), ne = 8 * ((nch + 31) / 32);  // flagged lanes; coordinate slots per lane
    const int cap = ecap - 16;                               // E's last 16 entries hold the flagged lanes
    int total = 0;
    if (nf) {
        uint32_t *fl = reinterpret_cast<uint32_t *>(E + cap);
        if (flag) fl[__popc(fm & lanes_below())] = (uint32_t)lane;
        __syncwarp();
        const uint16_t *xs = reinterpret_cast<const uint16_t *>(row);
#pragma unroll 1
        for (int q0 = 0; q0 < nf * ne; q0 += 32) {
            const int q = q0 + lane, f = q / ne, j = q - f * ne;
            const int owner = q < nf * ne ? (int)fl[f] : 0;
            const int ch = owner + 32 * (j >> 3), i = 8 * ch + (j & 7);
            const uint32_t km = __shfl_sync(kFull, kept_min, owner);
            uint32_t w = 0u;
            if (q < nf * ne && ch < nch) w = cword0(xs[i], (uint32_t)i);
            const bool take = w >= tau && w < km && w != 0u;
            const unsigned mb = __ballot_sync(kFull, take);
            const int pos = total + __popc(mb & lanes_below());
            if (take && pos < cap) E[pos] = widen0(w);
            total += __popc(mb);
        }
        __syncwarp();
    }
    if (total > cap) return false;
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const int e = lane * R + r;
        if (e < k) L[e] = widen0(top[r]);
    }
    if (total > 0) {
        __syncwarp();
        merge_sorted<KPL>(L, k, E, total, nullptr);
        if (lane < kBeam) beam[lane] = cword_idx(L[lane]);
    } else {
#pragma unroll
        for (int r = 0; r < R; ++r)
            if (lane * R + r < kBeam) beam[lane * R + r] = 0x7fffu - ((top[r] >> 1) & 0x7fffu);
    }
    __syncwarp();
    return true;
}

// Level 0 with standardisation tables: the union path above on 64-bit words
// of z = (x_i - mu_i) / sigma_i (a standardised score does not fit the 16-bit
// key of a bf16 coordinate). Each lane keeps its R best words; the k-th of the
// union is the threshold, and the few words at or above it that a lane did not
// keep (found by rescanning only the lanes that can hold them) are merged in.
// Returns false (nothing written) when they overflow E.
template <int R, int KPL>
__device__ __forceinline__ bool level0_union_std(const Args &a, const uint16_t *xh, int k, uint64_t *E, int ecap,
                                                 uint64_t *L, uint32_t *beam) {
    const int lane = threadIdx.x & 31, d = a.d;
    uint64_t top[R];
#pragma unroll
    for (int r = 0; r < R; ++r) top[r] = 0ull;
#pragma unroll 1
    for (int i = lane; i < d; i += 32) {
        uint64_t c = cword(standardise(x_at(xh, i), (uint32_t)i, a, a.status), (uint32_t)i);
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const uint64_t hi = whi(top[r], c);
            c = wlo(top[r], c);
            top[r] = hi;
        }
    }
    const uint64_t kept_min = top[R - 1];  // every word of this lane below it was not kept
    warp_sort_desc_runs<R>(top);
    uint64_t mine = 0ull;
#pragma unroll
    for (int r = 0; r < R; ++r)
        if (r == (k - 1) % R) mine = top[r];
    const uint64_t tau = __shfl_sync(kFull, mine, (k - 1) / R);
    // Extras are unkept words in [tau, kept_min): only lanes whose R kept
    // words all reach tau can have them. The warp rescans just those lanes'
    // coordinates (lane l owns l + 32 j) together, a few per lane, each with
    // its table entries, gathering the extras into E.
    const bool flag = kept_min >= tau && kept_min != 0ull;
    const unsigned fm = __ballot_sync(kFull, flag);
    const int nf = __popc(fm), ne = (d + 31) / 32;  // flagged lanes; coordinates per lane
    const int cap = ecap - 16;                      // E's last 16 entries hold the flagged lanes
    int total = 0;
    if (nf) {
        uint32_t *fl = reinterpret_cast<uint32_t *>(E + cap);
        if (flag) fl[__popc(fm & lanes_below())] = (uint32_t)lane;
        __syncwarp();
#pragma unroll 1
        for (int q0 = 0; q0 < nf * ne; q0 += 32) {
            const int q = q0 + lane, f = q / ne, j = q - f * ne;
            const int owner = q < nf * ne ? (int)fl[f] : 0;
            const int i = owner + 32 * j;
            const uint64_t km = __shfl_sync(kFull, kept_min, owner);
            uint64_t w = 0ull;
            if (q < nf * ne && i < d) w = cword(standardise(x_at(xh, i), (uint32_t)i, a, nullptr), (uint32_t)i);
            const bool take = w >= tau && w < km && w != 0ull;
            const unsigned mb = __ballot_sync(kFull, take);
            const int pos = total + __popc(mb & lanes_below());
            if (take && pos < cap) E[pos] = w;
            total += __popc(mb);
        }
        __syncwarp();
    }
    if (total > cap) return false;
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const int e = lane * R + r;
        if (e < k) L[e] = top[r];
    }
    if (total > 0) {
        __syncwarp();
        merge_sorted<KPL>(L, k, E, total, nullptr);
        if (lane < kBeam) beam[lane] = cword_idx(L[lane]);
    } else {
#pragma unroll
        for (int r = 0; r < R; ++r)
            if (lane * R + r < kBeam) beam[lane * R + r] = cword_idx(top[r]);
    }
    __syncwarp();
    return true;
}

// General path: every coordinate (standardised if tables are given) is a
// candidate; a threshold that at least k of them reach keeps them in the
// scratch (z, id) lists of capacity `cap`, the k-th is found by bisection, and
// the first k, sorted, become the code list; its first 8 are the beam.
template <bool STD>
__device__ __forceinline__ void level0_bisect(const Args &a, const uint16_t *xh, float *pz, uint32_t *pid, int cap,
                                              uint64_t *L, uint32_t *beam) {
    const int lane = threadIdx.x & 31, d = a.d, k = a.k;
    const int lowbit = STD ? 0 : 16;  // keys of unstandardised bf16 values have 16 zero bits
    // Each lane's R best keys, R = 2 ceil(k / 32) (at most 8): their union
    // holds at least k keys, and its k-th largest is a threshold that at least
    // k candidates reach and, unlike the smallest of the lanes' R-th keys,
    // only a few more.
    const int R = min(8, 2 * ((k + 31) >> 5));
    uint32_t best[8];
#pragma unroll
    for (int r = 0; r < 8; ++r) best[r] = 0u;
    for (int i = lane; i < d; i += 32) {
        uint32_t kv = akey(stdz<STD>(x_at(xh, i), (uint32_t)i, a, a.status)) + 1u;
#pragma unroll
        for (int r = 0; r < 8; ++r) {
            if (r < R && kv > best[r]) {
                const uint32_t tmp = best[r];
                best[r] = kv;
                kv = tmp;
            }
        }
    }
    uint32_t tau_low = 0;  // the union's k-th largest key, bit by bit
    for (int b = 31; b >= 0; --b) {
        const uint32_t c = tau_low | (1u << b);
        int cnt = 0;
#pragma unroll
        for (int r = 0; r < 8; ++r) cnt += r < R && best[r] >= c;
        if ((int)__reduce_add_sync(kFull, (uint32_t)cnt) >= k) tau_low = c;
    }
    int n = 0;
    bool overflow = false;
    for (int i0 = 0; i0 < d && !overflow; i0 += 32) {
        const int i = i0 + lane;
        float z = 0.f;
        bool take = false;
        if (i < d) {
            z = stdz<STD>(x_at(xh, i), (uint32_t)i, a, nullptr);
            take = akey(z) + 1u >= tau_low;
        }
        if (n + __popc(__ballot_sync(kFull, take)) > cap) {
            overflow = true;  // many equal keys at the threshold
        } else {
            n = warp_append(pz, pid, n, take, z, (uint32_t)i);
        }
    }
    __syncwarp();
    if (overflow) {
        // exact k-th key over the whole row, then every entry above it and the
        // first ties by index
        uint32_t tau = 0;
        for (int b = 30; b >= lowbit; --b) {
            const uint32_t c = tau | (1u << b);
            int cnt = 0;
            for (int i = lane; i < d; i += 32)
                cnt += akey(stdz<STD>(x_at(xh, i), (uint32_t)i, a, nullptr)) >= c;
            if (__reduce_add_sync(kFull, cnt) >= k) tau = c;
        }
        n = 0;
        for (int i0 = 0; i0 < d; i0 += 32) {
            const int i = i0 + lane;
            float z = 0.f;
            if (i < d) z = stdz<STD>(x_at(xh, i), (uint32_t)i, a, nullptr);
            n = warp_append(pz, pid, n, i < d && akey(z) > tau, z, (uint32_t)i);
        }
        for (int i0 = 0; i0 < d && n < k; i0 += 32) {
            const int i = i0 + lane;
            float z = 0.f;
            bool tie = false;
            if (i < d) {
                z = stdz<STD>(x_at(xh, i), (uint32_t)i, a, nullptr);
                tie = akey(z) == tau;
            }
            const unsigned mb = __ballot_sync(kFull, tie);
            const int rank = __popc(mb & lanes_below());
            if (tie && n + rank < k) {
                pz[n + rank] = z;
                pid[n + rank] = (uint32_t)i;
            }
            n = min(k, n + __popc(mb));
        }
        __syncwarp();
    }
    uint32_t tk, ti;
    warp_kth(pz, pid, n, k, lowbit, tk, ti);
    n = warp_compact_keep(pz, pid, n, tk, ti);
    int sc = 32;
    while (sc < n) sc <<= 1;
    warp_sort(pz, pid, n, sc);
    for (int e = lane; e < k; e += 32) L[e] = cword(pz[e], pid[e]);
    if (lane < kBeam) beam[lane] = pid[lane];
    __syncwarp();
}

// ---- the kernel ---------------------------------------------------------------------

// COSET: the generators of every level are one coset g0 ^ {0..15} (a variant
// outside the paper), and a parent's 16 child scores are the 16-point
// Walsh-Hadamard transform of its bucket sums B_u = sum over iota = u mod 16
// of x (.) phi~_{p ^ g0}; the shared memory of the B fragments holds the coset
// tables instead.
// WIDE: beams of 9 to 16. A warp then owns one token, whose beam slots
// 0..7 and 8..15 take the places of the two tokens (same x, one code list);
// repeats are found over all 120 slot pairs and the next beam is the top of
// both halves' children.
// STD: standardisation tables are given (a separate instantiation, so that
// the plain kernel carries none of their code).
template <int NKC, int KPL, bool COSET, bool WIDE, bool STD>
__global__ void __launch_bounds__(kMaxWarps * 32, 1) encode_kernel(Args a) {
    extern __shared__ __align__(16) uint32_t smem[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    const int d = a.d, nblk = a.nblk, L = a.levels, k = a.k, t = a.t;
    const int q4 = lane & 3, slot = lane >> 2;

    uint32_t *s_frag = smem;
    uint32_t *s_w5 = s_frag + (L - 1) * nblk * 256;
    uint32_t *s_vh = s_w5 + 32;
    uint32_t *s_dd = s_vh + NKC * 1024;
    uint32_t *s_g = s_dd + (L - 1) * kDedupSlots;
    {
        if (COSET) {
            for (int i = threadIdx.x; i < (L - 1) * (nblk + 16); i += blockDim.x) s_frag[i] = a.coset[i];
        } else {
            const uint4 *src = reinterpret_cast<const uint4 *>(a.frag);
            uint4 *dst = reinterpret_cast<uint4 *>(s_frag);
            for (int i = threadIdx.x; i < (L - 1) * nblk * 64; i += blockDim.x) dst[i] = src[i];
        }
        for (int v = threadIdx.x; v < 32; v += blockDim.x) {
            uint32_t word = 0;
            for (int l = 0; l < 32; ++l) word |= (uint32_t)(__popc(l & v) & 1) << l;
            s_w5[v] = word;
        }
        for (int i = threadIdx.x; i < NKC * 1024; i += blockDim.x) s_vh[i] = a.VH[i];
        for (int i = threadIdx.x; i < (L - 1) * kDedupSlots; i += blockDim.x) s_dd[i] = a.DD[i];
        for (int i = threadIdx.x; i < L * 16; i += blockDim.x) s_g[i] = a.G[(i >> 4) * DPB_MAX_CHILDREN + (i & 15)];
    }
    __syncthreads();

    uint32_t *xt = smem + block_words(L, nblk, NKC) + warp * warp_words(nblk, k);
    uint64_t *codes = reinterpret_cast<uint64_t *>(xt + 2 * nblk * 16);  // [2][k]
    uint64_t *E = codes + 2 * k;                                          // [ecap]
    uint32_t *beams = reinterpret_cast<uint32_t *>(E + a.ecap);           // [2][8]
    uint32_t *dup = beams + 16;                                           // [4]
    uint16_t *xh = reinterpret_cast<uint16_t *>(xt);
    const int nch = d / 8;  // 16-byte chunks of a row
    // the lane-th slot pair (sp, s), sp < s, of the beam
    const int ps = 1 + (lane >= 1) + (lane >= 3) + (lane >= 6) + (lane >= 10) + (lane >= 15) + (lane >= 21);
    const int psp = lane - ps * (ps - 1) / 2;
    const int64_t npairs = WIDE ? a.T : (a.T + 1) / 2;

    for (int64_t pr = (int64_t)blockIdx.x * nwarps + warp; pr < npairs; pr += (int64_t)gridDim.x * nwarps) {
        const int64_t t0 = WIDE ? pr : 2 * pr;
        const int ntok = WIDE ? 1 : (t0 + 1 < a.T ? 2 : 1);
        const int nhalf = WIDE ? 2 : ntok;  // row groups of 8 beam slots

        // ---- each row into the permuted tile; |x|; level 0 ----
        for (int tk = 0; tk < ntok; ++tk) {
            const uint4 *row = reinterpret_cast<const uint4 *>(a.x + (t0 + tk) * d);
            float ss = 0.f;
#pragma unroll 3  // the row's loads in flight together (3 chunks per lane at d = 768)
            for (int ch = lane; ch < nch; ch += 32) {
                const uint4 v = row[ch];
                const int m = ch >> 2, l0 = (ch & 3) * 8, half = l0 >> 4, pb = (l0 & 15) >> 2;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const uint32_t bits = elem16(v, e);
                    xh[(tk * nblk * 16 + m * 16 + (e & 3) * 4 + pb + (e >> 2)) * 2 + half] = (uint16_t)bits;
                    const float xf = __uint_as_float(bits << 16);
                    ss = fmaf(xf, xf, ss);
                }
            }
            ss = warp_sum(ss);
            if (lane == 0 && a.xnorm) a.xnorm[t0 + tk] = sqrtf(ss);
            __syncwarp();
            uint64_t *Lt = codes + tk * k;
            uint32_t *bt = beams + tk * kBeam;
            bool done = false;
            // each lane keeps R words, so the union of 32 R holds at least 2 k
            if constexpr (KPL <= 4) {
                if constexpr (STD)
                    done = level0_union_std<(KPL <= 2 ? 4 : 8), KPL>(a, xh + tk * nblk * 32, k, E, a.ecap, Lt, bt);
                else
                    done = level0_union<(KPL <= 2 ? 4 : 8), KPL>(row, nch, k, E, a.ecap, Lt, bt);
            }
            if (!done)
                level0_bisect<STD>(a, xh + tk * nblk * 32, reinterpret_cast<float *>(E),
                              reinterpret_cast<uint32_t *>(E) + a.ecap, a.ecap, Lt, bt);
            if constexpr (WIDE) {  // the beam: the first 16 of the sorted list (k >= beam)
                if (lane < 16) beams[lane] = cword_idx(Lt[lane]);
                __syncwarp();
            }
        }

        // ---- levels 1 .. L-1 ----
        for (int l = 1; l < L; ++l) {
            const uint32_t *frag = s_frag + (l - 1) * nblk * 256;
            // this lane's tensor-core rows: (token 0, slot) and (token 1, slot)
            const uint32_t p0 = beams[slot];
            const uint32_t p1 = nhalf > 1 ? beams[kBeam + slot] : 0u;
            // sign words of the 16 rows' parents over every block, row 2 slot + token
            uint2 *sgn = reinterpret_cast<uint2 *>(E);  // [nblk][8] (token 0, token 1)
            {
                const int row = lane & 15;
                const uint32_t pr = (row & 1) && nhalf < 2 ? 0u : beams[(row & 1) * kBeam + (row >> 1)];
                const ParentOff po = parent_offsets(pr, t, s_w5);
                uint32_t *sw = reinterpret_cast<uint32_t *>(E);
                for (int m = lane >> 4; m < nblk; m += 2) sw[m * 16 + row] = parent_signs<NKC>(po, s_vh, m);
            }
            __syncwarp();
            float sc[2][4];  // [token][2 h + (r & 1)]: this lane's children 8 h + 2 q4 + (r & 1)
            if constexpr (COSET) {
                // lane owns coordinates iota = 32 m + lane, all in bucket lane % 16;
                // row (token tk, slot s) adds x_tk[iota] (-1)^{sign of p_s,tk ^ g0}
                const uint32_t *cw = s_frag + (l - 1) * (nblk + 16);
                const int wl = ((lane & 3) << 2) | (((lane & 15) >> 3) << 1) | ((lane >> 2) & 1), hl = lane >> 4;
                float part[16];  // [tk * 8 + s]
#pragma unroll
                for (int r = 0; r < 16; ++r) part[r] = 0.f;
#pragma unroll 1
                for (int m = 0; m < nblk; ++m) {
                    const uint32_t gw = cw[m];
                    const float x0 = __uint_as_float((uint32_t)xh[(m * 16 + wl) * 2 + hl] << 16);
                    const float x1 = __uint_as_float((uint32_t)xh[((WIDE ? 0 : nblk * 16) + m * 16 + wl) * 2 + hl] << 16);
#pragma unroll
                    for (int sl = 0; sl < 8; ++sl) {
                        const uint2 sg = sgn[m * 8 + sl];
                        part[sl] += flip(x0, ((sg.x ^ gw) << (31 - lane)) & 0x80000000u);
                        part[8 + sl] += flip(x1, ((sg.y ^ gw) << (31 - lane)) & 0x80000000u);
                    }
                }
                uint32_t sj[4];  // S of this lane's 4 children: the WHT index that scores each
#pragma unroll
                for (int e = 0; e < 4; ++e) sj[e] = cw[nblk + 8 * (e >> 1) + 2 * q4 + (e & 1)];
#pragma unroll
                for (int r = 0; r < 16; ++r) {
                    float v = part[r] + __shfl_xor_sync(kFull, part[r], 16);  // bucket lane % 16
#pragma unroll
                    for (int b = 1; b < 16; b <<= 1) {
                        const float o = __shfl_xor_sync(kFull, v, b);
                        v = (lane & b) ? o - v : v + o;
                    }
                    // lane u now holds the score of child S = u of row r
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float got = __shfl_sync(kFull, v, (int)sj[e]) * a.inv_sqrt_d;
                        if ((r & 7) == slot) sc[r >> 3][e] = got;
                    }
                }
            } else {
                float acc[2][2][2][4];  // [m & 1][chunk][n-half][reg]
#pragma unroll
                for (int u = 0; u < 2; ++u)
#pragma unroll
                    for (int c = 0; c < 2; ++c)
#pragma unroll
                        for (int h = 0; h < 2; ++h)
#pragma unroll
                            for (int r = 0; r < 4; ++r) acc[u][c][h][r] = 0.f;
                const uint4 *xa = reinterpret_cast<const uint4 *>(xt) + q4;
                const uint4 *xb = reinterpret_cast<const uint4 *>(xt + (WIDE ? 0 : nblk * 16)) + q4;
                const uint4 *fr = reinterpret_cast<const uint4 *>(frag) + lane;
                const int sh = 15 - q4;
#pragma unroll 2
                for (int m = 0; m < nblk; ++m) {
                    const uint4 va = xa[m * 4], vb = xb[m * 4];
                    const uint2 sg = sgn[m * 8 + slot];
                    const uint32_t s0 = sg.x, s1 = sg.y;
                    const uint4 f0 = fr[m * 64], f1 = fr[m * 64 + 32];
                    // chunk 0 holds pairs 0 and 1 of the block, chunk 1 pairs 2 and 3
                    const uint32_t a00 = va.x ^ ((s0 << sh) & 0x80008000u);
                    const uint32_t a01 = vb.x ^ ((s1 << sh) & 0x80008000u);
                    const uint32_t a02 = va.y ^ ((s0 << (sh - 4)) & 0x80008000u);
                    const uint32_t a03 = vb.y ^ ((s1 << (sh - 4)) & 0x80008000u);
                    const uint32_t a10 = va.z ^ ((s0 << (sh - 8)) & 0x80008000u);
                    const uint32_t a11 = vb.z ^ ((s1 << (sh - 8)) & 0x80008000u);
                    const uint32_t a12 = va.w ^ ((s0 << (sh - 12)) & 0x80008000u);
                    const uint32_t a13 = vb.w ^ ((s1 << (sh - 12)) & 0x80008000u);
                    float(&cc)[2][2][4] = acc[m & 1];
                    mma_bf16(cc[0][0], a00, a01, a02, a03, f0.x, f0.y);
                    mma_bf16(cc[0][1], a00, a01, a02, a03, f0.z, f0.w);
                    mma_bf16(cc[1][0], a10, a11, a12, a13, f1.x, f1.y);
                    mma_bf16(cc[1][1], a10, a11, a12, a13, f1.z, f1.w);
                }
                // accumulator (n-half h, register r): row slot (r < 2) or slot + 8
                // (r >= 2), child 8 h + 2 q4 + (r & 1)
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int r = 0; r < 4; ++r)
                        sc[r >> 1][2 * h + (r & 1)] =
                            ((acc[0][0][h][r] + acc[0][1][h][r]) + (acc[1][0][h][r] + acc[1][1][h][r])) * a.inv_sqrt_d;
            }
            const uint32_t *gl = s_g + l * 16;
            if constexpr (STD) {  // standardise both rows' children now: their table loads go out together
#pragma unroll
                for (int tk = 0; tk < 2; ++tk)
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        if (tk < nhalf)
                            sc[tk][e] = standardise(sc[tk][e], (tk ? p1 : p0) ^ gl[8 * (e >> 1) + 2 * q4 + (e & 1)],
                                                    a, a.status);
            }
            const uint32_t *ddl = s_dd + (l - 1) * kDedupSlots;
            uint32_t pcur = p0;
            if constexpr (WIDE) {
                // repeats over all pairs S' < S < beam of the 16 slots: pair q = lane + 32 r
                if (lane < 8) dup[lane] = 0u;
                __syncwarp();
#pragma unroll 1
                for (int q = lane; q < 120; q += 32) {
                    int S = (int)((1.f + sqrtf(8.f * (float)q + 1.f)) * 0.5f);
                    while (S * (S - 1) / 2 > q) --S;
                    while ((S + 1) * S / 2 <= q) ++S;
                    const int Sp = q - S * (S - 1) / 2;
                    if (S >= a.beam) continue;
                    const uint32_t delta = beams[S] ^ beams[Sp];
                    uint32_t h = dedup_hash(delta);
                    for (int probe = 0; probe < kDedupSlots; ++probe) {
                        const uint32_t ent = ddl[h];
                        if (ent == 0u) break;
                        if ((ent >> 4) == delta + 1u) {
                            const uint32_t bit = (uint32_t)S * 16u + (ent & 15u);
                            atomicOr(&dup[bit >> 5], 1u << (bit & 31u));
                        }
                        h = (h + 1u) & (kDedupSlots - 1);
                    }
                }
                __syncwarp();
            }
            uint64_t cw0[4] = {0ull, 0ull, 0ull, 0ull};  // WIDE: the first half's candidate words
            for (int tk = 0; tk < nhalf; ++tk) {
                uint32_t *bt = beams + tk * kBeam;
                uint64_t *Lt = codes + (WIDE ? 0 : tk * k);
                // ---- duplicate children (R8): p_s ^ g_j' == p_s' ^ g_j with s' < s
                // exactly when p_s ^ p_s' == g_j ^ g_j'; slot s's copy is dropped
                uint32_t dmask = 0u;
                if constexpr (WIDE) {
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const uint32_t bit =
                            (uint32_t)(8 * tk + slot) * 16u + (uint32_t)(8 * (e >> 1) + 2 * q4 + (e & 1));
                        dmask |= ((dup[bit >> 5] >> (bit & 31u)) & 1u) << e;
                    }
                } else {
                    uint32_t delta = 0u;
                    bool hit = false;
                    if (lane < 28 && ps < a.beam) {  // both slots hold parents
                        delta = bt[ps] ^ bt[psp];
                        uint32_t h = dedup_hash(delta);
                        for (int probe = 0; probe < kDedupSlots; ++probe) {
                            const uint32_t ent = ddl[h];
                            if (ent == 0u) break;
                            if ((ent >> 4) == delta + 1u) {
                                hit = true;
                                break;
                            }
                            h = (h + 1u) & (kDedupSlots - 1);
                        }
                    }
                    if (__any_sync(kFull, hit)) {
                        if (lane < 4) dup[lane] = 0u;
                        __syncwarp();
                        if (hit) {
                            uint32_t h = dedup_hash(delta);
                            for (int probe = 0; probe < kDedupSlots; ++probe) {
                                const uint32_t ent = ddl[h];
                                if (ent == 0u) break;
                                if ((ent >> 4) == delta + 1u) {
                                    const uint32_t bit = (uint32_t)ps * 16u + (ent & 15u);
                                    atomicOr(&dup[bit >> 5], 1u << (bit & 31u));
                                }
                                h = (h + 1u) & (kDedupSlots - 1);
                            }
                        }
                        __syncwarp();
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const uint32_t bit = (uint32_t)slot * 16u + (uint32_t)(8 * (e >> 1) + 2 * q4 + (e & 1));
                            dmask |= ((dup[bit >> 5] >> (bit & 31u)) & 1u) << e;
                        }
                        __syncwarp();
                    }
                }
                // ---- this lane's 4 children of token tk as candidate words
                // (token 1's parent and scores move to token 0's registers after it)
                uint64_t c[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const uint32_t ci = pcur ^ gl[8 * (e >> 1) + 2 * q4 + (e & 1)];
                    const float z = sc[0][e];  // standardised above
                    // (WIDE: tk is the half of the beam; otherwise the token)
                    c[e] = ((dmask >> e) & 1u) || (WIDE ? 8 * tk + slot : slot) >= a.beam ? 0ull : cword(z, ci);
                    sc[0][e] = sc[1][e];
                }
                pcur = p1;
                const bool next = l + 1 < L;
                const int m = merge_entrants<KPL>(Lt, k, E, c, next && !WIDE ? bt : nullptr);
                if constexpr (WIDE) {
                    if (tk == 0) {
#pragma unroll
                        for (int e = 0; e < 4; ++e) cw0[e] = c[e];
                    } else if (next) {
                        beam_tournament16(cw0, c, beams, a.beam);
                    }
                } else {
                    if (next && (m < kBeam || m > 32)) beam_tournament(c, bt);
                }
                __syncwarp();
            }
        }

        // ---- the code of each token ----
        for (int tk = 0; tk < ntok; ++tk) {
            const uint64_t *Lt = codes + tk * k;
            const int64_t row = t0 + tk;
#pragma unroll
            for (int r = 0; r < KPL; ++r) {
                const int e = lane + 32 * r;
                if (e < k) {
                    const uint64_t w = Lt[e];
                    a.idx[row * k + e] = (int32_t)cword_idx(w);
                    a.val[row * k + e] = cword_z(w);
                }
            }
        }
        __syncwarp();
    }
}

template <int NKC, int KPL, bool COSET, bool WIDE, bool STD>
cudaError_t launch_kpl_std(const dpb_plan *p, const Args &a, int warps, cudaStream_t stream) {
    const size_t smem = encode_mma_smem(p, warps);
    const cudaError_t e = allow_smem((const void *)encode_kernel<NKC, KPL, COSET, WIDE, STD>, smem);
    if (e != cudaSuccess) return e;
    const int64_t pairs = WIDE ? a.T : (a.T + 1) / 2;
    const int grid = (int)std::min<int64_t>((pairs + warps - 1) / warps, (int64_t)std::max(p->sms, 1));
    encode_kernel<NKC, KPL, COSET, WIDE, STD><<<grid, warps * 32, smem, stream>>>(a);
    return cudaGetLastError();
}

template <int NKC, int KPL, bool COSET, bool WIDE = false>
cudaError_t launch_kpl(const dpb_plan *p, const Args &a, int warps, cudaStream_t stream) {
    return a.mu ? launch_kpl_std<NKC, KPL, COSET, WIDE, true>(p, a, warps, stream)
                : launch_kpl_std<NKC, KPL, COSET, WIDE, false>(p, a, warps, stream);
}

template <int NKC>
cudaError_t launch_nkc(const dpb_plan *p, const Args &a, int warps, cudaStream_t stream) {
    if (a.beam > kBeam) {
        if (a.k <= 32) return launch_kpl<NKC, 1, false, true>(p, a, warps, stream);
        if (a.k <= 64) return launch_kpl<NKC, 2, false, true>(p, a, warps, stream);
        if (a.k <= 128) return launch_kpl<NKC, 4, false, true>(p, a, warps, stream);
        return launch_kpl<NKC, 8, false, true>(p, a, warps, stream);
    }
    if (a.coset) {
        if (a.k <= 32) return launch_kpl<NKC, 1, true>(p, a, warps, stream);
        if (a.k <= 64) return launch_kpl<NKC, 2, true>(p, a, warps, stream);
        if (a.k <= 128) return launch_kpl<NKC, 4, true>(p, a, warps, stream);
        return launch_kpl<NKC, 8, true>(p, a, warps, stream);
    }
    if (a.k <= 32) return launch_kpl<NKC, 1, false>(p, a, warps, stream);
    if (a.k <= 64) return launch_kpl<NKC, 2, false>(p, a, warps, stream);
    if (a.k <= 128) return launch_kpl<NKC, 4, false>(p, a, warps, stream);
    return launch_kpl<NKC, 8, false>(p, a, warps, stream);
}

// One per table count, each in its own translation unit.
cudaError_t launch_nkc2(const dpb_plan *p, const Args &a, int warps, cudaStream_t stream);
cudaError_t launch_nkc3(const dpb_plan *p, const Args &a, int warps, cudaStream_t stream);
cudaError_t launch_nkc4(const dpb_plan *p, const Args &a, int warps, cudaStream_t stream);

}  // namespace mmaenc
}  // namespace dpb
