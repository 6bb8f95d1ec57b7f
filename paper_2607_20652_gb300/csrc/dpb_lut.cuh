// dpb_lut.cuh -- table-driven sums of generated parity signs (one warp per
// token, lane l owning coordinates iota = 32 q + l).
//
// The decoder's sum r[iota] = sum_e a_e (-1)^{parity(M[iota] AND c_e)}
// (§2.1 with App. A.4 Eq. 26) is evaluated 64 codes at a time (a "sweep"):
//
//  1. Signs, bit-sliced over codes. Z(iota) is a 64-bit word whose bit e is
//     the sign bit of code e at coordinate iota. The sign is linear in the
//     bits of M[iota] = iota | inv(iota) << t (App. A.4 Eq. 22), so
//       Z(iota) = ZL(iota & 31) ^ ZQ(iota >> 5) ^ XOR_k ZH_k(chunk_k(inv iota)),
//     each term the XOR of the ballots C_b = {bit b of c_e}_e over the set
//     bits of its argument: ZL is a register per lane, ZQ one word per block,
//     ZH_k 32-entry tables indexed by 5-bit chunks of inv(iota).
//  2. Sums, four Russians style. Each run of 5 codes has a 32-entry table of
//     all its signed sums sum_j (-1)^{v_j} a_j; the run's 5 sign bits in
//     Z(iota) index it, so one lookup and one add replace 5 sign-adds. Even
//     runs are held one entry per lane and read with a shuffle (which uses
//     only the low 5 bits of its index); odd runs live in shared memory (a
//     32-word table spans all banks: every lookup is conflict-free). The two
//     kinds of lookup go down different pipes. The odd tables are 128-byte
//     aligned, so a lookup's address is the table's address OR the run's 5
//     bits times 4, one logic instruction.
#pragma once

#include <cstdint>

#include "dpb_device.cuh"

namespace dpb {

constexpr int kMaxKChunks = 4;   // ceil(16 / 5) chunks of inv(iota) for t <= 16
constexpr int kMaxRuns = 13;     // ceil(64 / 5) runs of 5 codes per sweep
constexpr int kShflRuns = 7;     // even runs 0, 2, ..., 12

constexpr int kMaxBlocks = 64;   // 32-coordinate blocks of d <= 2048

// Shared-memory words of one sweep's tables for qn 32-coordinate blocks and
// nkc chunk tables of inv(iota): ZQ (a uint2 per block, padded to 128
// bytes), ZH (nkc tables of 2 x 32 words), the odd runs' value tables (6 x 32
// words, 128-byte aligned) and the coefficients (64). A multiple of 32 words.
__host__ __device__ constexpr int sweep_words(int qn, int nkc) {
    return ((2 * qn + 31) & ~31) + 64 * nkc + 32 * (kMaxRuns - kShflRuns) + 64;
}

struct Sweep {
    uint2 zl;                 // ZL(lane) for codes 0..31 (x) and 32..63 (y)
    float vt[kShflRuns];      // lane v holds the table of run 2i at v
    uint2 *zq;                // [qn] (shared)
    uint32_t *zh;             // [nkc][2][32]: codes 0..31, then 32..63 (shared)
    float *vto;               // [6][32] odd runs (shared)
    float *coef;              // [64] (shared)
    uint32_t vto_s;           // shared-window address of vto (128-byte aligned)
    int runs;                 // ceil(codes / 5)
    int nkc;                  // chunk tables of inv(iota) held
};

// Shared-window (32-bit) address of a pointer into this block's shared memory.
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// fp32 load from shared memory at byte address addr + OFF (a 32-bit
// shared-window address the caller composed by OR or byte permute, with the
// offset as an immediate). Every table read this way was written before a
// __syncwarp() of the same warp; the asm is volatile, so the compiler keeps it
// after that barrier.
template <int OFF>
__device__ __forceinline__ float lds_f32(uint32_t addr) {
    float v;
    asm volatile("ld.shared.f32 %0, [%1+%2];" : "=f"(v) : "r"(addr), "n"(OFF));
    return v;
}

// The first A-byte aligned word of a dynamic shared-memory buffer (the
// launch allocates A bytes more than the layout needs).
template <int A>
__device__ __forceinline__ uint32_t *aligned_smem(uint32_t *raw) {
    return raw + ((A - (smem_u32(raw) & (A - 1))) & (A - 1)) / 4;
}

// A sweep's tables at base (sweep_words(qn, nkc) words), which must be
// 128-byte aligned (the odd value tables are addressed by OR).
__device__ __forceinline__ Sweep sweep_at(uint32_t *base, int qn, int nkc) {
    Sweep s;
    s.zq = reinterpret_cast<uint2 *>(base);
    s.zh = base + ((2 * qn + 31) & ~31);
    s.vto = reinterpret_cast<float *>(s.zh + 64 * nkc);
    s.coef = s.vto + 32 * (kMaxRuns - kShflRuns);
    s.vto_s = smem_u32(s.vto);
    s.nkc = nkc;
    return s;
}

// Byte offsets (x4, for 32-bit tables) of the 5-bit chunks of kappa = inv(iota).
__device__ __forceinline__ uint32_t kappa_offsets4(uint32_t kappa) {
    uint32_t off = 0;
#pragma unroll
    for (int k = 0; k < kMaxKChunks; ++k) off |= (((kappa >> (5 * k)) & 31u) * 4u) << (8 * k);
    return off;
}

// Sign tables of a sweep from its codes (lane holds codes lane and 32 + lane;
// 0 for empty slots). qn = number of 32-coordinate blocks (<= kMaxBlocks).
__device__ __forceinline__ void sweep_build_signs(uint32_t ca, uint32_t cb, int t, int qn, Sweep &s) {
    const int lane = threadIdx.x & 31;
    uint2 zl = make_uint2(0u, 0u);
#pragma unroll
    for (int b = 0; b < 5; ++b) {
        const uint32_t xa = __ballot_sync(kFull, (ca >> b) & 1u), xb = __ballot_sync(kFull, (cb >> b) & 1u);
        if ((lane >> b) & 1) {
            zl.x ^= xa;
            zl.y ^= xb;
        }
    }
    s.zl = zl;
    uint32_t qa[6], qb[6];  // iota bits 5..10 are the bits of the block index q
#pragma unroll
    for (int b = 0; b < 6; ++b) {
        const bool live = 5 + b < t;
        qa[b] = live ? __ballot_sync(kFull, (ca >> (5 + b)) & 1u) : 0u;
        qb[b] = live ? __ballot_sync(kFull, (cb >> (5 + b)) & 1u) : 0u;
    }
    for (int q = lane; q < qn; q += 32) {
        uint2 z = make_uint2(0u, 0u);
#pragma unroll
        for (int b = 0; b < 6; ++b)
            if ((q >> b) & 1) {
                z.x ^= qa[b];
                z.y ^= qb[b];
            }
        s.zq[q] = z;
    }
#pragma unroll
    for (int k = 0; k < kMaxKChunks; ++k) {
        if (k >= s.nkc) break;  // chunks past the held ones are zero (t <= 5 nkc)
        uint2 acc = make_uint2(0u, 0u);
#pragma unroll
        for (int bb = 0; bb < 5; ++bb) {
            const int b = t + 5 * k + bb;
            const bool live = b < 2 * t && b < 32;
            const uint32_t xa = live ? __ballot_sync(kFull, (ca >> b) & 1u) : 0u;
            const uint32_t xb = live ? __ballot_sync(kFull, (cb >> b) & 1u) : 0u;
            if ((lane >> bb) & 1) {
                acc.x ^= xa;
                acc.y ^= xb;
            }
        }
        s.zh[k * 64 + lane] = acc.x;
        s.zh[k * 64 + 32 + lane] = acc.y;
    }
}

// Value tables of a sweep from its 64 coefficients (already in s.coef, zero
// beyond the sweep's codes).
__device__ __forceinline__ void sweep_build_values(Sweep &s) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int g = 0; g < kMaxRuns; ++g) {
        float v = 0.f;
        if (g < s.runs) {
#pragma unroll
            for (int j = 0; j < 5; ++j) {
                const int e = 5 * g + j;
                const float a = e < 64 ? s.coef[e] : 0.f;
                v += ((lane >> j) & 1) ? -a : a;
            }
        }
        if (g % 2 == 0)
            s.vt[g / 2] = v;
        else
            s.vto[(g / 2) * 32 + lane] = v;
    }
}

// Z(iota) of a sweep; koff = kappa_offsets4(inv iota), zq = ZQ(iota >> 5).
// Each half of a ZH entry is its own 32-word table, so that a lookup of
// random entries by the 32 lanes is free of bank conflicts.
template <int NKC>
__device__ __forceinline__ uint2 sweep_signs(const Sweep &s, uint2 zq, uint32_t koff) {
    const char *zh = reinterpret_cast<const char *>(s.zh);
    uint2 z = make_uint2(s.zl.x ^ zq.x, s.zl.y ^ zq.y);
#pragma unroll
    for (int k = 0; k < NKC; ++k) {
        const uint32_t o = __byte_perm(koff, 0, 0x4440 + k);
        z.x ^= *reinterpret_cast<const uint32_t *>(zh + k * 256 + o);
        z.y ^= *reinterpret_cast<const uint32_t *>(zh + k * 256 + 128 + o);
    }
    return z;
}

// Bits 5G..5G+4 of the 64-bit z in the low bits (high bits unspecified).
template <int G>
__device__ __forceinline__ uint32_t run_field(uint2 z) {
    constexpr int lo = 5 * G;
    if constexpr (lo + 5 <= 32) {
        return z.x >> lo;
    } else if constexpr (lo >= 32) {
        return z.y >> (lo - 32);
    } else {
        return __funnelshift_r(z.x, z.y, lo);
    }
}

// The same field times 4 (a byte offset into a 32-float table), G >= 1.
template <int G>
__device__ __forceinline__ uint32_t run_offset(uint2 z) {
    constexpr int lo = 5 * G - 2;
    uint32_t v;
    if constexpr (lo + 7 <= 32) {
        v = z.x >> lo;
    } else if constexpr (lo >= 32) {
        v = z.y >> (lo - 32);
    } else {
        v = __funnelshift_r(z.x, z.y, lo);
    }
    return v & 0x7Cu;
}

template <int G, int RUNS>
__device__ __forceinline__ void run_lookups(const Sweep &s, uint2 z, float *p) {
    if constexpr (G < RUNS) {
        if constexpr (G % 2 == 0) {
            p[G] = __shfl_sync(kFull, s.vt[G / 2], run_field<G>(z));
        } else {
            p[G] = lds_f32<(G / 2) * 128>(s.vto_s | run_offset<G>(z));
        }
        run_lookups<G + 1, RUNS>(s, z, p);
    }
}

// Sum of n floats: pairs added two at a time (packed fp32x2 adds), then the
// two halves and an odd last one.
template <int N>
__device__ __forceinline__ float sum_packed(const float *p) {
    if constexpr (N == 1) {
        return p[0];
    } else {
        constexpr int NP = N / 2;
        float2 q[NP];
#pragma unroll
        for (int i = 0; i < NP; ++i) q[i] = make_float2(p[2 * i], p[2 * i + 1]);
#pragma unroll
        for (int w = 1; w < NP; w *= 2)
#pragma unroll
            for (int g = 0; g + w < NP; g += 2 * w) q[g] = __fadd2_rn(q[g], q[g + w]);
        const float h = q[0].x + q[0].y;
        if constexpr (N % 2 == 1) return h + p[N - 1];
        return h;
    }
}

// sum_e coef_e (-1)^{bit e of z} over the sweep's RUNS runs of 5 codes.
template <int RUNS>
__device__ __forceinline__ float sweep_sum(const Sweep &s, uint2 z) {
    float p[RUNS];
    run_lookups<0, RUNS>(s, z, p);
    return sum_packed<RUNS>(p);
}

// Sizes rounded up to 4 words, so that every per-warp array of the kernels'
// shared-memory layouts starts 16-byte aligned.
__host__ __device__ constexpr int pad4(int v) { return (v + 3) & ~3; }
// Sizes rounded up to 32 words (128 bytes) and 64 words (256 bytes).
__host__ __device__ constexpr int pad32(int v) { return (v + 31) & ~31; }
__host__ __device__ constexpr int pad64(int v) { return (v + 63) & ~63; }
static_assert(sweep_words(24, 2) % 32 == 0 && sweep_words(64, 4) % 32 == 0,
              "a sweep's tables keep the 128-byte alignment of what follows");

// ---- a token's code -----------------------------------------------------------

// Compact list of a token's hashed entries (index >= d).
struct HashedList {
    uint32_t *c;    // [k] indices
    float *a;       // [k] coefficients
    int *pos;       // [k] position in the code (nullable)
};

// Adds the basis entries of a token's code (index < d) into `basis` (at
// their coordinate) and compacts the hashed entries into `hl`; entries
// outside [0, m_mask] are skipped and flagged. Returns the hashed count.
__device__ __forceinline__ int split_code(const int32_t *idx, const float *val, int k, int d,
                                          uint32_t m_mask, float *basis, HashedList &hl,
                                          int32_t *status) {
    const int lane = threadIdx.x & 31;
    int nh = 0;
    for (int e0 = 0; e0 < k; e0 += 32) {
        const int e = e0 + lane;
        int32_t ci = -1;
        float a = 0.f;
        if (e < k) {
            ci = idx[e];
            a = val[e];
        }
        const bool valid = e < k && ci >= 0 && (uint32_t)ci <= m_mask;
        if (e < k && !valid) set_status(status, DPB_DEV_BAD_INDEX);
        const bool hashed = valid && ci >= d;
        if (valid && !hashed && basis) atomicAdd(&basis[ci], a);
        const unsigned m = __ballot_sync(kFull, hashed);
        if (hashed) {
            const int pos = nh + __popc(m & ((1u << lane) - 1u));
            hl.c[pos] = (uint32_t)ci;
            hl.a[pos] = a;
            if (hl.pos) hl.pos[pos] = e;
        }
        nh += __popc(m);
    }
    __syncwarp();
    return nh;
}

// ---- synthesis over a hashed list ---------------------------------------------

// out[i] += scale * sum over one sweep, for every coordinate of the token.
// UNROLL coordinates blocks per loop trip.
template <int NKC, int RUNS, int UNROLL>
__device__ __forceinline__ void sweep_accumulate(const Sweep &s, float *out, const uint32_t *koff, int d,
                                                 float scale) {
    const int lane = threadIdx.x & 31;
    const int qn = (d + 31) / 32;
#pragma unroll UNROLL
    for (int q = 0; q < qn; ++q) {
        const int i = 32 * q + lane;
        const bool in = i < d;
        const uint2 z = sweep_signs<NKC>(s, s.zq[q], in ? koff[i] : 0u);
        const float v = sweep_sum<RUNS>(s, z);
        if (in) out[i] += scale * v;
    }
}

// Code shape of a sweep. kSweepWide rounds the runs up to one of five
// unrolled widths (the extra runs read all-zero tables) and does two blocks
// per trip: the fewest instructions. kSweepCompact does one block per trip
// and rounds the runs up to 8, 10 or 13 only: less code, for kernels whose
// other phases already fill the instruction caches.
enum SweepShape { kSweepWide, kSweepCompact };

template <int NKC, SweepShape SHAPE>
__device__ __forceinline__ void sweep_accumulate_runs(const Sweep &s, float *out, const uint32_t *koff,
                                                      int d, float scale) {
    if constexpr (SHAPE == kSweepCompact) {
        if (s.runs <= 8)
            sweep_accumulate<NKC, 8, 1>(s, out, koff, d, scale);
        else if (s.runs <= 10)
            sweep_accumulate<NKC, 10, 1>(s, out, koff, d, scale);
        else
            sweep_accumulate<NKC, kMaxRuns, 1>(s, out, koff, d, scale);
    } else if (s.runs <= 4) {
        sweep_accumulate<NKC, 4, 2>(s, out, koff, d, scale);
    } else if (s.runs <= 6) {
        sweep_accumulate<NKC, 6, 2>(s, out, koff, d, scale);
    } else if (s.runs <= 8) {
        sweep_accumulate<NKC, 8, 2>(s, out, koff, d, scale);
    } else if (s.runs <= 10) {
        sweep_accumulate<NKC, 10, 2>(s, out, koff, d, scale);
    } else {
        sweep_accumulate<NKC, kMaxRuns, 2>(s, out, koff, d, scale);
    }
}

// out[i] += scale * sum_e coef_e (-1)^{parity(M[i] AND c_e)} over n codes
// (indices c, coefficients coef), 64 codes per sweep. koff[i] holds the
// packed chunk offsets of inv(i) (kappa_offsets4).
template <int NKC, SweepShape SHAPE = kSweepWide>
__device__ __forceinline__ void synthesise(Sweep &s, const uint32_t *c, const float *coef, int n, int t, int d,
                                           const uint32_t *koff, float scale, float *out) {
    const int lane = threadIdx.x & 31;
    const int qn = (d + 31) / 32;
    for (int g0 = 0; g0 < n; g0 += 64) {
        const int m = min(64, n - g0);
        const uint32_t ca = lane < m ? c[g0 + lane] : 0u;
        const uint32_t cb = lane + 32 < m ? c[g0 + 32 + lane] : 0u;
        s.coef[lane] = lane < m ? coef[g0 + lane] : 0.f;
        s.coef[32 + lane] = lane + 32 < m ? coef[g0 + 32 + lane] : 0.f;
        sweep_build_signs(ca, cb, t, qn, s);
        s.runs = (m + 4) / 5;
        __syncwarp();
        sweep_build_values(s);
        __syncwarp();
        sweep_accumulate_runs<NKC, SHAPE>(s, out, koff, d, scale);
        __syncwarp();
    }
}

// Packed chunk offsets of inv(i) = M[i] >> t for the block's coordinates.
__device__ __forceinline__ void load_koff(const uint32_t *M, int d, int t, uint32_t *koff) {
    for (int i = threadIdx.x; i < d; i += blockDim.x) koff[i] = kappa_offsets4(M[i] >> t);
    __syncthreads();
}

// ---- per-code sign words of a 32-coordinate block (backward, moments) --------------

// Per-code parts of the sign words (bit l of block q = parity(M[32q + l] AND
// c), App. A.4 Eq. 26): o1 = W5[c & 31], the Walsh part; o2 = u | h0 << 11 |
// h1 << 16 | h2 << 21 | h3 << 26 with u = c_lo >> 5 (the block-parity mask)
// and h_k the 5-bit chunks of the high half.
__device__ __forceinline__ void code_offsets(uint32_t c, int t, const uint32_t *w5, uint32_t &o1, uint32_t &o2) {
    const uint32_t u = (c & ((1u << t) - 1u)) >> 5;
    uint32_t h = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) h |= ((c >> min(t + 5 * k, 31)) & 31u) << (5 * k);
    o1 = w5[c & 31u];
    o2 = u | (h << 11);
}

// Sign word of code (o1, o2) over block q (VH2 holds NKC chunk tables of
// nblk blocks x 32 words).
template <int NKC>
__device__ __forceinline__ uint32_t block_signs(const uint32_t *vh2, int nblk, int q, uint32_t o1, uint32_t o2) {
    const uint32_t *V = vh2 + q * 32;
    uint32_t s = o1 ^ (0u - (uint32_t)(__popc((uint32_t)q & (o2 & 0x7FFu)) & 1));
    s ^= V[(o2 >> 11) & 31u];
    s ^= V[nblk * 32 + ((o2 >> 16) & 31u)];
    if (NKC > 2) s ^= V[2 * nblk * 32 + ((o2 >> 21) & 31u)];
    if (NKC > 3) s ^= V[3 * nblk * 32 + ((o2 >> 26) & 31u)];
    return s;
}

}  // namespace dpb
