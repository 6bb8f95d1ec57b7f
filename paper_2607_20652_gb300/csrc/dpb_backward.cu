// dpb_backward.cu -- gradients of decode(encode(x)) with the selected set held
// fixed (the paper trains through the layer end to end but does not write the
// backward out; it is derived by the chain rule), one warp per token.
//
// With g = dL/dy, r = sum_e val_e phi_e, c = |x| / |r| and norm matching:
//   dL/dr      = c (g - (<g,r> / |r|^2) r)          (g without norm matching)
//   grad_val_e = <phi_e, dL/dr>
//   grad_x     = sum_e (grad_val_e / sigma_e) phi_e + (<g,r>/|r|) x / |x|.
// The table-driven kernel (d <= 2048) evaluates the two sums over phi with the
// sweeps of dpb_lut.cuh and the inner products <phi_e, dL/dr> with per-token
// tables of signed sums of dL/dr over 4 coordinates (see analyse()).
#include <algorithm>
#include <climits>
#include <cstdint>
#include <initializer_list>

#include "dpb_device.cuh"
#include "dpb_internal.h"
#include "dpb_lut.cuh"

namespace dpb {

namespace {

struct BackwardArgs {
    const void *x, *gy;
    const int32_t *idx;
    const float *val, *sigma;
    const float *R;  // nullable: r of the decode, fp32 [T][d], instead of rebuilding it
    void *gx;
    float *gval;
    int64_t T;
    int32_t *status;
    const uint32_t *M, *VH;
    int d, k, norm_match;
    uint32_t m_mask;
    float inv_sqrt_d;
};

// r (basis part rb, hashed +-sum rh) of one token into shared memory; lane l
// owns coordinates l, l+32, ... so no two lanes touch the same word.
__device__ void reconstruct(const int32_t *idx, const float *val, int k, int d, uint32_t m_mask,
                            const uint32_t *sM, float *rb, float *rh, int32_t *status) {
    const int lane = threadIdx.x & 31;
    for (int i = lane; i < d; i += 32) {
        rb[i] = 0.f;
        rh[i] = 0.f;
    }
    for (int e = 0; e < k; ++e) {
        const int32_t ci = idx[e];
        const float a = val[e];
        if (ci < 0 || (uint32_t)ci > m_mask) {
            if (lane == 0) set_status(status, DPB_DEV_BAD_INDEX);
            continue;
        }
        const uint32_t c = (uint32_t)ci;
        if (c < (uint32_t)d) {
            if ((int)(c & 31) == lane) rb[c] += a;
        } else {
            for (int i = lane; i < d; i += 32) rh[i] += flip(a, sign31(sM[i], c));
        }
    }
}

template <typename Tio>
__global__ void __launch_bounds__(128) backward_warp_kernel(BackwardArgs a) {
    extern __shared__ __align__(16) uint32_t smem[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    const int d = a.d;
    uint32_t *sM = smem;
    for (int i = threadIdx.x; i < d; i += blockDim.x) sM[i] = a.M[i];
    __syncthreads();
    float *rb = reinterpret_cast<float *>(sM + d) + (size_t)warp * 4 * d;
    float *rh = rb + d;    // hashed sum, then reused as dL/dr
    float *xs = rh + d;
    float *gx = xs + d;
    const Tio *X = static_cast<const Tio *>(a.x);
    const Tio *GY = static_cast<const Tio *>(a.gy);
    Tio *GX = static_cast<Tio *>(a.gx);
    for (int64_t t = (int64_t)blockIdx.x * nwarps + warp; t < a.T; t += (int64_t)gridDim.x * nwarps) {
        const int32_t *it = a.idx + t * a.k;
        const float *vt = a.val + t * a.k;
        float sxx = 0.f;
        for (int i = lane; i < d; i += 32) {
            const float v = ld_elem(X, t * d + i);
            xs[i] = v;
            sxx += v * v;
        }
        const float nx = sqrtf(warp_sum(sxx));
        float direct = 0.f;  // coefficient of x/|x| in grad_x
        if (a.norm_match) {
            if (!a.R) reconstruct(it, vt, a.k, d, a.m_mask, sM, rb, rh, a.status);
            __syncwarp();
            float srr = 0.f, sgr = 0.f;
            for (int i = lane; i < d; i += 32) {
                const float r = a.R ? a.R[t * d + i] : rb[i] + rh[i] * a.inv_sqrt_d;
                rb[i] = r;
                srr += r * r;
                sgr += ld_elem(GY, t * d + i) * r;
            }
            srr = warp_sum(srr);
            sgr = warp_sum(sgr);
            const float nr = sqrtf(srr);
            if (nr > 0.f) {
                const float c = nx / nr, beta = sgr / srr;
                for (int i = lane; i < d; i += 32) rh[i] = c * (ld_elem(GY, t * d + i) - beta * rb[i]);
                direct = nx > 0.f ? sgr / nr : 0.f;
            } else {
                for (int i = lane; i < d; i += 32) rh[i] = 0.f;
            }
        } else {
            for (int i = lane; i < d; i += 32) rh[i] = ld_elem(GY, t * d + i);
        }
        const float dx = nx > 0.f ? direct / nx : 0.f;
        for (int i = lane; i < d; i += 32) gx[i] = dx * xs[i];
        __syncwarp();
        // grad_val_e = <phi_e, dL/dr>; grad_x += (grad_val_e / sigma_e) phi_e
        for (int e = 0; e < a.k; ++e) {
            const int32_t ci = it[e];
            if (ci < 0 || (uint32_t)ci > a.m_mask) {
                if (lane == 0) {
                    set_status(a.status, DPB_DEV_BAD_INDEX);
                    a.gval[t * a.k + e] = 0.f;
                }
                continue;
            }
            const uint32_t c = (uint32_t)ci;
            float sd = 1.f;
            if (a.sigma) {
                sd = a.sigma[c];
                if (!(sd > 0.f) && lane == 0) set_status(a.status, DPB_DEV_BAD_SIGMA);
            }
            if (c < (uint32_t)d) {
                const float gv = rh[c];
                if (lane == 0) a.gval[t * a.k + e] = gv;
                if ((int)(c & 31) == lane) gx[c] += gv / sd;
            } else {
                float acc = 0.f;
                for (int i = lane; i < d; i += 32) acc += flip(rh[i], sign31(sM[i], c));
                const float gv = warp_sum(acc) * a.inv_sqrt_d;
                if (lane == 0) a.gval[t * a.k + e] = gv;
                const float w = (gv / sd) * a.inv_sqrt_d;
                for (int i = lane; i < d; i += 32) gx[i] += flip(w, sign31(sM[i], c));
            }
            __syncwarp();
        }
        for (int i = lane; i < d; i += 32) st_elem(GX, t * d + i, gx[i]);
        __syncwarp();
    }
}


// ---- table-driven backward (d <= 2048) ---------------------------------------

constexpr int kChunkBlocks = 4;                       // 32-coordinate blocks per analysis chunk
constexpr int kTabStride = 17;                        // 16 entries + 1 pad (bank spread)
constexpr int kChunkTables = kChunkBlocks * 8 * kTabStride;  // nibble tables of a chunk (words)
__host__ __device__ constexpr int bwd_scratch_words(int qn, int nkc) {
    return pad64(sweep_words(qn, nkc) > kChunkTables ? sweep_words(qn, nkc) : kChunkTables);
}
constexpr int kBwdWarps = 15;  // at most per block; two blocks of 15 per SM at d = 768
static_assert(kChunkBlocks == 4, "the analysis gives a code 4 lanes, one per block of a chunk");

// Per-warp words: the scratch (a sweep's tables, or a chunk's nibble tables;
// first, so that it keeps the region's 256-byte alignment), then r / dL/dr /
// grad_x (d) and the code's lists (list, map, sums, offsets).
__host__ __device__ constexpr int bwd_warp_words(int d, int k, int nkc) {
    return pad64(bwd_scratch_words((d + 31) / 32, nkc) + pad4(d) + 6 * pad4(k));
}

__host__ __device__ constexpr int bwd_block_words(int d, int nkc) {
    return pad64(pad4(d) /* koff */ + 32 /* W5 */ + nkc * ((d + 31) / 32) * 32 /* VH2 */);
}

struct BwdWarp {
    float *buf;     // [d] r, then dL/dr, then grad_x
    uint32_t *hc;   // [k] hashed indices
    float *ha;      // [k] hashed coefficients, later grad_val / sigma
    int *cmap;      // [k] code entry -> hashed position (>= 0) or -(c+1) (basis) or INT_MIN
    float *gv;      // [k] analysis sums per hashed position
    uint32_t *o1;   // [k] the Walsh word W5[c & 31] of each hashed code
    uint32_t *o2;   // [k] its block-parity index and high-half chunks; later basis grad_x terms
    uint32_t *scratch;
};

// The 4 nibble offsets (times 4, one per byte) of the even (ev) and odd (od)
// nibbles of a sign word: nibble n of s indexes table n of its block.
__device__ __forceinline__ void nibble_offsets(uint32_t s, uint32_t &ev, uint32_t &od) {
    ev = (s << 2) & 0x3C3C3C3Cu;  // nibbles 0, 2, 4, 6
    od = (s >> 2) & 0x3C3C3C3Cu;  // nibbles 1, 3, 5, 7
}

// The 8 table entries of one (code, block) term as a pair of partial sums.
// A table's address is its block's base with the entry offset in the low
// byte: base_s must be 256-byte aligned, the table offsets OFF + n 68 come
// as immediates.
template <int OFF>
__device__ __forceinline__ float2 nibble_sum(uint32_t base_s, uint32_t s) {
    constexpr int S4 = 4 * kTabStride;  // bytes per table
    uint32_t ev, od;
    nibble_offsets(s, ev, od);
    const float p0 = lds_f32<OFF + 0 * S4>(__byte_perm(ev, base_s, 0x7650));
    const float p1 = lds_f32<OFF + 1 * S4>(__byte_perm(od, base_s, 0x7650));
    const float p2 = lds_f32<OFF + 2 * S4>(__byte_perm(ev, base_s, 0x7651));
    const float p3 = lds_f32<OFF + 3 * S4>(__byte_perm(od, base_s, 0x7651));
    const float p4 = lds_f32<OFF + 4 * S4>(__byte_perm(ev, base_s, 0x7652));
    const float p5 = lds_f32<OFF + 5 * S4>(__byte_perm(od, base_s, 0x7652));
    const float p6 = lds_f32<OFF + 6 * S4>(__byte_perm(ev, base_s, 0x7653));
    const float p7 = lds_f32<OFF + 7 * S4>(__byte_perm(od, base_s, 0x7653));
    return __fadd2_rn(__fadd2_rn(make_float2(p0, p1), make_float2(p2, p3)),
                      __fadd2_rn(make_float2(p4, p5), make_float2(p6, p7)));
}

// The same with the block's base in a register (any 4-byte alignment).
__device__ __forceinline__ float nibble_sum_at(uint32_t blk_s, uint32_t s) {
    constexpr int S4 = 4 * kTabStride;
    uint32_t ev, od;
    nibble_offsets(s, ev, od);
    const float p0 = lds_f32<0 * S4>(blk_s + __byte_perm(ev, 0, 0x4440));
    const float p1 = lds_f32<1 * S4>(blk_s + __byte_perm(od, 0, 0x4440));
    const float p2 = lds_f32<2 * S4>(blk_s + __byte_perm(ev, 0, 0x4441));
    const float p3 = lds_f32<3 * S4>(blk_s + __byte_perm(od, 0, 0x4441));
    const float p4 = lds_f32<4 * S4>(blk_s + __byte_perm(ev, 0, 0x4442));
    const float p5 = lds_f32<5 * S4>(blk_s + __byte_perm(od, 0, 0x4442));
    const float p6 = lds_f32<6 * S4>(blk_s + __byte_perm(ev, 0, 0x4443));
    const float p7 = lds_f32<7 * S4>(blk_s + __byte_perm(od, 0, 0x4443));
    const float2 r = __fadd2_rn(__fadd2_rn(make_float2(p0, p1), make_float2(p2, p3)),
                                __fadd2_rn(make_float2(p4, p5), make_float2(p6, p7)));
    return r.x + r.y;
}

// Block QQ of the chunk at q0 (if the chunk has it) added into a code's sums.
template <int NKC, int QQ>
__device__ __forceinline__ void add_block(float2 &acc, const uint32_t *vh2, int qn, int q0, int cq, uint32_t o1,
                                          uint32_t o2, uint32_t th_s) {
    if (QQ < cq)
        acc = __fadd2_rn(acc, nibble_sum<QQ * 8 * kTabStride * 4>(th_s, block_signs<NKC>(vh2, qn, q0 + QQ, o1, o2)));
}

// gv[p] += sum_i h[i] (-1)^{parity(M[i] AND hc_p)} for the nh hashed codes.
// Per chunk of 4 blocks: nibble tables TH[b][n][v] = sum_j (-1)^{v_j}
// h[32b + 4n + j] (16 entries per 4 coordinates); a code's sign word over a
// block indexes that block's 8 tables. The first nh - nh % 32 codes go one
// per lane through all blocks of the chunk; each of the others gets 4 lanes,
// one block each, summed by shuffles. Every code's sum is taken in a fixed
// order.
template <int NKC>
__device__ __forceinline__ void analyse(const BwdWarp &w, int nh, int d, const uint32_t *vh2) {
    const int lane = threadIdx.x & 31;
    const int qn = (d + 31) / 32;
    const int full = nh & ~31, tail = nh - full;
    float *TH = reinterpret_cast<float *>(w.scratch);
    const uint32_t th_s = smem_u32(TH);  // 256-byte aligned
    for (int q0 = 0; q0 < qn; q0 += kChunkBlocks) {
        const int cq = min(kChunkBlocks, qn - q0);
        // both loops stay rolled: this kernel's hot code is at the instruction caches' size
#pragma unroll 1
        for (int tau = lane; tau < cq * 8; tau += 32) {
            const int i0 = 32 * (q0 + tau / 8) + 4 * (tau % 8);  // = 4 (8 q0 + tau)
            float4 hv = make_float4(0.f, 0.f, 0.f, 0.f);
            if (i0 + 3 < d) {
                hv = *reinterpret_cast<const float4 *>(w.buf + i0);
            } else {
                if (i0 < d) hv.x = w.buf[i0];
                if (i0 + 1 < d) hv.y = w.buf[i0 + 1];
                if (i0 + 2 < d) hv.z = w.buf[i0 + 2];
            }
            // entry v = (v3 v2 v1 v0): sum_j (-1)^{v_j} h_j = A[v1 v0] + B[v3 v2]
            const float a0 = hv.x + hv.y, a1 = hv.x - hv.y;
            const float b0 = hv.z + hv.w, b1 = hv.z - hv.w;
            float *T = TH + tau * kTabStride;
            // v0 = 1 negates h0: A[01] = -h0 + h1 = -a1, A[10] = h0 - h1 = a1
            const float A[4] = {a0, -a1, a1, -a0};
            const float B[4] = {b0, -b1, b1, -b0};
#pragma unroll
            for (int v = 0; v < 16; ++v) T[v] = A[v & 3] + B[v >> 2];
        }
        __syncwarp();
#pragma unroll 1
        for (int e = lane; e < full; e += 32) {  // full is a multiple of 32: no lane drops out
            const uint32_t o1 = w.o1[e], o2 = w.o2[e];
            float2 acc = make_float2(0.f, 0.f);
            add_block<NKC, 0>(acc, vh2, qn, q0, cq, o1, o2, th_s);
            add_block<NKC, 1>(acc, vh2, qn, q0, cq, o1, o2, th_s);
            add_block<NKC, 2>(acc, vh2, qn, q0, cq, o1, o2, th_s);
            add_block<NKC, 3>(acc, vh2, qn, q0, cq, o1, o2, th_s);
            w.gv[e] += acc.x + acc.y;  // this lane's own code
        }
#pragma unroll 1
        for (int it0 = 0; it0 < 4 * tail; it0 += 32) {
            const int it = it0 + lane, e = full + (it >> 2), qq = it & 3;
            float v = 0.f;
            if (it < 4 * tail && qq < cq)
                v = nibble_sum_at(th_s + qq * (8 * kTabStride * 4),
                                  block_signs<NKC>(vh2, qn, q0 + qq, w.o1[e], w.o2[e]));
            v += __shfl_xor_sync(kFull, v, 1);
            v += __shfl_xor_sync(kFull, v, 2);
            if (it < 4 * tail && qq == 0) w.gv[e] += v;  // the code's 4 lanes are lanes 4j .. 4j+3
        }
        __syncwarp();
    }
}

// KEPT: norm matching with the decode's r given (a separate instantiation,
// without the path that rebuilds r).
template <typename Tio, int NKC, bool VEC, bool KEPT>
__global__ void __launch_bounds__(kBwdWarps * 32, 2) backward_lut_kernel(BackwardArgs a, int t) {
    extern __shared__ __align__(16) uint32_t smem_raw[];
    uint32_t *smem = aligned_smem<256>(smem_raw);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    const int d = a.d, k = a.k;
    const int dp = pad4(d), kp = pad4(k);
    uint32_t *koff = smem;
    uint32_t *w5 = koff + dp;
    uint32_t *vh2 = w5 + 32;
    for (int v = threadIdx.x; v < 32; v += blockDim.x) {
        uint32_t word = 0;
        for (int l = 0; l < 32; ++l) word |= (uint32_t)(__popc(l & v) & 1) << l;
        w5[v] = word;
    }
    for (int i = threadIdx.x; i < NKC * ((d + 31) / 32) * 32; i += blockDim.x) vh2[i] = a.VH[i];
    load_koff(a.M, d, t, koff);  // ends with __syncthreads()

    uint32_t *base = smem + bwd_block_words(d, NKC) + (size_t)warp * bwd_warp_words(d, k, NKC);
    BwdWarp w;
    w.scratch = base;
    w.buf = reinterpret_cast<float *>(base + bwd_scratch_words((d + 31) / 32, NKC));
    w.hc = reinterpret_cast<uint32_t *>(w.buf + dp);
    w.ha = reinterpret_cast<float *>(w.hc + kp);
    w.cmap = reinterpret_cast<int *>(w.ha + kp);
    w.gv = reinterpret_cast<float *>(w.cmap + kp);
    w.o1 = reinterpret_cast<uint32_t *>(w.gv + kp);
    w.o2 = w.o1 + kp;
    float *bterm = reinterpret_cast<float *>(w.o2);  // basis grad_x terms, after the analysis
    Sweep sw = sweep_at(w.scratch, (d + 31) / 32, NKC);

    const Tio *X = static_cast<const Tio *>(a.x);
    const Tio *GY = static_cast<const Tio *>(a.gy);
    Tio *GX = static_cast<Tio *>(a.gx);
    for (int64_t tk = (int64_t)blockIdx.x * nwarps + warp; tk < a.T; tk += (int64_t)gridDim.x * nwarps) {
        const int32_t *it = a.idx + tk * k;
        const float *vt = a.val + tk * k;
        const Tio *xr = X + tk * d, *gr = GY + tk * d;
        // the code's first 64 entries, loaded ahead of the rows so that the
        // two loads overlap
        int32_t ci_pre[2] = {-1, -1};
        float v_pre[2] = {0.f, 0.f};
#pragma unroll
        for (int j = 0; j < 2; ++j)
            if (32 * j + lane < k) {
                ci_pre[j] = it[32 * j + lane];
                v_pre[j] = vt[32 * j + lane];
            }
        // With norm matching and the decode's r, dL/dr comes first, from one
        // sweep over x, grad_y and r; otherwise buf starts as the basis part
        // of r (rebuilt below) or as grad_y.
        constexpr bool kept_r = KEPT;  // the launcher's choice: a.norm_match && a.R
        float nx, direct = 0.f;  // direct: coefficient of x / |x| in grad_x
        if (kept_r) {
            float sxx = 0.f, srr = 0.f, sgr = 0.f;
            RowOps<VEC>::rows3(w.buf, xr, gr, a.R + tk * d, d, sxx, srr, sgr);
            nx = sqrtf(warp_sum(sxx));
            srr = warp_sum(srr);
            sgr = warp_sum(sgr);
            const float nr = sqrtf(srr);
            if (nr > 0.f) {
                RowOps<VEC>::project(w.buf, gr, d, nx / nr, sgr / srr);  // this lane's own coordinates
                direct = nx > 0.f ? sgr / nr : 0.f;
            } else {
                RowOps<VEC>::fill(w.buf, d, 0.f);
            }
        } else {
            RowOps<VEC>::fill(w.buf, d, 0.f);
        }
        __syncwarp();
        // ---- split the code: hashed entries listed (basis entries into buf when r is rebuilt) ----
        int nh = 0;
        for (int e0 = 0; e0 < k; e0 += 32) {
            const int e = e0 + lane;
            int32_t ci = -1;
            float v = 0.f;
            if (e0 < 64) {
                ci = ci_pre[e0 >> 5];
                v = v_pre[e0 >> 5];
            } else if (e < k) {
                ci = it[e];
                v = vt[e];
            }
            const bool valid = e < k && ci >= 0 && (uint32_t)ci <= a.m_mask;
            const bool hashed = valid && ci >= d;
            if (e < k && !valid) {
                set_status(a.status, DPB_DEV_BAD_INDEX);
                w.cmap[e] = INT_MIN;
            }
            if (valid && !hashed) {
                if (!kept_r && a.norm_match) atomicAdd(&w.buf[ci], v);
                w.cmap[e] = -(ci + 1);
            }
            const unsigned m = __ballot_sync(kFull, hashed);
            if (hashed) {
                const int pos = nh + __popc(m & ((1u << lane) - 1u));
                w.hc[pos] = (uint32_t)ci;
                w.ha[pos] = v;
                w.cmap[e] = pos;
                w.gv[pos] = 0.f;
                code_offsets((uint32_t)ci, t, w5, w.o1[pos], w.o2[pos]);
            }
            nh += __popc(m);
        }
        __syncwarp();
        if (!kept_r) nx = sqrtf(warp_sum(RowOps<VEC>::sumsq(xr, d)));
        if (!kept_r && !a.norm_match) {
            RowOps<VEC>::scale_in(w.buf, gr, d, 1.f);
            __syncwarp();
        }
        // Two synthesis passes share one call site: pass 0 builds r (norm
        // matching only) and turns it into dL/dr; pass 1 adds the hashed
        // entries' sum to grad_x.
#pragma unroll 1
        for (int pass = !kept_r && a.norm_match ? 0 : 1;; ++pass) {
            if (pass == 1) {
                // ---- grad_val = <phi_e, dL/dr> ----
                analyse<NKC>(w, nh, d, vh2);
                // ---- grad_val of every entry; the grad_x coefficients ----
                for (int e = lane; e < k; e += 32) {
                    const int cm = w.cmap[e];
                    float gvv = 0.f, term = 0.f;
                    if (cm >= 0) {
                        gvv = w.gv[cm] * a.inv_sqrt_d;
                        float sd = 1.f;
                        if (a.sigma) {
                            sd = a.sigma[w.hc[cm]];
                            if (!(sd > 0.f)) set_status(a.status, DPB_DEV_BAD_SIGMA);
                        }
                        w.ha[cm] = gvv / sd;
                    } else if (cm != INT_MIN) {
                        const int c = -cm - 1;
                        gvv = w.buf[c];
                        float sd = 1.f;
                        if (a.sigma) {
                            sd = a.sigma[c];
                            if (!(sd > 0.f)) set_status(a.status, DPB_DEV_BAD_SIGMA);
                        }
                        term = gvv / sd;
                    }
                    bterm[e] = term;
                    a.gval[tk * k + e] = gvv;
                }
                __syncwarp();
                // ---- grad_x: direct term and basis terms, then the hashed sum ----
                const float dx = nx > 0.f ? direct / nx : 0.f;
                RowOps<VEC>::scale_in(w.buf, xr, d, dx);
                __syncwarp();
                for (int e = lane; e < k; e += 32) {
                    const int cm = w.cmap[e];
                    if (cm < 0 && cm != INT_MIN) w.buf[-cm - 1] += bterm[e];  // indices are distinct
                }
                __syncwarp();
            }
            synthesise<NKC, kSweepCompact>(sw, w.hc, w.ha, nh, t, d, koff, a.inv_sqrt_d, w.buf);
            if (pass == 1) break;
            // ---- dL/dr = c (g - (<g,r>/|r|^2) r) in place of r ----
            float srr = 0.f, sgr = 0.f;
            RowOps<VEC>::dots(w.buf, gr, d, srr, sgr);
            srr = warp_sum(srr);
            sgr = warp_sum(sgr);
            const float nr = sqrtf(srr);
            if (nr > 0.f) {
                RowOps<VEC>::project(w.buf, gr, d, nx / nr, sgr / srr);
                direct = nx > 0.f ? sgr / nr : 0.f;
            } else {
                RowOps<VEC>::fill(w.buf, d, 0.f);
            }
            __syncwarp();
        }
        RowOps<VEC>::store(GX + tk * d, w.buf, d, 1.f);
        __syncwarp();
    }
}

int grid_for(const dpb_plan *p, int64_t T, int warps) {
    return (int)std::min<int64_t>((T + warps - 1) / warps, (int64_t)std::max(p->sms, 1) * 16);
}

template <typename Tio, int NKC, bool VEC, bool KEPT>
cudaError_t run_backward_lut(const dpb_plan *p, const BackwardArgs &a, int64_t T, cudaStream_t stream) {
    const size_t per_block = 256 /* alignment */ + sizeof(uint32_t) * (size_t)bwd_block_words(p->cfg.d, NKC);
    const size_t per_warp = sizeof(uint32_t) * (size_t)bwd_warp_words(p->cfg.d, p->code_len, NKC);
    const void *fn = (const void *)backward_lut_kernel<Tio, NKC, VEC, KEPT>;
    const int warps = best_warps(fn, kBwdWarps, per_block, per_warp);
    if (warps <= 0) return cudaErrorInvalidConfiguration;
    const size_t smem = per_block + (size_t)warps * per_warp;
    const cudaError_t e = allow_smem((const void *)backward_lut_kernel<Tio, NKC, VEC, KEPT>, smem);
    if (e != cudaSuccess) return e;
    backward_lut_kernel<Tio, NKC, VEC, KEPT><<<grid_for(p, T, warps), warps * 32, smem, stream>>>(a, p->t);
    return cudaGetLastError();
}

// Rows can be read 4 elements at a time: d % 4 == 0 and every row pointer
// aligned to 4 elements.
template <typename Tio>
bool rows_vec(int d, std::initializer_list<const void *> ptrs) {
    if (d % 4 != 0) return false;
    for (const void *q : ptrs)
        if (reinterpret_cast<uintptr_t>(q) % (4 * sizeof(Tio)) != 0) return false;
    return true;
}

template <typename Tio, int NKC, bool VEC>
cudaError_t run_backward_lut(const dpb_plan *p, const BackwardArgs &a, int64_t T, cudaStream_t stream) {
    if (a.norm_match && a.R) return run_backward_lut<Tio, NKC, VEC, true>(p, a, T, stream);
    return run_backward_lut<Tio, NKC, VEC, false>(p, a, T, stream);
}

template <typename Tio, int NKC>
cudaError_t run_backward_lut(const dpb_plan *p, const BackwardArgs &a, int64_t T, cudaStream_t stream) {
    if (rows_vec<Tio>(p->cfg.d, {a.x, a.gy, a.gx}) && reinterpret_cast<uintptr_t>(a.R) % 16 == 0)
        return run_backward_lut<Tio, NKC, true>(p, a, T, stream);
    return run_backward_lut<Tio, NKC, false>(p, a, T, stream);
}

template <typename Tio>
cudaError_t dispatch_backward_lut(const dpb_plan *p, const BackwardArgs &a, int64_t T, cudaStream_t stream) {
    if (p->kvh <= 2) return run_backward_lut<Tio, 2>(p, a, T, stream);
    if (p->kvh == 3) return run_backward_lut<Tio, 3>(p, a, T, stream);
    return run_backward_lut<Tio, 4>(p, a, T, stream);
}

}  // namespace

cudaError_t launch_backward(const dpb_plan *p, const void *x, const int32_t *idx,
                            const float *val, int64_t T, const float *sigma, const float *r_in,
                            const void *grad_y, void *grad_x, float *grad_val, int32_t *status,
                            cudaStream_t stream) {
    const dpb_config &c = p->cfg;
    BackwardArgs a{x, grad_y, idx, val, sigma, r_in, grad_x, grad_val, T, status, p->dM, p->dVH2,
                   c.d, p->code_len, c.norm_match, p->m_mask, p->inv_sqrt_d};
    if (c.d <= 2048) {
        return c.dtype == DPB_BF16 ? dispatch_backward_lut<__nv_bfloat16>(p, a, T, stream)
                                   : dispatch_backward_lut<float>(p, a, T, stream);
    }
    // 4 warps, fewer when the four d-length buffers per warp would not fit (d = 4096: 3)
    int warps = 4;
    while (warps > 1 && sizeof(uint32_t) * ((size_t)c.d + (size_t)warps * 4 * c.d) > kMaxSmemPerBlock) --warps;
    const size_t smem = sizeof(uint32_t) * ((size_t)c.d + (size_t)warps * 4 * c.d);
    const int grid = grid_for(p, T, warps);
    if (c.dtype == DPB_BF16) {
        const cudaError_t e = allow_smem((const void *)backward_warp_kernel<__nv_bfloat16>, smem);
        if (e != cudaSuccess) return e;
        backward_warp_kernel<__nv_bfloat16><<<grid, warps * 32, smem, stream>>>(a);
    } else {
        const cudaError_t e = allow_smem((const void *)backward_warp_kernel<float>, smem);
        if (e != cudaSuccess) return e;
        backward_warp_kernel<float><<<grid, warps * 32, smem, stream>>>(a);
    }
    return cudaGetLastError();
}

}  // namespace dpb
