// dpb_decode.cu -- the §2.1 parity decoder, one warp per token.
//
// r = sum_e val_e phi_{idx_e}: a basis entry (idx < d, Eq. 2) adds to one
// coordinate; a hashed entry adds +-val to every coordinate with the sign
// parity(M[iota] AND idx) generated on chip (Eq. 26-27), and the hashed sum is
// scaled by 1/sqrt(d) once at the end. "Normalized Reconstruction" (§2.2)
// rescales r to |x|.
#include <algorithm>

#include "dpb_device.cuh"
#include "dpb_internal.h"
#include "dpb_lut.cuh"

namespace dpb {

namespace {

struct DecodeArgs {
    const int32_t *idx;
    const float *val, *xnorm;
    void *y;
    float *R;  // nullable: r itself, fp32 [T][d], for a later backward
    int64_t T;
    int32_t *status;
    const uint32_t *M;
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
__global__ void __launch_bounds__(128) decode_warp_kernel(DecodeArgs a) {
    extern __shared__ __align__(16) uint32_t smem[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    const int d = a.d;
    uint32_t *sM = smem;
    for (int i = threadIdx.x; i < d; i += blockDim.x) sM[i] = a.M[i];
    __syncthreads();
    float *rb = reinterpret_cast<float *>(sM + d) + (size_t)warp * 2 * d;
    float *rh = rb + d;
    Tio *Y = static_cast<Tio *>(a.y);
    for (int64_t t = (int64_t)blockIdx.x * nwarps + warp; t < a.T; t += (int64_t)gridDim.x * nwarps) {
        reconstruct(a.idx + t * a.k, a.val + t * a.k, a.k, d, a.m_mask, sM, rb, rh, a.status);
        __syncwarp();
        float ss = 0.f;
        for (int i = lane; i < d; i += 32) {
            const float r = rb[i] + rh[i] * a.inv_sqrt_d;
            rb[i] = r;
            ss += r * r;
        }
        if (a.R)
            for (int i = lane; i < d; i += 32) a.R[t * d + i] = rb[i];
        float scale = 1.f;
        if (a.norm_match) {
            ss = warp_sum(ss);
            const float nr = sqrtf(ss);
            scale = nr > 0.f ? a.xnorm[t] / nr : 0.f;
        }
        for (int i = lane; i < d; i += 32) st_elem(Y, t * d + i, rb[i] * scale);
        __syncwarp();
    }
}

// ---- table-driven decoder (d <= 2048) -----------------------------------------

// Per-warp shared memory of the decoder, in 4-byte words: one sweep's tables
// (first, so that they keep the region's 128-byte alignment), r (d) and the
// hashed list (indices, coefficients).
__host__ __device__ constexpr int decode_warp_words(int d, int k, int nkc) {
    return pad32(sweep_words((d + 31) / 32, nkc) + pad4(d) + 2 * pad4(k));
}

constexpr int kDecWarps = 9;  // at most per block; four such blocks per SM at 56 registers

// R[i] = r[i] (r kept for the backward) and this lane's share of |r|^2, in
// one pass over r.
template <bool VEC>
__device__ __forceinline__ float keep_r(float *R, const float *r, int d) {
    const int lane = threadIdx.x & 31;
    float ss = 0.f;
    if (VEC) {
        for (int i = 4 * lane; i < d; i += 128) {
            const float4 v = *reinterpret_cast<const float4 *>(r + i);
            *reinterpret_cast<float4 *>(R + i) = v;
            ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
        }
    } else {
        for (int i = lane; i < d; i += 32) {
            const float v = r[i];
            R[i] = v;
            ss += v * v;
        }
    }
    return ss;
}

// KEPT: norm matching, and r kept for the backward (a separate instantiation).
template <typename Tio, int NKC, bool VEC, bool KEPT>
__global__ void __launch_bounds__(kDecWarps * 32, 4) decode_lut_kernel(DecodeArgs a, int t) {
    extern __shared__ __align__(16) uint32_t smem_raw[];
    uint32_t *smem = aligned_smem<128>(smem_raw);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    const int d = a.d;
    uint32_t *koff = smem;
    load_koff(a.M, d, t, koff);
    const int dp = pad4(d), kp = pad4(a.k);
    const int sww = sweep_words((d + 31) / 32, NKC);
    uint32_t *base = smem + pad32(d) + (size_t)warp * decode_warp_words(d, a.k, NKC);
    Sweep sw = sweep_at(base, (d + 31) / 32, NKC);
    float *r = reinterpret_cast<float *>(base + sww);
    HashedList hl{base + sww + dp, reinterpret_cast<float *>(base + sww + dp + kp), nullptr};
    Tio *Y = static_cast<Tio *>(a.y);
    for (int64_t tk = (int64_t)blockIdx.x * nwarps + warp; tk < a.T; tk += (int64_t)gridDim.x * nwarps) {
        RowOps<VEC>::fill(r, d, 0.f);
        __syncwarp();
        const int nh = split_code(a.idx + tk * a.k, a.val + tk * a.k, a.k, d, a.m_mask, r, hl, a.status);
        synthesise<NKC>(sw, hl.c, hl.a, nh, t, d, koff, a.inv_sqrt_d, r);
        float scale = 1.f;
        if (KEPT) {  // r kept and its norm in one pass
            const float nr = sqrtf(warp_sum(keep_r<VEC>(a.R + tk * d, r, d)));
            scale = nr > 0.f ? a.xnorm[tk] / nr : 0.f;
        } else {
            if (a.R) RowOps<VEC>::store(a.R + tk * d, r, d, 1.f);
            if (a.norm_match) {
                float ss = 0.f, unused = 0.f;
                RowOps<VEC>::dots(r, r, d, ss, unused);
                const float nr = sqrtf(warp_sum(ss));
                scale = nr > 0.f ? a.xnorm[tk] / nr : 0.f;
            }
        }
        RowOps<VEC>::store(Y + tk * d, r, d, scale);
        __syncwarp();
    }
}

int grid_for(const dpb_plan *p, int64_t T, int warps) {
    return (int)std::min<int64_t>((T + warps - 1) / warps, (int64_t)std::max(p->sms, 1) * 16);
}

}  // namespace

namespace {

template <typename Tio, int NKC, bool VEC, bool KEPT>
cudaError_t run_decode_lut(const dpb_plan *p, const DecodeArgs &a, int64_t T, cudaStream_t stream) {
    const size_t per_block = 128 /* alignment */ + sizeof(uint32_t) * (size_t)pad32(p->cfg.d);
    const size_t per_warp = sizeof(uint32_t) * (size_t)decode_warp_words(p->cfg.d, p->code_len, NKC);
    const void *fn = (const void *)decode_lut_kernel<Tio, NKC, VEC, KEPT>;
    const int warps = best_warps(fn, kDecWarps, per_block, per_warp);
    if (warps <= 0) return cudaErrorInvalidConfiguration;
    const size_t smem = per_block + (size_t)warps * per_warp;
    const cudaError_t e = allow_smem(fn, smem);
    if (e != cudaSuccess) return e;
    decode_lut_kernel<Tio, NKC, VEC, KEPT><<<grid_for(p, T, warps), warps * 32, smem, stream>>>(a, p->t);
    return cudaGetLastError();
}

template <typename Tio, int NKC, bool VEC>
cudaError_t run_decode_lut(const dpb_plan *p, const DecodeArgs &a, int64_t T, cudaStream_t stream) {
    if (a.norm_match && a.R) return run_decode_lut<Tio, NKC, VEC, true>(p, a, T, stream);
    return run_decode_lut<Tio, NKC, VEC, false>(p, a, T, stream);
}

template <typename Tio, int NKC>
cudaError_t run_decode_lut(const dpb_plan *p, const DecodeArgs &a, int64_t T, cudaStream_t stream) {
    // y (and r) can be written 4 elements at a time: d % 4 == 0 and both aligned to 4 elements
    if (p->cfg.d % 4 == 0 && reinterpret_cast<uintptr_t>(a.y) % (4 * sizeof(Tio)) == 0 &&
        reinterpret_cast<uintptr_t>(a.R) % 16 == 0)
        return run_decode_lut<Tio, NKC, true>(p, a, T, stream);
    return run_decode_lut<Tio, NKC, false>(p, a, T, stream);
}

template <typename Tio>
cudaError_t dispatch_decode_lut(const dpb_plan *p, const DecodeArgs &a, int64_t T, cudaStream_t stream) {
    const int nkc = (p->t + 4) / 5;
    if (nkc <= 2) return run_decode_lut<Tio, 2>(p, a, T, stream);
    if (nkc == 3) return run_decode_lut<Tio, 3>(p, a, T, stream);
    return run_decode_lut<Tio, 4>(p, a, T, stream);
}

}  // namespace

cudaError_t launch_decode(const dpb_plan *p, const int32_t *idx, const float *val, int64_t T,
                          const float *xnorm, void *y, float *r_out, int32_t *status, cudaStream_t stream) {
    const dpb_config &c = p->cfg;
    DecodeArgs a{idx, val, xnorm, y, r_out, T, status, p->dM, c.d, p->code_len, c.norm_match, p->m_mask,
                 p->inv_sqrt_d};
    if (c.d <= 2048) {
        return c.dtype == DPB_BF16 ? dispatch_decode_lut<__nv_bfloat16>(p, a, T, stream)
                                   : dispatch_decode_lut<float>(p, a, T, stream);
    }
    int warps = 4;  // fewer when the two d-length buffers per warp would not fit
    while (warps > 1 && sizeof(uint32_t) * ((size_t)c.d + (size_t)warps * 2 * c.d) > kMaxSmemPerBlock) --warps;
    const size_t smem = sizeof(uint32_t) * ((size_t)c.d + (size_t)warps * 2 * c.d);
    const int grid = grid_for(p, T, warps);
    if (c.dtype == DPB_BF16) {
        const cudaError_t e = allow_smem((const void *)decode_warp_kernel<__nv_bfloat16>, smem);
        if (e != cudaSuccess) return e;
        decode_warp_kernel<__nv_bfloat16><<<grid, warps * 32, smem, stream>>>(a);
    } else {
        const cudaError_t e = allow_smem((const void *)decode_warp_kernel<float>, smem);
        if (e != cudaSuccess) return e;
        decode_warp_kernel<float><<<grid, warps * 32, smem, stream>>>(a);
    }
    return cudaGetLastError();
}

}  // namespace dpb
