// dpb_decode.cu -- the §2.1 parity decoder and the backward of the whole
// encode-then-decode map, one warp per token.
//
// r = sum_e val_e phi_{idx_e}: a basis entry (idx < d, Eq. 2) adds to one
// coordinate; a hashed entry adds +-val to every coordinate with the sign
// parity(M[iota] AND idx) generated on chip (Eq. 26-27), and the hashed sum is
// scaled by 1/sqrt(d) once at the end. "Normalized Reconstruction" (§2.2)
// rescales r to |x|.
#include <algorithm>

#include "dpb_device.cuh"
#include "dpb_internal.h"

namespace dpb {

namespace {

struct DecodeArgs {
    const int32_t *idx;
    const float *val, *xnorm;
    void *y;
    int64_t T;
    int32_t *status;
    const uint32_t *M;
    int d, k, norm_match;
    uint32_t m_mask;
    float inv_sqrt_d;
};

struct BackwardArgs {
    const void *x, *gy;
    const int32_t *idx;
    const float *val, *sigma;
    void *gx;
    float *gval;
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
            reconstruct(it, vt, a.k, d, a.m_mask, sM, rb, rh, a.status);
            __syncwarp();
            float srr = 0.f, sgr = 0.f;
            for (int i = lane; i < d; i += 32) {
                const float r = rb[i] + rh[i] * a.inv_sqrt_d;
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

int grid_for(const dpb_plan *p, int64_t T, int warps) {
    int sms = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, p->device);
    return (int)std::min<int64_t>((T + warps - 1) / warps, (int64_t)sms * 16);
}

}  // namespace

cudaError_t launch_decode(const dpb_plan *p, const int32_t *idx, const float *val, int64_t T,
                          const float *xnorm, void *y, int32_t *status, cudaStream_t stream) {
    const dpb_config &c = p->cfg;
    DecodeArgs a{idx, val, xnorm, y, T, status, p->dM, c.d, p->code_len, c.norm_match, p->m_mask,
                 p->inv_sqrt_d};
    const int warps = 4;
    const size_t smem = sizeof(uint32_t) * ((size_t)c.d + (size_t)warps * 2 * c.d);
    const int grid = grid_for(p, T, warps);
    if (c.dtype == DPB_BF16) {
        cudaFuncSetAttribute(decode_warp_kernel<__nv_bfloat16>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        decode_warp_kernel<__nv_bfloat16><<<grid, warps * 32, smem, stream>>>(a);
    } else {
        cudaFuncSetAttribute(decode_warp_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        decode_warp_kernel<float><<<grid, warps * 32, smem, stream>>>(a);
    }
    return cudaGetLastError();
}

cudaError_t launch_backward(const dpb_plan *p, const void *x, const int32_t *idx,
                            const float *val, int64_t T, const float *sigma, const void *grad_y,
                            void *grad_x, float *grad_val, int32_t *status,
                            cudaStream_t stream) {
    const dpb_config &c = p->cfg;
    BackwardArgs a{x, grad_y, idx, val, sigma, grad_x, grad_val, T, status, p->dM,
                   c.d, p->code_len, c.norm_match, p->m_mask, p->inv_sqrt_d};
    const int warps = 4;
    const size_t smem = sizeof(uint32_t) * ((size_t)c.d + (size_t)warps * 4 * c.d);
    const int grid = grid_for(p, T, warps);
    if (c.dtype == DPB_BF16) {
        cudaFuncSetAttribute(backward_warp_kernel<__nv_bfloat16>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        backward_warp_kernel<__nv_bfloat16><<<grid, warps * 32, smem, stream>>>(a);
    } else {
        cudaFuncSetAttribute(backward_warp_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        backward_warp_kernel<float><<<grid, warps * 32, smem, stream>>>(a);
    }
    return cudaGetLastError();
}

}  // namespace dpb
