// dpb_encode_mma.cu -- launch shape and dispatch of the tensor-core encoder
// (kernels in dpb_encode_mma.cuh, one translation unit per table count).
#include <algorithm>

#include "dpb_encode_mma.cuh"

namespace dpb {

size_t encode_mma_smem(const dpb_plan *p, int warps) {
    const int nblk = p->cfg.d / 32, nkc = std::max(2, p->kvh);
    return sizeof(uint32_t) * ((size_t)mmaenc::block_words(p->cfg.levels, nblk, nkc) +
                               (size_t)warps * mmaenc::warp_words(nblk, p->cfg.k));
}

int encode_mma_warps(const dpb_plan *p) {
    for (int w : {20, 16, 12, 8, 4})
        if (encode_mma_smem(p, w) <= kMaxSmemPerBlock) return w;
    return 0;
}

cudaError_t launch_encode_mma(const dpb_plan *p, const void *x, int64_t T, const float *mu,
                              const float *sigma, const float2 *tab, int32_t *idx, float *val, float *xnorm,
                              int32_t *status, cudaStream_t stream) {
    const dpb_config &c = p->cfg;
    mmaenc::Args a{};
    a.x = static_cast<const __nv_bfloat16 *>(x);
    a.T = T;
    a.mu = mu;
    a.sigma = sigma;
    a.tab = tab;
    a.coset = c.scoring == DPB_SCORING_COSET_WHT ? p->dCOSET : nullptr;
    a.idx = idx;
    a.val = val;
    a.xnorm = xnorm;
    a.status = status;
    a.frag = p->dFRAG;
    a.G = p->dG;
    a.VH = p->dVH;
    a.DD = p->dDD;
    a.d = c.d;
    a.nblk = c.d / 32;
    a.levels = c.levels;
    a.k = c.k;
    a.beam = c.beam;
    a.t = p->t;
    a.ecap = mmaenc::entrant_cap(c.k, c.d / 32);
    a.inv_sqrt_d = p->inv_sqrt_d;
    const int warps = encode_mma_warps(p);
    const int nkc = std::max(2, p->kvh);
    if (nkc == 2) return mmaenc::launch_nkc2(p, a, warps, stream);
    if (nkc == 3) return mmaenc::launch_nkc3(p, a, warps, stream);
    return mmaenc::launch_nkc4(p, a, warps, stream);
}

}  // namespace dpb
