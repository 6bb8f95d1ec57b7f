// dpb_capi.cu -- the extern "C" entry points of include/dpb.h: argument
// validation on the host, then one kernel launch per call on the caller's
// stream. No allocation happens in encode/decode/backward.
#include <cstdint>
#include <cstring>
#include <map>
#include <mutex>
#include <new>
#include <tuple>
#include <utility>

#include "dpb_internal.h"

namespace dpb {
const char *last_error_message();

cudaError_t allow_smem(const void *func, size_t bytes) {
    static std::mutex mu;
    static std::map<std::pair<const void *, int>, size_t> granted;  // (kernel, device) -> bytes set
    if (bytes <= 48 * 1024) return cudaSuccess;                      // within the default limit
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    size_t &have = granted[{func, dev}];
    if (have >= bytes) return cudaSuccess;
    e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess)
        have = bytes;
    else
        cudaGetLastError();  // returned to the caller: not left for its next CUDA check
    return e;
}

int best_warps(const void *func, int max_warps, size_t per_block, size_t per_warp) {
    static std::mutex mu;
    static std::map<std::tuple<const void *, int, size_t, size_t>, int> chosen;
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    const auto key = std::make_tuple(func, dev, per_block, per_warp);
    {
        std::lock_guard<std::mutex> lock(mu);
        const auto it = chosen.find(key);
        if (it != chosen.end()) return it->second;
    }
    int best = 0, best_resident = 0;
    for (int w = max_warps; w >= 1; --w) {
        const size_t smem = per_block + (size_t)w * per_warp;
        if (smem > kMaxSmemPerBlock || allow_smem(func, smem) != cudaSuccess) continue;
        int blocks = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&blocks, func, 32 * w, smem) != cudaSuccess) {
            cudaGetLastError();
            continue;
        }
        if (blocks * w > best_resident) {
            best_resident = blocks * w;
            best = w;
        }
    }
    std::lock_guard<std::mutex> lock(mu);
    chosen[key] = best;
    return best;
}
}  // namespace dpb

namespace {

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

dpb_status check_plan(const dpb_plan *p) {
    if (!p) return dpb::fail(DPB_ERR_INVALID_ARG, "plan is NULL");
    return DPB_OK;
}

dpb_status check_workspace(void *ws, size_t bytes) {
    if (!ws) return dpb::fail(DPB_ERR_INVALID_ARG, "workspace is NULL");
    if (!aligned(ws, 256)) return dpb::fail(DPB_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
    if (bytes < 256) return dpb::fail(DPB_ERR_INVALID_ARG, "workspace needs 256 bytes, got %zu", bytes);
    return DPB_OK;
}

dpb_status check_rows(const void *ptr, const char *name, bool required) {
    if (!ptr) return required ? dpb::fail(DPB_ERR_INVALID_ARG, "%s is NULL", name) : DPB_OK;
    if (!aligned(ptr, 16)) return dpb::fail(DPB_ERR_INVALID_ARG, "%s must be 16-byte aligned", name);
    return DPB_OK;
}

dpb_status check_vec(const void *ptr, const char *name, bool required) {
    if (!ptr) return required ? dpb::fail(DPB_ERR_INVALID_ARG, "%s is NULL", name) : DPB_OK;
    if (!aligned(ptr, 4)) return dpb::fail(DPB_ERR_INVALID_ARG, "%s must be 4-byte aligned", name);
    return DPB_OK;
}

// A failed launch is reported through the returned status; the runtime's
// last-error slot is cleared so that the caller's next CUDA check (PyTorch's,
// for instance) does not see it again.
dpb_status launched(cudaError_t e, const char *what) {
    if (e != cudaSuccess) {
        cudaGetLastError();
        return dpb::fail(DPB_ERR_CUDA, "%s launch failed: %s", what, cudaGetErrorString(e));
    }
    return DPB_OK;
}

// The plan's tables live on the device current at creation; calls must be
// made with that device current.
dpb_status check_device(const dpb_plan *p) {
    if (p->device < 0) return dpb::fail(DPB_ERR_CUDA, "plan was created without a CUDA device");
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) return dpb::fail(DPB_ERR_CUDA, "cudaGetDevice failed");
    if (dev != p->device)
        return dpb::fail(DPB_ERR_INVALID_ARG, "plan lives on device %d but device %d is current", p->device, dev);
    return DPB_OK;
}

#define DPB_TRY(expr)                    \
    do {                                 \
        dpb_status s_ = (expr);          \
        if (s_ != DPB_OK) return s_;     \
    } while (0)

}  // namespace

extern "C" {

dpb_status dpb_plan_create(const dpb_config *cfg, const uint32_t *generators, dpb_plan **out) {
    if (!cfg || !out) return dpb::fail(DPB_ERR_INVALID_ARG, "cfg and out must be non-NULL");
    *out = nullptr;
    dpb_plan *p = new (std::nothrow) dpb_plan();
    if (!p) return dpb::fail(DPB_ERR_NO_MEMORY, "host allocation failed");
    dpb_status s = dpb::resolve_and_build(cfg, generators, p);
    if (s != DPB_OK) {
        delete p;
        return s;
    }
    const size_t smem = p->cfg.select_mode == DPB_SELECT_GLOBAL
                            ? dpb::encode_smem_header(p) + dpb::encode_smem_per_warp(p)
                            : dpb::encode_pl_smem(p);
    if (smem > (p->cfg.select_mode == DPB_SELECT_GLOBAL ? (size_t)200 * 1024 : dpb::kMaxSmemPerBlock)) {
        delete p;
        return dpb::fail(DPB_ERR_UNSUPPORTED, "encoder needs %zu bytes of shared memory per warp", smem);
    }
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || ndev == 0) {
        cudaGetLastError();  // host-only plan: tables and config, no compute
        p->device = -1;
        *out = p;
        return DPB_OK;
    }
    if (cudaGetDevice(&p->device) != cudaSuccess ||
        cudaDeviceGetAttribute(&p->sms, cudaDevAttrMultiProcessorCount, p->device) != cudaSuccess) {
        delete p;
        return dpb::fail(DPB_ERR_CUDA, "cudaGetDevice or its multiprocessor count failed");
    }
    const size_t mb = sizeof(uint32_t) * p->M.size(), gb = sizeof(uint32_t) * p->G.size();
    struct Up {
        uint32_t **dst;
        const std::vector<uint32_t> *src;
    } ups[] = {{&p->dM, &p->M}, {&p->dG, &p->G}, {&p->dVH, &p->VH}, {&p->dFRAG, &p->FRAG}, {&p->dDD, &p->DD},
                {&p->dGT, &p->GT},     {&p->dVH2, &p->VH2}, {&p->dCOSET, &p->COSET}};
    for (const Up &u : ups) {
        if (u.src->empty()) continue;
        const size_t bytes = sizeof(uint32_t) * u.src->size();
        if (cudaMalloc(u.dst, bytes) != cudaSuccess) {
            cudaGetLastError();
            for (const Up &v : ups) cudaFree(*v.dst);
            delete p;
            return dpb::fail(DPB_ERR_NO_MEMORY, "device table allocation failed");
        }
        if (cudaMemcpy(*u.dst, u.src->data(), bytes, cudaMemcpyHostToDevice) != cudaSuccess) {
            cudaGetLastError();
            for (const Up &v : ups) cudaFree(*v.dst);
            delete p;
            return dpb::fail(DPB_ERR_CUDA, "device table upload failed");
        }
    }
    *out = p;
    return DPB_OK;
}

dpb_status dpb_plan_destroy(dpb_plan *plan) {
    if (!plan) return DPB_OK;
    if (plan->device < 0) {
        delete plan;
        return DPB_OK;
    }
    int cur = -1;
    cudaGetDevice(&cur);
    if (cur != plan->device) cudaSetDevice(plan->device);
    cudaFree(plan->dM);
    cudaFree(plan->dG);
    cudaFree(plan->dVH);
    cudaFree(plan->dFRAG);
    cudaFree(plan->dDD);
    cudaFree(plan->dGT);
    cudaFree(plan->dVH2);
    cudaFree(plan->dCOSET);
    if (cur >= 0 && cur != plan->device) cudaSetDevice(cur);
    delete plan;
    return DPB_OK;
}

dpb_status dpb_plan_config(const dpb_plan *plan, dpb_config *out) {
    DPB_TRY(check_plan(plan));
    if (!out) return dpb::fail(DPB_ERR_INVALID_ARG, "out is NULL");
    *out = plan->cfg;
    return DPB_OK;
}

dpb_status dpb_plan_tables(const dpb_plan *plan, uint32_t *M_out, uint32_t *G_out) {
    DPB_TRY(check_plan(plan));
    if (M_out) std::memcpy(M_out, plan->M.data(), sizeof(uint32_t) * plan->M.size());
    if (G_out) std::memcpy(G_out, plan->G.data(), sizeof(uint32_t) * plan->G.size());
    return DPB_OK;
}

dpb_status dpb_code_length(const dpb_plan *plan, int32_t *k_out) {
    DPB_TRY(check_plan(plan));
    if (!k_out) return dpb::fail(DPB_ERR_INVALID_ARG, "k_out is NULL");
    *k_out = plan->code_len;
    return DPB_OK;
}

dpb_status dpb_workspace_size(const dpb_plan *plan, int64_t T, size_t *bytes) {
    DPB_TRY(check_plan(plan));
    if (!bytes || T < 0) return dpb::fail(DPB_ERR_INVALID_ARG, "bytes is NULL or T < 0");
    *bytes = dpb::kStatusBytes + dpb::tab_bytes(plan);
    return DPB_OK;
}

dpb_status dpb_encode(const dpb_plan *plan, const void *x, int64_t T, const float *mu,
                      const float *sigma, int32_t *idx, float *val, float *xnorm,
                      void *workspace, size_t workspace_bytes, void *stream) {
    DPB_TRY(check_plan(plan));
    if (T < 0) return dpb::fail(DPB_ERR_INVALID_ARG, "T < 0");
    if (T == 0) return DPB_OK;
    if ((mu == nullptr) != (sigma == nullptr))
        return dpb::fail(DPB_ERR_INVALID_ARG, "mu and sigma must both be given or both be NULL");
    DPB_TRY(check_rows(x, "x", true));
    DPB_TRY(check_vec(mu, "mu", false));
    DPB_TRY(check_vec(sigma, "sigma", false));
    DPB_TRY(check_vec(idx, "idx", true));
    DPB_TRY(check_vec(val, "val", true));
    DPB_TRY(check_vec(xnorm, "xnorm", false));
    DPB_TRY(check_workspace(workspace, workspace_bytes));
    DPB_TRY(check_device(plan));
    const size_t tb = dpb::tab_bytes(plan);
    float2 *tab = tb > 0 && workspace_bytes >= dpb::kStatusBytes + tb
                      ? reinterpret_cast<float2 *>(static_cast<char *>(workspace) + dpb::kStatusBytes)
                      : nullptr;
    return launched(dpb::launch_encode(plan, x, T, mu, sigma, idx, val, xnorm,
                                       static_cast<int32_t *>(workspace), tab,
                                       static_cast<cudaStream_t>(stream)),
                    "encode");
}

dpb_status dpb_decode(const dpb_plan *plan, const int32_t *idx, const float *val, int64_t T,
                      const float *xnorm, void *y, float *r_out, void *workspace, size_t workspace_bytes,
                      void *stream) {
    DPB_TRY(check_plan(plan));
    if (T < 0) return dpb::fail(DPB_ERR_INVALID_ARG, "T < 0");
    if (T == 0) return DPB_OK;
    DPB_TRY(check_vec(idx, "idx", true));
    DPB_TRY(check_vec(val, "val", true));
    DPB_TRY(check_vec(xnorm, "xnorm", plan->cfg.norm_match != 0));
    DPB_TRY(check_rows(y, "y", true));
    DPB_TRY(check_rows(r_out, "r_out", false));
    DPB_TRY(check_workspace(workspace, workspace_bytes));
    DPB_TRY(check_device(plan));
    return launched(dpb::launch_decode(plan, idx, val, T, xnorm, y, r_out, static_cast<int32_t *>(workspace),
                                       static_cast<cudaStream_t>(stream)),
                    "decode");
}

dpb_status dpb_backward(const dpb_plan *plan, const void *x, const int32_t *idx,
                        const float *val, int64_t T, const float *sigma, const float *r,
                        const void *grad_y, void *grad_x, float *grad_val, void *workspace,
                        size_t workspace_bytes, void *stream) {
    DPB_TRY(check_plan(plan));
    if (T < 0) return dpb::fail(DPB_ERR_INVALID_ARG, "T < 0");
    if (T == 0) return DPB_OK;
    DPB_TRY(check_rows(x, "x", true));
    DPB_TRY(check_vec(idx, "idx", true));
    DPB_TRY(check_vec(val, "val", true));
    DPB_TRY(check_vec(sigma, "sigma", false));
    DPB_TRY(check_rows(r, "r", false));
    DPB_TRY(check_rows(grad_y, "grad_y", true));
    DPB_TRY(check_rows(grad_x, "grad_x", true));
    DPB_TRY(check_vec(grad_val, "grad_val", true));
    DPB_TRY(check_workspace(workspace, workspace_bytes));
    DPB_TRY(check_device(plan));
    return launched(dpb::launch_backward(plan, x, idx, val, T, sigma, r, grad_y, grad_x, grad_val,
                                         static_cast<int32_t *>(workspace),
                                         static_cast<cudaStream_t>(stream)),
                    "backward");
}

dpb_status dpb_forward(const dpb_plan *plan, const void *x, int64_t T, const float *mu, const float *sigma,
                       int32_t *idx, float *val, float *xnorm, void *y, float *r_out, void *workspace,
                       size_t workspace_bytes, void *stream) {
    DPB_TRY(check_plan(plan));
    if (plan->cfg.norm_match && T > 0 && !xnorm)
        return dpb::fail(DPB_ERR_INVALID_ARG, "xnorm is required with norm_match");
    DPB_TRY(dpb_encode(plan, x, T, mu, sigma, idx, val, xnorm, workspace, workspace_bytes, stream));
    return dpb_decode(plan, idx, val, T, xnorm, y, r_out, workspace, workspace_bytes, stream);
}

dpb_status dpb_stats_accumulate(const dpb_plan *plan, const void *x, int64_t T, const float *mu,
                                const float *sigma, const int32_t *sample, int32_t n_sample, double *acc,
                                void *workspace, size_t workspace_bytes, void *stream) {
    DPB_TRY(check_plan(plan));
    if (T < 0 || n_sample < 0) return dpb::fail(DPB_ERR_INVALID_ARG, "T < 0 or n_sample < 0");
    if (T == 0 && n_sample > 0) return dpb::fail(DPB_ERR_INVALID_ARG, "sampled rows of an empty batch");
    if (T == 0) return DPB_OK;
    if ((mu == nullptr) != (sigma == nullptr))
        return dpb::fail(DPB_ERR_INVALID_ARG, "mu and sigma must both be given or both be NULL");
    if (!dpb::stats_supported(plan, nullptr))
        return dpb::fail(DPB_ERR_UNSUPPORTED, "kept sets above 64 or the sampled search exceeds shared memory");
    DPB_TRY(check_rows(x, "x", true));
    DPB_TRY(check_vec(mu, "mu", false));
    DPB_TRY(check_vec(sigma, "sigma", false));
    DPB_TRY(check_vec(sample, "sample", n_sample > 0));
    if (!acc) return dpb::fail(DPB_ERR_INVALID_ARG, "acc is NULL");
    if (!aligned(acc, 8)) return dpb::fail(DPB_ERR_INVALID_ARG, "acc must be 8-byte aligned");
    DPB_TRY(check_workspace(workspace, workspace_bytes));
    DPB_TRY(check_device(plan));
    return launched(dpb::launch_stats_accumulate(plan, x, T, mu, sigma, sample, n_sample, acc,
                                                 static_cast<int32_t *>(workspace),
                                                 static_cast<cudaStream_t>(stream)),
                    "stats accumulate");
}

dpb_status dpb_stats_update(const dpb_plan *plan, double *acc, float alpha, float *mu, float *sigma,
                            void *stream) {
    DPB_TRY(check_plan(plan));
    if (!(alpha > 0.f && alpha < 1.f)) return dpb::fail(DPB_ERR_INVALID_ARG, "alpha must lie in (0, 1)");
    if (!acc) return dpb::fail(DPB_ERR_INVALID_ARG, "acc is NULL");
    if (!aligned(acc, 8)) return dpb::fail(DPB_ERR_INVALID_ARG, "acc must be 8-byte aligned");
    DPB_TRY(check_vec(mu, "mu", true));
    DPB_TRY(check_vec(sigma, "sigma", true));
    DPB_TRY(check_device(plan));
    return launched(dpb::launch_stats_update(plan, acc, alpha, mu, sigma, static_cast<cudaStream_t>(stream)),
                    "stats update");
}

dpb_status dpb_workspace_status(const void *workspace, int clear, int32_t *status_out, void *stream) {
    if (!workspace || !status_out) return dpb::fail(DPB_ERR_INVALID_ARG, "workspace and status_out must be non-NULL");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int32_t v = 0;
    if (cudaMemcpyAsync(&v, workspace, sizeof(v), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
        return dpb::fail(DPB_ERR_CUDA, "reading the workspace status failed");
    if (clear && v != 0) {
        if (cudaMemsetAsync(const_cast<void *>(workspace), 0, sizeof(int32_t), s) != cudaSuccess ||
            cudaStreamSynchronize(s) != cudaSuccess)
            return dpb::fail(DPB_ERR_CUDA, "clearing the workspace status failed");
    }
    *status_out = v;
    return v ? dpb::fail(DPB_ERR_DEVICE, "device status 0x%x", v) : DPB_OK;
}

const char *dpb_status_string(dpb_status s) {
    switch (s) {
        case DPB_OK: return "ok";
        case DPB_ERR_INVALID_ARG: return "invalid argument";
        case DPB_ERR_UNSUPPORTED: return "unsupported configuration";
        case DPB_ERR_CUDA: return "CUDA error";
        case DPB_ERR_TIMEOUT: return "device wait timed out";
        case DPB_ERR_NO_MEMORY: return "out of memory";
        case DPB_ERR_DEVICE: return "device-side error flagged";
    }
    return "unknown status";
}

const char *dpb_last_error(void) { return dpb::last_error_message(); }

}  // extern "C"
