// dpb_noalloc.cu -- dpb_encode_noalloc: the encoder for callers that cannot
// allocate device memory.
//
// Some callers cannot call cudaMalloc or hand the library a workspace: code
// that runs inside another runtime's memory arena (an inference server or a
// game engine that owns every device allocation and gives plug-ins only
// their input and output buffers), or plain-C callers with no allocator of
// their own. This entry point needs nothing from them but x and the output
// buffers: the scratch that dpb_encode keeps in the caller's workspace (the
// device status word) lives here in a file-scope device array instead.
//
// The array is a fixed kNoAllocScratchBytes per device; every GPU that loads
// the library holds it until the process exits. What the encoder needs of it
// is the status word alone (kStatusBytes), whatever the plan and T: the
// optional packed (mu, 1/sigma) copy of the standardisation tables, which
// dpb_encode keeps in a large enough workspace, is left out here, so a
// standardised call reads mu and sigma from the caller's two tables (the same
// arithmetic, one more load per candidate). No plan or batch size can need
// more than the array holds; a static_assert ties the two sizes together.
// Host code cannot use the array's name as a device address, so the address
// is looked up once per device with cudaGetSymbolAddress and cached.
#include <cstdint>
#include <mutex>

#include "dpb_internal.h"

namespace {

constexpr size_t kNoAllocScratchBytes = 4096;
constexpr int kMaxDevices = 64;
static_assert(dpb::kStatusBytes <= kNoAllocScratchBytes,
              "the built-in scratch must hold the device status word");

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_scratch_mu;
void *g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch array on `dev` (which must be current).
dpb_status scratch_on(int dev, void **out) {
    if (dev < 0 || dev >= kMaxDevices)
        return dpb::fail(DPB_ERR_UNSUPPORTED, "device %d is beyond the %d devices the built-in scratch tracks",
                         dev, kMaxDevices);
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (!g_scratch_ptr[dev]) {
        void *p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || !p)
            return dpb::fail(DPB_ERR_CUDA, "cudaGetSymbolAddress of the built-in scratch failed: %s",
                             cudaGetErrorString(e));
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return DPB_OK;
}

bool misaligned(const void *p, size_t a) { return p && (reinterpret_cast<uintptr_t>(p) % a) != 0; }

}  // namespace

extern "C" dpb_status dpb_encode_noalloc(const dpb_plan *plan, const void *x, int64_t T,
                                         const float *mu, const float *sigma, int32_t *idx,
                                         float *val, float *xnorm, int32_t *status_out,
                                         void *stream) {
    if (!plan) return dpb::fail(DPB_ERR_INVALID_ARG, "plan is NULL");
    if (T < 0) return dpb::fail(DPB_ERR_INVALID_ARG, "T < 0");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (misaligned(status_out, 4)) return dpb::fail(DPB_ERR_INVALID_ARG, "status_out must be 4-byte aligned");
    if (T == 0) {
        if (status_out && cudaMemsetAsync(status_out, 0, sizeof(int32_t), s) != cudaSuccess)
            return dpb::fail(DPB_ERR_CUDA, "clearing status_out failed");
        return DPB_OK;
    }
    if (!x || !idx || !val) return dpb::fail(DPB_ERR_INVALID_ARG, "x, idx and val must be non-NULL");
    if (misaligned(x, 16)) return dpb::fail(DPB_ERR_INVALID_ARG, "x must be 16-byte aligned");
    if (misaligned(idx, 4) || misaligned(val, 4) || misaligned(xnorm, 4) || misaligned(mu, 4) ||
        misaligned(sigma, 4))
        return dpb::fail(DPB_ERR_INVALID_ARG, "idx, val, xnorm, mu and sigma must be 4-byte aligned");
    if ((mu == nullptr) != (sigma == nullptr))
        return dpb::fail(DPB_ERR_INVALID_ARG, "mu and sigma must both be given or both be NULL");
    // the built-in scratch holds the status word only (see the static_assert);
    // the optional packed tables of a workspace are left out, and the encoder
    // then reads mu and sigma apart
    if (plan->device < 0) return dpb::fail(DPB_ERR_CUDA, "plan was created without a CUDA device");
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) return dpb::fail(DPB_ERR_CUDA, "cudaGetDevice failed");
    if (dev != plan->device)
        return dpb::fail(DPB_ERR_INVALID_ARG, "plan lives on device %d but device %d is current",
                         plan->device, dev);
    void *scratch = nullptr;
    const dpb_status ss = scratch_on(dev, &scratch);
    if (ss != DPB_OK) return ss;
    int32_t *status = static_cast<int32_t *>(scratch);
    // the array keeps the previous call's contents: the status word starts at zero
    if (cudaMemsetAsync(status, 0, sizeof(int32_t), s) != cudaSuccess)
        return dpb::fail(DPB_ERR_CUDA, "clearing the built-in scratch failed");
    const cudaError_t e = dpb::launch_encode(plan, x, T, mu, sigma, idx, val, xnorm, status, nullptr, s);
    if (e != cudaSuccess) return dpb::fail(DPB_ERR_CUDA, "encode launch failed: %s", cudaGetErrorString(e));
    if (status_out &&
        cudaMemcpyAsync(status_out, status, sizeof(int32_t), cudaMemcpyDeviceToDevice, s) != cudaSuccess)
        return dpb::fail(DPB_ERR_CUDA, "copying the status word failed");
    return DPB_OK;
}
