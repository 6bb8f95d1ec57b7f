// dpb_encode_mma_n4.cu -- the tensor-core encoder for fields whose inverse
// coordinates take 4 five-bit sign tables (see dpb_encode_mma.cuh).
#include "dpb_encode_mma.cuh"

namespace dpb {
namespace mmaenc {

cudaError_t launch_nkc4(const dpb_plan *p, const Args &a, int warps, cudaStream_t stream) {
    return launch_nkc<4>(p, a, warps, stream);
}

}  // namespace mmaenc
}  // namespace dpb
