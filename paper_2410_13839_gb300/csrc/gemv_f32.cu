// gemv_f32.cu -- fp32-weight instantiations of the weight-streaming projection.
#include "gemv_impl.cuh"

namespace mtp {

cudaError_t launch_gemv_f32(const GemvArgs& a, int epi, int grid, size_t smem, cudaStream_t s, bool pdl) {
    return gemv_detail::dispatch<float>(a, epi, grid, smem, s, pdl);
}

}  // namespace mtp
