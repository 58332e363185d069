// gemv_bf16.cu -- bf16-weight instantiations of the weight-streaming projection.
#include "gemv_impl.cuh"

namespace mtp {

cudaError_t launch_gemv_f32(const GemvArgs& a, int epi, int grid, size_t smem, cudaStream_t s, bool pdl);

size_t gemv_smem_bytes(int rows_per_cta, int K, int wbytes, int M) {
    const int mt = M <= 1 ? 1 : M <= 2 ? 2 : M <= 4 ? 4 : 8;
    const int warps = 8;
    const int groups = (rows_per_cta + 32 / mt - 1) / (32 / mt);
    const size_t wpad = ((size_t)rows_per_cta * K * wbytes + 127) & ~(size_t)127;
    const size_t xs = K > 1024 ? (size_t)mt * K * sizeof(float) : 0;  // staged wide inputs
    return wpad + (size_t)warps * groups * 32 * sizeof(float) + xs;
}

cudaError_t launch_gemv(const GemvArgs& a, int epi, bool ln, bool w_bf16, int grid, cudaStream_t s, bool pdl) {
    const bool want_ln = epi != EPI_RESID;
    if (ln != want_ln || a.M < 1 || a.M > MAX_ROWS || a.K > 4096 || a.K % 256 != 0) return cudaErrorInvalidValue;
    const size_t smem = gemv_smem_bytes(a.rows_per_cta, a.K, w_bf16 ? 2 : 4, a.M);
    if (smem > 200 * 1024) return cudaErrorInvalidValue;
    if (!w_bf16) return launch_gemv_f32(a, epi, grid, smem, s, pdl);
    return gemv_detail::dispatch<__nv_bfloat16>(a, epi, grid, smem, s, pdl);
}

}  // namespace mtp
