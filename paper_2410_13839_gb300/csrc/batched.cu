// batched.cu -- the row-wise steps of the batched path (many fed rows per
// pass), between the tensor-core projections of tc_gemm.cu:
//
//   pack_rows   one CTA per row: LayerNorm (LN1 / LN2, Sec. III-A), a plain
//               copy (attention output) or GELU (FFN hidden rows, which are
//               zeroed after reading so the next split-K GEMM can accumulate
//               into them), then the fp32 row as bf16 hi + lo parts, the
//               activation operand of the tensor-core GEMM.  Rows of no
//               sequence are written as zeros.
#include <math.h>

#include "common.cuh"
#include "kernels.cuh"

namespace mtp {
namespace {

constexpr int PK_THREADS = 256;

__device__ __forceinline__ float block_sum(float v, float* red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_sum(v);
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < PK_THREADS / 32; ++w) t += red[w];
    return t;
}

// ALL: every row is packed (no row_seq) and zero_buf is zeroed first.
template <bool ALL>
__global__ void __launch_bounds__(PK_THREADS) pack_rows_kernel(const PackArgs a) {
    __shared__ float red[PK_THREADS / 32];
    constexpr int MAXV = 16;  // values per thread: K <= 4096
    const int r = blockIdx.x, tid = threadIdx.x;
    TraceEnd trace_guard(a.trace);
    pdl_launch_dependents();
    pdl_wait();
    trace_wait(a.trace);
    if constexpr (ALL)
        for (long long i = (long long)r * PK_THREADS + tid; i < a.zero_n; i += (long long)a.m * PK_THREADS)
            a.zero_buf[i] = 0.f;
    const bool on = ALL || a.row_seq[r] >= 0;
    const int K = a.k;
    float v[MAXV];
#pragma unroll
    for (int i = 0; i < MAXV; ++i) {
        const int c = tid + i * PK_THREADS;
        v[i] = on && c < K ? a.x[(size_t)r * a.ldx + c] : 0.f;
    }
    if (a.mode == PACK_LN) {  // two-pass mean / variance over the row
        float s = 0.f;
#pragma unroll
        for (int i = 0; i < MAXV; ++i) s += v[i];
        const float mean = block_sum(s, red) / (float)K;
        float q = 0.f;
#pragma unroll
        for (int i = 0; i < MAXV; ++i) {
            const int c = tid + i * PK_THREADS;
            const float t = c < K ? v[i] - mean : 0.f;
            q += t * t;
        }
        const float rstd = 1.0f / sqrtf(block_sum(q, red) / (float)K + a.eps);
#pragma unroll
        for (int i = 0; i < MAXV; ++i) {
            const int c = tid + i * PK_THREADS;
            if (c < K) v[i] = on ? (v[i] - mean) * rstd * a.gamma[c] + a.beta[c] : 0.f;
        }
    } else if (a.mode == PACK_GELU) {
#pragma unroll
        for (int i = 0; i < MAXV; ++i) {
            const int c = tid + i * PK_THREADS;
            if (c < K) {
                if (on) v[i] = gelu_erf(v[i]);
                if (a.zero_after) a.zero_after[(size_t)r * a.ldx + c] = 0.f;
            }
        }
    }
#pragma unroll
    for (int i = 0; i < MAXV; ++i) {
        const int c = tid + i * PK_THREADS;
        if (c < K) {
            const __nv_bfloat16 hi = __float2bfloat16_rn(v[i]);
            a.hi[(size_t)r * K + c] = hi;
            a.lo[(size_t)r * K + c] = __float2bfloat16_rn(v[i] - __bfloat162float(hi));
        }
    }
}

template <typename K, typename A>
cudaError_t launch_rows(K kern, const A& args, int rows, cudaStream_t s, bool pdl) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(rows);
    cfg.blockDim = dim3(PK_THREADS);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, args);
}

}  // namespace

cudaError_t launch_pack_rows(const PackArgs& a, cudaStream_t s, bool pdl) {
    if (a.k < 1 || a.k > 16 * PK_THREADS || a.m < 1) return cudaErrorInvalidValue;
    if (a.row_seq == nullptr) {
        if (a.zero_n > 0 && a.zero_buf == nullptr) return cudaErrorInvalidValue;
        return launch_rows(pack_rows_kernel<true>, a, a.m, s, pdl);
    }
    if (a.zero_buf) return cudaErrorInvalidValue;  // zeroing comes with the every-row variant
    return launch_rows(pack_rows_kernel<false>, a, a.m, s, pdl);
}

}  // namespace mtp
