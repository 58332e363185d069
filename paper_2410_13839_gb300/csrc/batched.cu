// batched.cu -- the row-wise steps of the batched path (many fed rows per
// pass), between the tensor-core projections of tc_gemm.cu:
//
//   pack_rows   one CTA per row: LayerNorm (LN1 / LN2, Sec. III-A), a plain
//               copy (attention output) or GELU (FFN hidden rows, which are
//               zeroed after reading so the next split-K GEMM can accumulate
//               into them), then the fp32 row as bf16 hi + lo parts, the
//               activation operand of the tensor-core GEMM.  Rows of no
//               sequence are written as zeros.
//   qkv_finish  one CTA per row: the projected q|k|v row (bias included,
//               head-major features h*192 + {0,64,128} + dd) -> the query row
//               for the attention, keys and values -> the paged cache (bf16,
//               16-byte chunks of key row t at chunk ^ (t & 7)); the row is
//               zeroed for the next layer's split-K accumulation.
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

constexpr int QF_THREADS = 128;

// One CTA per row; each thread takes 8 consecutive features (one 16-byte
// chunk of a key/value row): two float4 loads, then the query as two float4
// stores or the key/value chunk as one 16-byte store at its swizzled place.
__global__ void __launch_bounds__(QF_THREADS) qkv_finish_kernel(const QkvFinishArgs a) {
    const int r = blockIdx.x, tid = threadIdx.x;
    TraceEnd trace_guard(a.trace);
    pdl_launch_dependents();
    pdl_wait();
    trace_wait(a.trace);
    const int seq = a.row_seq[r], pos = a.row_pos[r];
    const int H = a.n_heads, P = a.page_size, d = H * HEAD_DIM;
    float* row = a.qkv + (size_t)r * 3 * d;
    int page = -1;
    if (seq >= 0) {
        page = a.block_table[(size_t)seq * a.bt_stride + pos / P];
        if (page < 0 && tid == 0) atomicOr(a.err, ERR_BOUNDS);
    }
    const int t = pos % P;
    const float4 zero = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int c = tid; c < 3 * d / 8; c += QF_THREADS) {
        float4* src = reinterpret_cast<float4*>(row + c * 8);
        const float4 y0 = src[0], y1 = src[1];
        src[0] = zero;
        src[1] = zero;
        if (seq < 0) continue;
        const int i = c * 8, h = i / (3 * HEAD_DIM), sec = (i / HEAD_DIM) % 3, dd = i % HEAD_DIM;
        if (sec == 0) {
            float4* q = reinterpret_cast<float4*>(a.q + (size_t)r * d + h * HEAD_DIM + dd);
            q[0] = y0;
            q[1] = y1;
        } else if (page >= 0) {
            uint4 pk;
            auto pair = [](float lo, float hi) {
                return (uint32_t)f32_to_bf16_bits(lo) | ((uint32_t)f32_to_bf16_bits(hi) << 16);
            };
            pk.x = pair(y0.x, y0.y);
            pk.y = pair(y0.z, y0.w);
            pk.z = pair(y1.x, y1.y);
            pk.w = pair(y1.z, y1.w);
            const long long idx = (long long)page * a.page_elems + a.layer_off + (long long)(sec - 1) * H * P * HEAD_DIM +
                                  (long long)h * P * HEAD_DIM + (long long)t * HEAD_DIM + (((dd >> 3) ^ (t & 7)) << 3);
            *reinterpret_cast<uint4*>(reinterpret_cast<uint16_t*>(a.kv_pool) + idx) = pk;
        }
    }
}

template <typename K, typename A>
cudaError_t launch_rows(K kern, const A& args, int rows, cudaStream_t s, bool pdl, int threads = PK_THREADS) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(rows);
    cfg.blockDim = dim3(threads);
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

cudaError_t launch_qkv_finish(const QkvFinishArgs& a, cudaStream_t s, bool pdl) {
    if (a.m < 1) return cudaErrorInvalidValue;
    return launch_rows(qkv_finish_kernel, a, a.m, s, pdl, QF_THREADS);
}

}  // namespace mtp
