// batched.cu -- the row-wise steps of the batched path (many fed rows per
// pass), between the tensor-core projections of tc_gemm.cu:
//
//   pack_rows   one CTA per row (float4 chunks per thread): LayerNorm (LN1 /
//               LN2, Sec. III-A; gain and offset read before the dependency
//               wait, one block barrier for the statistics), a plain
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

// ALL: every row is packed (no row_seq) and zero_buf is zeroed first.  Thread t
// holds the float4 chunks t, t + PK_THREADS, ... of its row (k % 4 == 0).
// MAXQ: chunks per thread (k <= 4 * PK_THREADS * MAXQ), a template argument so that rows of
// d = 1024 keep few registers and one wave of CTAs fits 512 rows.
template <bool ALL, int MAXQ>
__global__ void __launch_bounds__(PK_THREADS) pack_rows_kernel(const PackArgs a) {
    constexpr int NW = PK_THREADS / 32;
    __shared__ float s_wstat[3][NW];  // per warp: element count, mean, sum of squared deviations
    const int r = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int K = a.k, nq = K / 4;
    TraceEnd trace_guard(a.trace);
    float4 gam[MAXQ], bet[MAXQ];  // LayerNorm gain and offset: weights, read before the dependency wait
    if (a.mode == PACK_LN) {
#pragma unroll
        for (int i = 0; i < MAXQ; ++i) {
            const int q = tid + i * PK_THREADS;
            gam[i] = q < nq ? __ldg(reinterpret_cast<const float4*>(a.gamma) + q) : make_float4(0.f, 0.f, 0.f, 0.f);
            bet[i] = q < nq ? __ldg(reinterpret_cast<const float4*>(a.beta) + q) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
    }
    pdl_launch_dependents();
    pdl_wait();
    trace_wait(a.trace);
    if constexpr (ALL)
        for (long long i = (long long)r * PK_THREADS + tid; i < a.zero_n; i += (long long)a.m * PK_THREADS)
            a.zero_buf[i] = 0.f;
    const bool on = ALL || a.row_seq[r] >= 0;
    const float4* xr = reinterpret_cast<const float4*>(a.x + (size_t)r * a.ldx);
    float4 v[MAXQ];
#pragma unroll
    for (int i = 0; i < MAXQ; ++i) {
        const int q = tid + i * PK_THREADS;
        v[i] = on && q < nq ? xr[q] : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    if (a.mode == PACK_LN) {
        // each warp's mean and sum of squared deviations over its own elements (two passes
        // over registers), merged over the warps: mean = sum n_w mean_w / K and
        // M2 = sum [M2_w + n_w (mean_w - mean)^2]; one block barrier
        float s = 0.f, cnt = 0.f;
#pragma unroll
        for (int i = 0; i < MAXQ; ++i)
            if (tid + i * PK_THREADS < nq) {
                s += (v[i].x + v[i].y) + (v[i].z + v[i].w);
                cnt += 4.f;
            }
        const float n_w = warp_sum(cnt);
        const float mean_w = n_w > 0.f ? warp_sum(s) / n_w : 0.f;
        float q2 = 0.f;
#pragma unroll
        for (int i = 0; i < MAXQ; ++i)
            if (tid + i * PK_THREADS < nq) {
                const float d0 = v[i].x - mean_w, d1 = v[i].y - mean_w, d2 = v[i].z - mean_w, d3 = v[i].w - mean_w;
                q2 += (d0 * d0 + d1 * d1) + (d2 * d2 + d3 * d3);
            }
        const float m2_w = warp_sum(q2);
        if (lane == 0) {
            s_wstat[0][warp] = n_w;
            s_wstat[1][warp] = mean_w;
            s_wstat[2][warp] = m2_w;
        }
        __syncthreads();
        float mean = 0.f;
#pragma unroll
        for (int w = 0; w < NW; ++w) mean += s_wstat[0][w] * s_wstat[1][w];
        mean /= (float)K;
        float m2 = 0.f;
#pragma unroll
        for (int w = 0; w < NW; ++w) {
            const float dm = s_wstat[1][w] - mean;
            m2 += s_wstat[2][w] + s_wstat[0][w] * dm * dm;
        }
        const float rstd = 1.0f / sqrtf(m2 / (float)K + a.eps);
#pragma unroll
        for (int i = 0; i < MAXQ; ++i) {
            v[i].x = on ? (v[i].x - mean) * rstd * gam[i].x + bet[i].x : 0.f;
            v[i].y = on ? (v[i].y - mean) * rstd * gam[i].y + bet[i].y : 0.f;
            v[i].z = on ? (v[i].z - mean) * rstd * gam[i].z + bet[i].z : 0.f;
            v[i].w = on ? (v[i].w - mean) * rstd * gam[i].w + bet[i].w : 0.f;
        }
    } else if (a.mode == PACK_GELU) {
#pragma unroll
        for (int i = 0; i < MAXQ; ++i) {
            const int q = tid + i * PK_THREADS;
            if (q < nq) {
                if (on) v[i] = make_float4(gelu_erf(v[i].x), gelu_erf(v[i].y), gelu_erf(v[i].z), gelu_erf(v[i].w));
                if (a.zero_after)
                    reinterpret_cast<float4*>(a.zero_after + (size_t)r * a.ldx)[q] = make_float4(0.f, 0.f, 0.f, 0.f);
            }
        }
    }
#pragma unroll
    for (int i = 0; i < MAXQ; ++i) {
        const int q = tid + i * PK_THREADS;
        if (q < nq) {
            const float x[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
            uint32_t hi[2], lo[2];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const __nv_bfloat16 h0 = __float2bfloat16_rn(x[2 * h]), h1 = __float2bfloat16_rn(x[2 * h + 1]);
                const __nv_bfloat16 l0 = __float2bfloat16_rn(x[2 * h] - __bfloat162float(h0));
                const __nv_bfloat16 l1 = __float2bfloat16_rn(x[2 * h + 1] - __bfloat162float(h1));
                hi[h] = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
                lo[h] = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
            }
            reinterpret_cast<uint2*>(a.hi + (size_t)r * K)[q] = make_uint2(hi[0], hi[1]);
            reinterpret_cast<uint2*>(a.lo + (size_t)r * K)[q] = make_uint2(lo[0], lo[1]);
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
    if (a.k < 4 || a.k > 16 * PK_THREADS || a.k % 4 || a.ldx % 4 || a.m < 1) return cudaErrorInvalidValue;
    if ((reinterpret_cast<uintptr_t>(a.x) | reinterpret_cast<uintptr_t>(a.hi) | reinterpret_cast<uintptr_t>(a.lo) |
         reinterpret_cast<uintptr_t>(a.zero_after) | reinterpret_cast<uintptr_t>(a.gamma) |
         reinterpret_cast<uintptr_t>(a.beta)) & 15)
        return cudaErrorInvalidValue;  // float4 rows
    const int chunks = (a.k / 4 + PK_THREADS - 1) / PK_THREADS;
    if (a.row_seq == nullptr) {
        if (a.zero_n > 0 && a.zero_buf == nullptr) return cudaErrorInvalidValue;
        if (chunks <= 1) return launch_rows(pack_rows_kernel<true, 1>, a, a.m, s, pdl);
        return launch_rows(pack_rows_kernel<true, 4>, a, a.m, s, pdl);
    }
    if (a.zero_buf) return cudaErrorInvalidValue;  // zeroing comes with the every-row variant
    if (chunks <= 1) return launch_rows(pack_rows_kernel<false, 1>, a, a.m, s, pdl);
    return launch_rows(pack_rows_kernel<false, 4>, a, a.m, s, pdl);
}

}  // namespace mtp
