// frag.cuh -- warp-level tensor-core fragments and row helpers shared by the
// block kernels (layer_fused.cu) and the persistent step kernel
// (step_kernel.cu): mma.sync m16n8k16 (bf16 in, fp32 accumulate), ldmatrix
// loads of 128-byte-swizzled rows, fp32 values as bf16 hi + lo pairs, and the
// fed rows' LayerNorm held in registers.  Eight warps (256 threads) share a
// row: warp w holds columns [w K/8, (w + 1) K/8).
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

#include "common.cuh"

namespace mtp {
namespace frag {

constexpr int NWARPS = 8;
constexpr int NTHREADS = NWARPS * 32;

// Synchronisation of the threads that share a row: the whole CTA, or (when a
// CTA also runs a producer warp) named barrier 1 over the 256 consumer threads.
struct CtaSync {
    __device__ __forceinline__ void operator()() const { __syncthreads(); }
};
struct ConsumerSync {
    __device__ __forceinline__ void operator()() const { asm volatile("bar.sync 1, 256;" ::: "memory"); }
};

// ---- tensor-core building blocks ----
// Fed rows are at most 8 tokens: they are the N = 8 side of the MMA and the
// weight rows the M = 16 side, so no token padding beyond 8 is needed.

__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}
// The transpose of the 8 x 8 b16 matrix whose row lane / 4, columns 2 (lane % 4) and + 1, this
// lane holds in r: returns the same elements of the transposed matrix.
__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t r) {
    uint32_t d;
    asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(r));
    return d;
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}
__device__ __forceinline__ void ldsm_x2(uint32_t (&r)[2], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0, %1}, [%2];" : "=r"(r[0]), "=r"(r[1]) : "r"(addr));
}
__device__ __forceinline__ void mma_bf16(float (&d)[4], const uint32_t (&a)[4], const uint32_t (&b)[2]) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

// x0, x1 as bf16 pairs hi + lo with hi + lo = x to about 2^-16 relative
// (low halves hold the first element, as the MMA fragments expect).
__device__ __forceinline__ void split_bf16x2(float x0, float x1, uint32_t& hi, uint32_t& lo) {
    const __nv_bfloat16 h0 = __float2bfloat16_rn(x0), h1 = __float2bfloat16_rn(x1);
    const __nv_bfloat16 l0 = __float2bfloat16_rn(x0 - __bfloat162float(h0));
    const __nv_bfloat16 l1 = __float2bfloat16_rn(x1 - __bfloat162float(h1));
    hi = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
    lo = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
}

// Shared address of 16-byte chunk `chunk` of weight row `row` (row_bytes each):
// the weights are stored with chunk c of global row g at position c ^ (g & 7)
// (made at create), which keeps ldmatrix free of bank conflicts.
__device__ __forceinline__ uint32_t wchunk(uint32_t base, int row, int row_bytes, int chunk, int key) {
    return base + (uint32_t)row * row_bytes + ((uint32_t)(chunk ^ (key & 7)) << 4);
}

// Input rows for a projection: lane holds columns warp*Kw + lane*4 .. +3 of
// each of the MT rows (K <= 1024, one 4-column chunk per lane), LayerNorm'd.
template <int MT>
struct RowRegs {
    float v[MT][4];
};

template <int MT>
__device__ __forceinline__ void load_rows(const float* x, int ld, int M, int K, RowRegs<MT>& r) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int Kw = K / NWARPS;
    const bool valid = lane * 4 < Kw;
#pragma unroll
    for (int m = 0; m < MT; ++m) {
        if (m < M && valid) {
            load4(x + (size_t)m * ld + warp * Kw + lane * 4, r.v[m]);
        } else {
#pragma unroll
            for (int i = 0; i < 4; ++i) r.v[m][i] = 0.f;
        }
    }
}

// Fed rows as bf16 hi and lo parts in shared memory, [MT][K + 8] each (lo
// right after hi; the 16-byte pad spreads banks).
template <int MT>
__device__ __forceinline__ void store_rows_split(const RowRegs<MT>& r, int K, __nv_bfloat16* xb) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int Kw = K / NWARPS;
    if (lane * 4 >= Kw) return;
#pragma unroll
    for (int m = 0; m < MT; ++m) {
        uint2 h, l;
        split_bf16x2(r.v[m][0], r.v[m][1], h.x, l.x);
        split_bf16x2(r.v[m][2], r.v[m][3], h.y, l.y);
        const size_t at = (size_t)m * (K + 8) + warp * Kw + lane * 4;
        *reinterpret_cast<uint2*>(xb + at) = h;
        *reinterpret_cast<uint2*>(xb + (size_t)MT * (K + 8) + at) = l;
    }
}

// LayerNorm of the register rows in place.  Each warp takes the mean and the
// sum of squared deviations of its K/NWARPS columns (two passes over
// registers), and one block reduction merges the warps' equal-sized slices:
// mean = average of the warp means, M2 = sum of warp M2 + Kw * sum (mean_w - mean)^2.
template <int MT, class Sync = CtaSync>
__device__ __forceinline__ void layer_norm_rows(RowRegs<MT>& r, int K, const float (&gam)[4], const float (&bet)[4],
                                                float eps, float (*part)[MT], float (*stat)[MT]) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int Kw = K / NWARPS;
    const bool valid = lane * 4 < Kw;
    float (*pm2)[MT] = part + NWARPS;  // second half of the scratch
#pragma unroll
    for (int m = 0; m < MT; ++m) {
        float s1 = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i) s1 += valid ? r.v[m][i] : 0.f;
        const float mw = warp_sum(s1) / (float)Kw;
        float s2 = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float t = r.v[m][i] - mw;
            s2 += valid ? t * t : 0.f;
        }
        const float m2 = warp_sum(s2);
        if (lane == 0) {
            part[warp][m] = mw;
            pm2[warp][m] = m2;
        }
    }
    Sync()();
    if (threadIdx.x < MT) {
        const int m = threadIdx.x;
        float mean = 0.f;
#pragma unroll
        for (int w = 0; w < NWARPS; ++w) mean += part[w][m];
        mean /= (float)NWARPS;
        float m2 = 0.f;
#pragma unroll
        for (int w = 0; w < NWARPS; ++w) {
            const float dm = part[w][m] - mean;
            m2 += pm2[w][m] + (float)Kw * dm * dm;
        }
        stat[0][m] = mean;
        stat[1][m] = 1.0f / sqrtf(m2 / (float)K + eps);
    }
    Sync()();
#pragma unroll
    for (int m = 0; m < MT; ++m)
#pragma unroll
        for (int i = 0; i < 4; ++i) r.v[m][i] = (r.v[m][i] - stat[0][m]) * stat[1][m] * gam[i] + bet[i];
}

// Column of element dd of key/value row t inside a cached page: the row's
// 16-byte chunks are stored in the order chunk ^ (t & 7), which keeps the
// attention's ldmatrix reads of eight consecutive rows free of bank conflicts.
__device__ __forceinline__ int kv_col(int t, int dd) { return (((dd >> 3) ^ (t & 7)) << 3) | (dd & 7); }


}  // namespace frag
}  // namespace mtp
