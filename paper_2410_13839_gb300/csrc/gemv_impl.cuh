// gemv_impl.cuh -- weight-streaming projection for up to 8 rows (the per-layer
// linear layers of the decode step and the MTP heads, Sec. III-A/B).
//
// At B * n <= 8 rows a projection moves K * N weights and does 2 * M flops per
// weight: it is bound by HBM bandwidth, not by the tensor cores.  Design:
//   * one CTA per SM-sized slice of output features; the slice's weight rows
//     are contiguous and land in shared memory through cp.async.bulk (TMA 1-D)
//     issued before griddepcontrol.wait, so under programmatic dependent
//     launch the weights stream in while the previous kernel still runs;
//   * warp w owns a fixed K-slice; each lane keeps its 4 (or 8) input columns
//     of all M rows in registers, LayerNorm applied in the prologue;
//   * 32 partial dot products per lane (G rows x M inputs) are combined with a
//     31-shuffle reduce-scatter, then across warps through shared memory in a
//     fixed order (deterministic);
//   * fused epilogues: bias + q / key-value append into the paged cache,
//     bias + residual add (+ copy of a slot's last hidden state), bias + GELU,
//     bias (head logits).
#pragma once

#include "common.cuh"
#include "kernels.cuh"

namespace mtp {
namespace gemv_detail {

constexpr uint32_t BULK_CHUNK = 32768;

// Sum v[i] over the 32 lanes for every i; lane l returns the total of v[l].
__device__ __forceinline__ float reduce_scatter32(float (&v)[32], int lane) {
#pragma unroll
    for (int width = 16; width >= 1; width >>= 1) {
        const bool upper = (lane & width) != 0;
#pragma unroll
        for (int i = 0; i < width; ++i) {
            const float send = upper ? v[i] : v[i + width];
            const float keep = upper ? v[i + width] : v[i];
            v[i] = keep + __shfl_xor_sync(FULL_MASK, send, width);
        }
    }
    return v[0];
}

template <typename WT, int MT, int WARPS, int NSUB, int EPI, bool LN>
__global__ void __launch_bounds__(WARPS * 32, 2) gemv_kernel(const GemvArgs a) {
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ uint64_t bar;
    __shared__ float ln_part[WARPS][MT];
    __shared__ float ln_stat[2][MT];
    __shared__ int s_seq[MT], s_pos[MT], s_last[MT], s_page[MT];
    constexpr int G = 32 / MT;           // weight rows per reduce-scatter group
    constexpr int NT = WARPS * 32;
    constexpr bool XSMEM = NSUB > 1;     // wide inputs are staged in shared memory
    TraceEnd trace_guard(a.trace);

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int r0 = blockIdx.x * a.rows_per_cta;
    const int R = min(a.rows_per_cta, a.N - r0);
    const int K = a.K;
    const size_t wbytes = R > 0 ? (size_t)R * K * sizeof(WT) : 0;
    const size_t wpad = ((size_t)a.rows_per_cta * K * sizeof(WT) + 127) & ~(size_t)127;
    const WT* wsm = reinterpret_cast<const WT*>(smem);
    const int ngroups = (max(R, 0) + G - 1) / G;
    float* red = reinterpret_cast<float*>(smem + wpad);                   // [WARPS][ngroups * 32]
    float* xs = red + (size_t)WARPS * ((a.rows_per_cta + G - 1) / G) * 32;  // [MT][K] when XSMEM

    if (tid == 0) {
        mbar_init(&bar, 1);
        fence_barrier_init();
    }
    __syncthreads();
    if (tid == 0 && wbytes > 0) {
        mbar_arrive_expect_tx(&bar, (uint32_t)wbytes);
        const char* src = reinterpret_cast<const char*>(a.W) + (size_t)r0 * K * sizeof(WT);
        const uint64_t pol = l2_evict_first_policy();
        for (size_t off = 0; off < wbytes; off += BULK_CHUNK)
            bulk_copy_g2s_hint(smem + off, src + off, (uint32_t)min((size_t)BULK_CHUNK, wbytes - off), &bar, pol);
    }

    // ---- parameters (weights): read before the wait ----
    const int Kw = K / WARPS;  // columns of this warp
    float gam[XSMEM ? 1 : NSUB][4], bet[XSMEM ? 1 : NSUB][4];
    if (LN && !XSMEM) {
#pragma unroll
        for (int s = 0; s < NSUB; ++s) {
            const int c = s * 32 + lane;
            if (c * 4 < Kw) {
                load4(a.ln_g + warp * Kw + c * 4, gam[s]);
                load4(a.ln_b + warp * Kw + c * 4, bet[s]);
            } else {
#pragma unroll
                for (int i = 0; i < 4; ++i) gam[s][i] = bet[s][i] = 0.f;
            }
        }
    }
    float bias_r[2];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
        const int o = tid + u * NT;
        bias_r[u] = (o < R * MT) ? __ldg(a.bias + r0 + o / MT) : 0.f;
    }

    pdl_launch_dependents();
    pdl_wait();
    trace_wait(a.trace);

    // ---- inputs of this launch (written by the previous kernel) ----
    if (tid < MT) {
        const bool in = tid < a.M;
        s_seq[tid] = (in && a.row_seq) ? a.row_seq[tid] : (in ? 0 : -1);
        if (EPI == EPI_QKV || EPI == EPI_RESID) {
            s_pos[tid] = (in && a.row_pos) ? a.row_pos[tid] : -1;
            s_last[tid] = (in && a.row_last) ? a.row_last[tid] : 0;
        }
    }
    float xv[MT][XSMEM ? 1 : NSUB][4];
    const float* xrow[MT];
#pragma unroll
    for (int m = 0; m < MT; ++m) {  // input row m, or the slot's last fed row of this step
        xrow[m] = a.A + (size_t)m * a.lda;
        if (a.gather_x != nullptr && m < a.M) {
            const int np = a.gather_npend[a.gather_base + m];
            if (np > 0) xrow[m] = a.gather_x + (size_t)(m * a.gather_n + np - 1) * a.lda;
        }
    }
    if (!XSMEM) {
#pragma unroll
        for (int m = 0; m < MT; ++m)
#pragma unroll
            for (int s = 0; s < (XSMEM ? 1 : NSUB); ++s) {
                const int c = s * 32 + lane;
                if (m < a.M && c * 4 < Kw) {
                    load4(xrow[m] + warp * Kw + c * 4, xv[m][s]);
                } else {
#pragma unroll
                    for (int i = 0; i < 4; ++i) xv[m][s][i] = 0.f;
                }
            }
    } else {
        for (int i = tid; i < MT * (K / 4); i += NT) {
            const int m = i / (K / 4), c = i % (K / 4);
            float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
            if (m < a.M) v = *reinterpret_cast<const float4*>(xrow[m] + c * 4);
            *reinterpret_cast<float4*>(xs + (size_t)m * K + c * 4) = v;
        }
    }
    __syncthreads();
    if (EPI == EPI_QKV && tid < MT) {  // page of each row's key/value slot; used in the epilogue
        const int seq = s_seq[tid], pos = s_pos[tid];
        s_page[tid] = (seq >= 0 && pos >= 0) ? a.block_table[(size_t)seq * a.bt_stride + pos / a.page_size] : -1;
    }

    if (LN) {
        // mean, then variance of (x - mean), each a reduction in fixed order
#pragma unroll
        for (int pass = 0; pass < 2; ++pass) {
            if (!XSMEM) {
#pragma unroll
                for (int m = 0; m < MT; ++m) {
                    float part = 0.f;
#pragma unroll
                    for (int s = 0; s < (XSMEM ? 1 : NSUB); ++s) {
                        const bool valid = (s * 32 + lane) * 4 < Kw;
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const float t = pass == 0 ? xv[m][s][i] : xv[m][s][i] - ln_stat[0][m];
                            part += valid ? (pass == 0 ? t : t * t) : 0.f;
                        }
                    }
                    part = warp_sum(part);
                    if (lane == 0) ln_part[warp][m] = part;
                }
            } else {
#pragma unroll
                for (int m = 0; m < MT; ++m) {
                    float part = 0.f;
                    for (int e = 0; e < Kw; e += 128) {
                        const int kk = warp * Kw + e + lane * 4;
                        if (e + lane * 4 < Kw) {
#pragma unroll
                            for (int i = 0; i < 4; ++i) {
                                const float t = pass == 0 ? xs[(size_t)m * K + kk + i]
                                                          : xs[(size_t)m * K + kk + i] - ln_stat[0][m];
                                part += pass == 0 ? t : t * t;
                            }
                        }
                    }
                    part = warp_sum(part);
                    if (lane == 0) ln_part[warp][m] = part;
                }
            }
            __syncthreads();
            if (tid < MT) {
                float tot = 0.f;
#pragma unroll
                for (int w = 0; w < WARPS; ++w) tot += ln_part[w][tid];
                tot /= (float)K;
                ln_stat[pass][tid] = pass == 0 ? tot : 1.0f / sqrtf(tot + a.ln_eps);
            }
            __syncthreads();
        }
        if (!XSMEM) {
#pragma unroll
            for (int m = 0; m < MT; ++m)
#pragma unroll
                for (int s = 0; s < (XSMEM ? 1 : NSUB); ++s)
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        xv[m][s][i] = (xv[m][s][i] - ln_stat[0][m]) * ln_stat[1][m] * gam[s][i] + bet[s][i];
        } else {
            for (int i = tid; i < MT * K; i += NT) {
                const int m = i / K, k = i % K;
                xs[i] = (xs[i] - ln_stat[0][m]) * ln_stat[1][m] * a.ln_g[k] + a.ln_b[k];
            }
            __syncthreads();
        }
    }

    if (wbytes == 0) return;
    bool ok = mbar_wait(&bar, 0, a.err);
    ok = __syncthreads_and(ok) != 0;
    if (!ok) {
        mbar_wait(&bar, 0, nullptr);  // let copies in flight land before leaving
        return;
    }

    // ---- dot products: 32 partial sums per lane per group ----
    for (int g = 0; g < ngroups; ++g) {
        float acc[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) acc[i] = 0.f;
#pragma unroll
        for (int s = 0; s < NSUB; ++s) {
            const int c = s * 32 + lane;
            if (c * 4 < Kw) {
                const int k = warp * Kw + c * 4;
                float xr[MT][4];
#pragma unroll
                for (int m = 0; m < MT; ++m) {
                    if (XSMEM) {
                        const float4 v = *reinterpret_cast<const float4*>(xs + (size_t)m * K + k);
                        xr[m][0] = v.x; xr[m][1] = v.y; xr[m][2] = v.z; xr[m][3] = v.w;
                    } else {
#pragma unroll
                        for (int i = 0; i < 4; ++i) xr[m][i] = xv[m][XSMEM ? 0 : s][i];
                    }
                }
#pragma unroll
                for (int r = 0; r < G; ++r) {
                    const int row = g * G + r;
                    if (row < R) {
                        float w[4];
                        load4(wsm + (size_t)row * K + k, w);
#pragma unroll
                        for (int m = 0; m < MT; ++m) {
                            float t = acc[r * MT + m];
                            t = fmaf(w[0], xr[m][0], t);
                            t = fmaf(w[1], xr[m][1], t);
                            t = fmaf(w[2], xr[m][2], t);
                            t = fmaf(w[3], xr[m][3], t);
                            acc[r * MT + m] = t;
                        }
                    }
                }
            }
        }
        const float v = reduce_scatter32(acc, lane);
        red[warp * (ngroups * 32) + g * 32 + lane] = v;
    }
    __syncthreads();

    // ---- epilogue: output o = row * MT + m ----
    for (int o = tid; o < R * MT; o += NT) {
        const int row = o / MT, m = o - row * MT;
        if (m >= a.M) continue;
        float y = 0.f;
#pragma unroll
        for (int w = 0; w < WARPS; ++w) y += red[w * (ngroups * 32) + o];
        const int f = r0 + row;
        y += o < NT ? bias_r[0] : o < 2 * NT ? bias_r[1] : __ldg(a.bias + f);
        const bool active = s_seq[m] >= 0;
        if (EPI == EPI_QKV) {
            const int d = a.d_model;
            if (f < d) {
                a.out[(size_t)m * a.ldo + f] = y;
            } else if (active) {
                const int sec = f / d;  // 1 = key, 2 = value
                const int within = f - sec * d;
                const int head = within / HEAD_DIM, dd = within % HEAD_DIM;
                const int pos = s_pos[m], page = s_page[m];
                if (page < 0) {
                    atomicOr(a.err, ERR_BOUNDS);
                    continue;
                }
                const long long idx = (long long)page * a.page_elems + a.layer_off +
                                      ((long long)(sec - 1) * a.n_heads + head) * a.page_size * HEAD_DIM +
                                      (long long)(pos % a.page_size) * HEAD_DIM + dd;
                a.kv_pool[idx] = f32_to_bf16_bits(y);
            }
        } else if (EPI == EPI_RESID) {
            if (active) {
                const float x = a.out[(size_t)m * a.ldo + f] + y;
                a.out[(size_t)m * a.ldo + f] = x;
                if (a.h_last != nullptr && s_last[m]) a.h_last[(size_t)s_seq[m] * a.ld_h + f] = x;
            }
        } else if (EPI == EPI_GELU) {
            a.out[(size_t)m * a.ldo + f] = gelu_erf(y);
        } else {
            a.out[(size_t)m * a.ldo + f] = y;
        }
    }
}

template <typename WT, int MT, int WARPS, int NSUB, int EPI, bool LN>
cudaError_t launch_one(const GemvArgs& a, int grid, size_t smem, cudaStream_t s, bool pdl) {
    auto kern = gemv_kernel<WT, MT, WARPS, NSUB, EPI, LN>;
    cudaError_t e = ensure_kernel_smem(reinterpret_cast<const void*>(kern), 200 * 1024);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(WARPS * 32);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, a);
}

template <typename WT, int MT, int WARPS, int NSUB>
cudaError_t dispatch_epi(const GemvArgs& a, int epi, int grid, size_t smem, cudaStream_t s, bool pdl) {
    switch (epi) {
        case EPI_QKV: return launch_one<WT, MT, WARPS, NSUB, EPI_QKV, true>(a, grid, smem, s, pdl);
        case EPI_RESID: return launch_one<WT, MT, WARPS, NSUB, EPI_RESID, false>(a, grid, smem, s, pdl);
        case EPI_GELU: return launch_one<WT, MT, WARPS, NSUB, EPI_GELU, true>(a, grid, smem, s, pdl);
        case EPI_LOGITS: return launch_one<WT, MT, WARPS, NSUB, EPI_LOGITS, true>(a, grid, smem, s, pdl);
    }
    return cudaErrorInvalidValue;
}

template <typename WT, int MT>
cudaError_t dispatch_k(const GemvArgs& a, int epi, int grid, size_t smem, cudaStream_t s, bool pdl) {
    if (a.K <= 1024) return dispatch_epi<WT, MT, 8, 1>(a, epi, grid, smem, s, pdl);
    return dispatch_epi<WT, MT, 8, 4>(a, epi, grid, smem, s, pdl);
}

template <typename WT>
cudaError_t dispatch(const GemvArgs& a, int epi, int grid, size_t smem, cudaStream_t s, bool pdl) {
    if (a.M <= 1) return dispatch_k<WT, 1>(a, epi, grid, smem, s, pdl);
    if (a.M <= 2) return dispatch_k<WT, 2>(a, epi, grid, smem, s, pdl);
    if (a.M <= 4) return dispatch_k<WT, 4>(a, epi, grid, smem, s, pdl);
    return dispatch_k<WT, 8>(a, epi, grid, smem, s, pdl);
}

}  // namespace gemv_detail
}  // namespace mtp
