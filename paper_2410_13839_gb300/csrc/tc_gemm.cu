// tc_gemm.cu -- tensor-core GEMM of the batched path (the block's
// projections, Sec. III-A, once B * n fed rows make them a dense contraction):
//
//   out[n][f] (+)= sum_k (a_hi[n][k] + a_lo[n][k]) * w[f][k]
//
// w: bf16 weights, K-major ([N_w][K]); a_hi + a_lo: the fp32 activations as
// two bf16 parts, K-major ([M][K]).  The weights are the MMA's M = 128 side
// (one 128-row tile per CTA) and the activation rows its N side (NT per
// tile), so a handful of fed rows still fills the tensor core; both parts of
// the activations go through the same accumulator (two MMAs per k-step),
// which keeps the product to fp32 accuracy.
//
// Per CTA: one elected thread streams 64-wide k-chunks of the weight tile
// and of both activation parts into a 4-stage shared-memory ring with TMA
// (128-byte swizzled tiles), a second elected thread issues tcgen05.mma
// into a TMEM accumulator (128 lanes x NT fp32 columns) and releases each
// stage with tcgen05.commit, and the eight warps read the accumulator back
// with tcgen05.ld (warps w and w + 4 own TMEM lanes 32w..32w+31, i.e. weight
// rows, and take alternate 32-column chunks) and
// store or atomically add it to out.  Grid: (N_w / 128 weight tiles, K
// splits, activation tiles).  The weight copies of the first stages are
// issued before griddepcontrol.wait; the activation copies after it.
#include <cuda.h>

#include <cstdio>
#include <cstring>
#include <mutex>

#include "common.cuh"
#include "kernels.cuh"
#include "mtp.h"
#include "tcgen05.cuh"

namespace mtp {
namespace {

constexpr int TC_M = 128;      // weight rows per CTA (MMA M)
constexpr int TC_K = 64;       // k per stage: one 128-byte swizzle row of bf16
// ring stages per activation tile size: about 190 KB of copies in flight per CTA
__host__ __device__ constexpr int tc_stages(int nt) { return nt <= 32 ? 8 : (nt <= 64 ? 6 : 4); }
constexpr int TC_MAX_STAGES = 8;
// 8 warps: two elected lanes run the ring; in the epilogue warps w and w + 4 share TMEM lane
// quarter w % 4 and take alternate 32-column chunks, and every row loop has twice the threads
// (the epilogue is instruction-latency bound: one warp per scheduler hid nothing)
constexpr int TC_THREADS = 256;
constexpr int TC_MAX_CLUSTER_SPLITS = 8;  // K splits reduced in one (portable) cluster
constexpr uint32_t TC_W_BYTES = TC_M * TC_K * 2;

// ---- PTX wrappers (tcgen05, TMA) ----
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            smem_addr(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar))
        : "memory");
}
// Bulk copy of `bytes` from this CTA's shared memory to shared memory of a CTA of the cluster
// (dst, bar: shared::cluster addresses), completing on that CTA's barrier.  16-byte aligned.
__device__ __forceinline__ void bulk_copy_s2s_cluster(uint32_t dst, uint32_t src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "r"(src), "r"(bytes), "r"(bar)
                 : "memory");
}

// Shared-memory address `saddr` of this CTA mapped to the CTA of cluster rank `rank`.
__device__ __forceinline__ uint32_t mapa_rank(uint32_t saddr, int rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
    return r;
}

// Instruction descriptor of kind::f16: fp32 accumulator, bf16 A and B, both
// K-major, M = 128, N = nt.
__host__ __device__ constexpr uint32_t tc_idesc(int nt) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(nt >> 3) << 17) | ((uint32_t)(TC_M >> 4) << 24);
}

template <int NT, bool PART>
__global__ void __launch_bounds__(TC_THREADS, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tw, const __grid_constant__ CUtensorMap tah,
                   const __grid_constant__ CUtensorMap tal, const TcGemmArgs a) {
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    constexpr uint32_t A_BYTES = NT * TC_K * 2, STAGE = TC_W_BYTES + 2 * A_BYTES;
    constexpr uint32_t TMEM_COLS = NT < 32 ? 32 : NT;
    constexpr int TC_STAGES = tc_stages(NT);
    __shared__ uint64_t full[TC_MAX_STAGES], empty[TC_MAX_STAGES], done, red_bar;
    __shared__ uint32_t tmem_base;
    __shared__ int s_ok;
    __shared__ long long s_rowbase[NT];  // TC_QKV: element offset of the row's key row in its page (-1: none)
    __shared__ int s_rowt[NT];           // TC_QKV: key row within the page; TC_GELU_PACK: row of a sequence
    unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    TraceEnd trace_guard(a.trace);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int tile = blockIdx.x, split = blockIdx.y, ntile = blockIdx.z;
    const int chunks = a.k_chunks;
    const int kc0 = split * chunks;
    const int arow = ntile * NT;

    if (warp == 0) {
        tmem_alloc(&tmem_base, TMEM_COLS);
        tmem_relinquish();
    }
    if (tid == 32) {
        for (int s = 0; s < TC_STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(&done, 1);
        mbar_init(&red_bar, 1);
        fence_barrier_init();
        s_ok = 1;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base;

    // weights of the first stages: independent of the previous kernel
    auto w_coords = [&](int c, int& x, int& y) {
        const int kc = kc0 + c;
        if (a.w_rows_per_kchunk) {  // k-chunk kc is a block of rows (W_o stored per head)
            x = 0;
            y = kc * a.w_rows_per_kchunk + tile * TC_M;
        } else {
            x = kc * TC_K;
            y = tile * TC_M;
        }
    };
    const int pre = chunks < TC_STAGES ? chunks : TC_STAGES;
    if (tid == 0) {
        for (int c = 0; c < pre; ++c) {
            unsigned char* st = smem + (size_t)c * STAGE;
            mbar_arrive_expect_tx(&full[c], STAGE);
            int x, y;
            w_coords(c, x, y);
            tma_load_2d(st, &tw, x, y, &full[c]);
        }
    }
    pdl_launch_dependents();
    pdl_wait();
    trace_wait(a.trace);

    // The elected lanes run the ring; the rest of warps 0 and 1 wait at __syncwarp
    // (not in the barrier poll below, which would hold up their elected lane).
    if (tid == 0) {  // producer: activations of the first stages, then the rest of the ring
        for (int c = 0; c < chunks; ++c) {
            const int s = c % TC_STAGES;
            unsigned char* st = smem + (size_t)s * STAGE;
            if (c >= TC_STAGES) {
                if (!mbar_wait(&empty[s], (uint32_t)((c / TC_STAGES) - 1) & 1, a.err)) {
                    s_ok = 0;
                    break;
                }
                mbar_arrive_expect_tx(&full[s], STAGE);
                int x, y;
                w_coords(c, x, y);
                tma_load_2d(st, &tw, x, y, &full[s]);
            }
            const int kx = (kc0 + c) * TC_K;
            tma_load_2d(st + TC_W_BYTES, &tah, kx, arow, &full[s]);
            tma_load_2d(st + TC_W_BYTES + A_BYTES, &tal, kx, arow, &full[s]);
        }
    } else if (tid == 32) {  // MMA issuer
        constexpr uint32_t IDESC = tc_idesc(NT);
        int c = 0;
        for (; c < chunks; ++c) {
            const int s = c % TC_STAGES;
            if (!mbar_wait(&full[s], (uint32_t)(c / TC_STAGES) & 1, a.err)) break;
            tc_fence_after();
            const uint32_t wb = smem_addr(smem + (size_t)s * STAGE);
            const uint32_t hb = wb + TC_W_BYTES, lb = hb + A_BYTES;
#pragma unroll
            for (int kk = 0; kk < TC_K / 16; ++kk) {
                const uint64_t dw = sw128_desc(wb + kk * 32);
                tc_mma(tmem, dw, sw128_desc(hb + kk * 32), IDESC, (c | kk) != 0);
                tc_mma(tmem, dw, sw128_desc(lb + kk * 32), IDESC, 1u);
            }
            tc_commit(&empty[s]);  // stage s is free once these MMAs have read it
        }
        if (c < chunks) s_ok = 0;
        tc_commit(&done);  // every MMA issued above has completed
    } else if (warp >= 2 && (a.epilogue == TC_QKV || a.epilogue == TC_GELU_PACK)) {
        // per-row facts of the epilogue, gathered by the two idle warps while the ring runs
        for (int j = tid - 64; j < NT; j += TC_THREADS - 64) {
            const int n = arow + j;
            const int seq = n < a.m ? a.row_seq[n] : -1;
            long long base = -1;
            int t = 0;
            if (a.epilogue == TC_QKV && seq >= 0) {
                const int pos = a.row_pos[n];
                t = pos % a.page_size;
                const int page = a.block_table[(size_t)seq * a.bt_stride + pos / a.page_size];
                if (page < 0)
                    atomicOr(a.err, ERR_BOUNDS);
                else
                    base = (long long)page * a.page_elems + a.layer_off + (long long)t * HEAD_DIM;
            }
            s_rowbase[j] = seq >= 0 ? base : -2;  // -2: no sequence
            s_rowt[j] = a.epilogue == TC_QKV ? t : (seq >= 0);
        }
    }
    if (warp < 2) __syncwarp();

    // epilogue: lane = weight row f (TMEM lane of the warp's quarter), 32 activation rows per load
    // one thread polls (a poll costs each polling thread, even on a completed phase); the block
    // barrier hands the result to the others
    const bool fin = __syncthreads_and(tid == 0 ? mbar_wait(&done, 0, a.err) : true) != 0;
    tc_fence_after();
    trace_mark(a.trace, 0);  // accumulator complete
    // K splits reduced in a cluster: Sc consecutive splits of this tile are one cluster; each
    // stages its partial tile, then sums one Sc-th of the activation rows over the cluster's tiles
    // (DSMEM) and runs the epilogue on those rows only.  Clusters of the same tile (TC_ACCUM with
    // more splits than one cluster holds) still add their sums with atomics.
    const int Sc = a.cluster_reduce > 1 ? a.cluster_reduce : 1;
    const bool creduce = Sc > 1;
    const int rank = split % Sc;
    const bool good = fin && s_ok;
    constexpr int TP = TC_M + 4;  // row pitch of the staged tile (floats)
    float* T = reinterpret_cast<float*>(smem);
    if (good) {
        // accumulator -> shared tile T[n][f] (the stages are free: every MMA has read them)
        const int quarter = warp & 3;  // the TMEM lanes (weight rows) this warp may read
        for (int j0 = (warp >> 2) * 32; j0 < NT; j0 += (TC_THREADS / 128) * 32) {
            float v[32];
            tmem_ld32(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)j0, v);
#pragma unroll
            for (int j = 0; j < 32; ++j) T[(j0 + j) * TP + quarter * 32 + lane] = v[j];
        }
    }
    trace_mark(a.trace, 1);  // thread 0's rows staged
    int jbeg = 0, jend = NT;  // activation rows of the tile this CTA finishes
    if (creduce) {
        // each CTA pushes the rows that another CTA finishes to that CTA (one bulk copy per peer,
        // completing on the receiver's barrier), then sums the Sc partial copies of its own rows
        jbeg = rank * NT / Sc;
        jend = (rank + 1) * NT / Sc;
        const uint32_t seg = (uint32_t)(NT / Sc) * TP * 4;  // bytes of one CTA's share of rows
        float* recv = T + (size_t)NT * TP;                  // [Sc][NT / Sc][TP]: slot = sender's rank
        if (tid == 0) mbar_arrive_expect_tx(&red_bar, seg * (uint32_t)(Sc - 1));
        __syncthreads();
        cluster_arrive_release();  // every split's partial tile is staged and every receiver armed
        cluster_wait();
        trace_mark(a.trace, 2);  // the cluster's tiles staged
        if (tid < Sc - 1 && good) {  // one copy per issuing thread
            fence_proxy_async();  // the tile was written by this CTA's threads
            const int p = (rank + 1 + tid) % Sc;
            bulk_copy_s2s_cluster(mapa_rank(smem_addr(recv + (size_t)rank * (NT / Sc) * TP), p),
                                  smem_addr(T + (size_t)p * (NT / Sc) * TP), seg, mapa_rank(smem_addr(&red_bar), p));
        }
        const bool got = __syncthreads_and(tid == 0 ? mbar_wait(&red_bar, 0, a.err) : true) != 0;
        trace_mark(a.trace, 3);  // the peers' partial rows received
        if (good && got) {
            for (int i = tid; i < (jend - jbeg) * (TC_M / 4); i += TC_THREADS) {
                const int jl = i / (TC_M / 4), f4 = (i % (TC_M / 4)) * 4;
                float* t = T + (size_t)(jbeg + jl) * TP + f4;
                float4 part[TC_MAX_CLUSTER_SPLITS];
#pragma unroll
                for (int src = 0; src < TC_MAX_CLUSTER_SPLITS; ++src)  // every partial loaded before any is added
                    if (src < Sc)
                        part[src] = *reinterpret_cast<const float4*>(
                            src == rank ? t : recv + ((size_t)src * (NT / Sc) + jl) * TP + f4);
                float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int src = 0; src < TC_MAX_CLUSTER_SPLITS; ++src) {  // every split's partial, in rank order
                    if (src >= Sc) continue;
                    acc.x += part[src].x;
                    acc.y += part[src].y;
                    acc.z += part[src].z;
                    acc.w += part[src].w;
                }
                *reinterpret_cast<float4*>(t) = acc;
            }
        }
        if (!got) s_ok = 0;
        cluster_arrive_relaxed();  // this CTA's pushes have landed (waited for before leaving)
    }
    __syncthreads();
    trace_mark(a.trace, 4);  // rows to finish summed
    if (good && s_ok) {
        // float4 rows of T -> out, coalesced
        const int rows = min(NT, a.m - arow);
        const bool add_bias = a.bias && split < Sc;  // the tile's first cluster (or split 0) adds it
        const int P = a.page_size, H = a.n_heads, d = H * HEAD_DIM;
        const int j1 = min(jend, rows);
        if constexpr (PART) {  // TC_ACCUM of features < n_valid only, element atomics (rows of any pitch)
            for (int i = tid; i < (j1 - jbeg) * TC_M; i += TC_THREADS) {
                const int j = jbeg + i / TC_M, fl = i % TC_M, f = tile * TC_M + fl;
                if (f < a.n_valid)
                    atomicAdd(a.out + (size_t)(arow + j) * a.ldo + f, T[j * TP + fl] + (add_bias ? a.bias[f] : 0.f));
            }
        } else {
        // every item of this thread has the same 4 features (TC_THREADS is a multiple of TC_M / 4):
        // their bias is read once, ahead of the stores
        static_assert(TC_THREADS % (TC_M / 4) == 0, "one feature quad per thread");
        float4 bq = make_float4(0.f, 0.f, 0.f, 0.f);
        if (add_bias) {
            const int f = tile * TC_M + (tid % (TC_M / 4)) * 4;
            bq = make_float4(__ldg(a.bias + f), __ldg(a.bias + f + 1), __ldg(a.bias + f + 2), __ldg(a.bias + f + 3));
        }
        for (int i = tid; i < (j1 - jbeg) * (TC_M / 4); i += TC_THREADS) {
            const int j = jbeg + i / (TC_M / 4), f4 = (i % (TC_M / 4)) * 4;
            const int f = tile * TC_M + f4, n = arow + j;
            float4 y = *reinterpret_cast<const float4*>(T + j * TP + f4);
            y.x += bq.x;
            y.y += bq.y;
            y.z += bq.z;
            y.w += bq.w;
            if (a.epilogue == TC_ACCUM) {
                atomicAdd(reinterpret_cast<float4*>(a.out + (size_t)n * a.ldo + f), y);
            } else if (a.epilogue == TC_STORE) {
                *reinterpret_cast<float4*>(a.out + (size_t)n * a.ldo + f) = y;
            } else if (a.epilogue == TC_QKV) {  // features h*192 + {q,k,v}*64 + dd
                const long long base = s_rowbase[j];
                if (base == -2) continue;  // no sequence
                const int h = f / (3 * HEAD_DIM), sec = (f / HEAD_DIM) % 3, dd = f % HEAD_DIM;
                if (sec == 0) {
                    *reinterpret_cast<float4*>(a.out + (size_t)n * d + h * HEAD_DIM + dd) = y;
                    continue;
                }
                if (base < 0) continue;  // unreserved page (reported)
                const int t = s_rowt[j];
                const long long idx = base + (long long)(sec - 1) * H * P * HEAD_DIM + (long long)h * P * HEAD_DIM +
                                      ((((dd >> 3) ^ (t & 7)) << 3) | (dd & 7));
                uint2 pk;
                pk.x = (uint32_t)f32_to_bf16_bits(y.x) | ((uint32_t)f32_to_bf16_bits(y.y) << 16);
                pk.y = (uint32_t)f32_to_bf16_bits(y.z) | ((uint32_t)f32_to_bf16_bits(y.w) << 16);
                *reinterpret_cast<uint2*>(reinterpret_cast<uint16_t*>(a.kv_pool) + idx) = pk;
            } else {  // TC_GELU_PACK
                const bool on = s_rowt[j] != 0;
                const float v[4] = {on ? gelu_erf(y.x) : 0.f, on ? gelu_erf(y.y) : 0.f, on ? gelu_erf(y.z) : 0.f,
                                    on ? gelu_erf(y.w) : 0.f};
                uint32_t hi[2], lo[2];
#pragma unroll
                for (int q = 0; q < 2; ++q) {
                    const __nv_bfloat16 h0 = __float2bfloat16_rn(v[2 * q]), h1 = __float2bfloat16_rn(v[2 * q + 1]);
                    const __nv_bfloat16 l0 = __float2bfloat16_rn(v[2 * q] - __bfloat162float(h0));
                    const __nv_bfloat16 l1 = __float2bfloat16_rn(v[2 * q + 1] - __bfloat162float(h1));
                    hi[q] = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
                    lo[q] = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
                }
                *reinterpret_cast<uint2*>(a.pack_hi + (size_t)n * a.ldo + f) = make_uint2(hi[0], hi[1]);
                *reinterpret_cast<uint2*>(a.pack_lo + (size_t)n * a.ldo + f) = make_uint2(lo[0], lo[1]);
            }
        }
        }
        trace_mark(a.trace, 5);  // thread 0's stores issued
    } else if (!fin) {
        // the MMAs may still be running: wait for them (bounded) before freeing TMEM
        mbar_wait(&done, 0, nullptr);
    }
    if (creduce) cluster_wait();  // the peers are done with this CTA's tile
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, TMEM_COLS);
}

// ---- tensor maps ----
using EncodeTiled = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                 const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                 CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiled encode_fn() {
    static EncodeTiled fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiled>(p);
    });
    return fn;
}

template <int NT>
size_t tc_smem() {
    return (size_t)tc_stages(NT) * (TC_W_BYTES + 2u * NT * TC_K * 2) + 1024;
}

template <int NT, typename K>
cudaError_t launch_kern(K kern, const TcGemm& g, cudaStream_t s, bool pdl) {
    const size_t smem = tc_smem<NT>();
    cudaError_t e = ensure_kernel_smem(reinterpret_cast<const void*>(kern), smem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(g.n_w / TC_M, g.splits, (g.args.m + NT - 1) / NT);
    cfg.blockDim = dim3(TC_THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (g.args.cluster_reduce > 1) {  // consecutive K splits of a tile form one cluster
        attr[1].id = cudaLaunchAttributeClusterDimension;
        attr[1].val.clusterDim.x = 1;
        attr[1].val.clusterDim.y = g.args.cluster_reduce;
        attr[1].val.clusterDim.z = 1;
        cfg.numAttrs = 2;
    }
    return cudaLaunchKernelEx(&cfg, kern, g.w, g.a_hi, g.a_lo, g.args);
}

template <int NT>
cudaError_t launch_nt(const TcGemm& g, cudaStream_t s, bool pdl) {
    if (g.args.n_valid) return launch_kern<NT>(tc_gemm_kernel<NT, true>, g, s, pdl);
    return launch_kern<NT>(tc_gemm_kernel<NT, false>, g, s, pdl);
}

}  // namespace

int tc_encode_2d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows, uint32_t box_rows,
                 bool pre_swizzled) {
    EncodeTiled fn = encode_fn();
    if (!fn) return -1;
    if ((reinterpret_cast<uintptr_t>(base) & 15) || (inner * 2) % 16 || box_rows == 0 || box_rows > 256) return -2;
    const cuuint64_t dims[2] = {inner, rows};
    const cuuint64_t strides[1] = {inner * 2};
    const cuuint32_t box[2] = {(cuuint32_t)TC_K, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    // pre-swizzled tensors already hold chunk c of row r at c ^ (r & 7): copy them verbatim
    const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE,
                          pre_swizzled ? CU_TENSOR_MAP_SWIZZLE_NONE : CU_TENSOR_MAP_SWIZZLE_128B,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? 0 : -3;
}

int tc_tile_rows(int m) { return m <= 32 ? 32 : (m <= 64 ? 64 : 128); }

cudaError_t launch_tc_gemm(const TcGemm& g, cudaStream_t s, bool pdl) {
    if (g.n_w % TC_M || g.args.k_chunks < 1 || g.splits < 1 || g.args.m < 1) return cudaErrorInvalidValue;
    const int sc = g.args.cluster_reduce > 1 ? g.args.cluster_reduce : 1;
    if (sc > TC_MAX_CLUSTER_SPLITS || g.splits % sc) return cudaErrorInvalidValue;
    if (g.args.epilogue != TC_ACCUM && g.splits != sc) return cudaErrorInvalidValue;  // one cluster finishes a tile
    switch (g.nt) {
        case 32: return launch_nt<32>(g, s, pdl);
        case 64: return launch_nt<64>(g, s, pdl);
        case 128: return launch_nt<128>(g, s, pdl);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace mtp

using namespace mtp;

namespace {
int gemm_fail(int code, const char* fmt, int a = 0, int b = 0, int c = 0, int d = 0, int e = 0) {
    char buf[256];
    snprintf(buf, sizeof(buf), fmt, a, b, c, d, e);
    return report_error(code, buf);
}
}  // namespace

extern "C" MTP_API int mtp_gemm_bf16x2(const void* w, const void* a_hi, const void* a_lo, float* out, int n_w, int k,
                                       int m, int splits, int accumulate, void* stream) {
    clear_error();
    if (!w || !a_hi || !a_lo || !out) return gemm_fail(MTP_ERR_INVALID, "mtp_gemm_bf16x2: null pointer");
    if (n_w < TC_M || n_w % TC_M || k < TC_K || k % TC_K || m < 1 || m > 4096 || splits < 1 ||
        (k / TC_K) % splits || (!accumulate && splits != 1))
        return gemm_fail(MTP_ERR_INVALID, "mtp_gemm_bf16x2: n_w=%d k=%d m=%d splits=%d accumulate=%d", n_w, k, m,
                         splits, accumulate);
    TcGemm g;
    std::memset(&g, 0, sizeof(g));
    g.n_w = n_w;
    g.splits = splits;
    g.nt = tc_tile_rows(m);
    g.args.out = out;
    g.args.ldo = n_w;
    g.args.bias = nullptr;
    g.args.m = m;
    g.args.k_chunks = k / TC_K / splits;
    g.args.w_rows_per_kchunk = 0;
    g.args.epilogue = accumulate ? TC_ACCUM : TC_STORE;
    int* d_err = nullptr;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (cudaMallocAsync(&d_err, sizeof(int), st) != cudaSuccess)
        return gemm_fail(MTP_ERR_CUDA, "mtp_gemm_bf16x2: error word allocation failed");
    cudaMemsetAsync(d_err, 0, sizeof(int), st);
    g.args.err = d_err;
    int rc = 0;
    if (tc_encode_2d(&g.w, w, (uint64_t)k, (uint64_t)n_w, TC_M, false) ||
        tc_encode_2d(&g.a_hi, a_hi, (uint64_t)k, (uint64_t)m, (uint32_t)g.nt, false) ||
        tc_encode_2d(&g.a_lo, a_lo, (uint64_t)k, (uint64_t)m, (uint32_t)g.nt, false)) {
        rc = gemm_fail(MTP_ERR_INVALID, "mtp_gemm_bf16x2: tensor map encoding failed (alignment?)");
    } else {
        const cudaError_t e = launch_tc_gemm(g, st, false);
        if (e != cudaSuccess) rc = report_error(MTP_ERR_CUDA, cudaGetErrorString(e));
    }
    int h_err = 0;
    cudaMemcpyAsync(&h_err, d_err, sizeof(int), cudaMemcpyDeviceToHost, st);
    const cudaError_t es = cudaStreamSynchronize(st);
    cudaFreeAsync(d_err, st);
    if (rc) return rc;
    if (es != cudaSuccess) return report_error(MTP_ERR_CUDA, cudaGetErrorString(es));
    if (h_err) return gemm_fail(MTP_ERR_DEVICE, "mtp_gemm_bf16x2: device error word 0x%x", h_err);
    return MTP_OK;
}
