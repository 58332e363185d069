// heads_tc.cu -- the n prediction heads fused with their log-softmax and
// top-k on the tensor cores (Sec. III-B: head i scores z W_i^T + b_i, z =
// LN_f(h), and its k best tokens become the candidates of lattice position i),
// one pass over the head weights, logits kept on chip.
//
// Grid (8 vocabulary slices, n heads, tiles of 128 rows), 256 threads; the 8 slices of one
// (tile, head) form a thread-block cluster.  Slice j holds the head's vocabulary
// rows [128 j, 128 j + 128) (slice 7 up to V, at most 137 rows).  Per CTA:
//
//   D = (Z_hi + Z_lo) W_slice^T      tcgen05.mma, M = 128 rows (TMEM lanes),
//                                    N = 128 or 144 vocabulary columns, K = d
//                                    in 64-wide chunks through a 4-stage TMA
//                                    ring (128-byte swizzled tiles)
//   phase 1   thread = (row, half of the columns), one pass: max, sum of exp,
//             sum and sum of squares of the logits (logit = D + b, read back
//             from TMEM), the two halves combined in shared memory; the 8
//             slices' values are merged over DSMEM in slice order, so every CTA
//             of the cluster holds the same lse = M + log sum_j s_j exp(m_j - M)
//             and the row's mean and sd
//   phase 2   logp = logit - lse (one fp32 subtraction); the candidates are
//             logp >= T, T = mean + z sd - lse with z such that a normal row
//             would have about 4k + 16 of them; each half's best KM candidates
//             by (logp desc, id asc), kept sorted in registers, merged into the
//             slice's list, which goes to the CTA that owns the row (16 rows per
//             CTA) in its shared memory
//   merge     the owner merges the 8 sorted lists into the row's top-k (8 lanes
//             per row, one per list, a shuffle arg-max per step); if any
//             row of the tile had fewer than k candidates in all, the cluster
//             runs phase 2 again with no threshold
//
// Ranking on logp after the lse is known (not on the logits) keeps the
// candidates exactly those of a top-k over the logp row, equal values
// included.  Logits go to memory only when the caller asks for them.
#include <cuda.h>

#include <algorithm>
#include <cmath>
#include <cstring>

#include "common.cuh"
#include "kernels.cuh"
#include "tcgen05.cuh"

namespace mtp {
namespace {

constexpr int HT_M = 128;        // rows per tile (MMA M, TMEM lanes)
constexpr int HT_K = 64;         // k per stage
constexpr int HT_SLICES = 8;     // vocabulary slices per head (cluster size)
constexpr int HT_SLICE = 128;    // vocabulary rows of slices 0..6
constexpr int HT_NMAX = 144;     // N of the last slice (up to 137 rows)
constexpr int HT_THREADS = 256;  // two warps per TMEM lane quarter (halves of the columns)
constexpr int HT_STAGES = 4;
constexpr int HT_ROWS_PER_OWNER = HT_M / HT_SLICES;  // rows whose merge each CTA of the cluster does
constexpr uint32_t HT_A_BYTES = HT_M * HT_K * 2;
constexpr uint32_t HT_B_BYTES = HT_NMAX * HT_K * 2;
constexpr uint32_t HT_STAGE = 2 * HT_A_BYTES + HT_B_BYTES;  // multiple of 1024
constexpr uint32_t HT_SMEM = HT_STAGES * HT_STAGE + 1024;
constexpr uint32_t HT_TMEM_COLS = 256;
// after the MMAs the ring is free: the candidate lists pushed by the cluster (at most
// 2 x 16 rows x 8 slices x 32 entries x 4 B = 32 KB), each thread's staging row of 33 floats,
// then the logit rows (128 x 137 floats, phase 1) or the two halves' lists (phase 2)
constexpr uint32_t HT_STAGING = 32 * 1024;
constexpr uint32_t HT_LOGIT_STAGE = 68 * 1024;
constexpr uint32_t HT_HALF_LISTS = 68 * 1024;
constexpr int HT_LOGIT_PITCH = 137;
static_assert(HT_STAGING + HT_THREADS * 33 * 4 <= HT_LOGIT_STAGE, "staging rows");
static_assert(HT_LOGIT_STAGE + HT_M * HT_LOGIT_PITCH * 4 <= HT_STAGES * HT_STAGE, "logit rows fit the ring");
static_assert(HT_HALF_LISTS + 2 * HT_M * 32 * 8 <= HT_STAGES * HT_STAGE, "half lists fit the ring");

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            smem_addr(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar))
        : "memory");
}

__device__ __forceinline__ int ld_dsmem_i32(uint32_t addr) {
    int v;
    asm volatile("ld.shared::cluster.s32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
    return v;
}

__device__ __forceinline__ void st_dsmem4(uint32_t addr, float4 v) {
    asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(v.x), "f"(v.y), "f"(v.z),
                 "f"(v.w)
                 : "memory");
}

// Insert (v, id) into the sorted list (value desc; an equal value already in the
// list, which has the lower id, stays first); the caller checked that v beats
// the last entry.  v takes the last place and moves up past every entry it beats.
template <int KM>
__device__ __forceinline__ void topk_insert(float (&val)[KM], int (&ids)[KM], float v, int id) {
    val[KM - 1] = v;
    ids[KM - 1] = id;
#pragma unroll
    for (int q = KM - 1; q > 0; --q) {
        if (val[q] > val[q - 1]) {
            const float tv = val[q];
            val[q] = val[q - 1];
            val[q - 1] = tv;
            const int ti = ids[q];
            ids[q] = ids[q - 1];
            ids[q - 1] = ti;
        }
    }
}

template <int KM>
__global__ void __cluster_dims__(HT_SLICES, 1, 1) __launch_bounds__(HT_THREADS, 1)
    heads_tc_kernel(const __grid_constant__ CUtensorMap tw128, const __grid_constant__ CUtensorMap tw144,
                    const __grid_constant__ CUtensorMap tah, const __grid_constant__ CUtensorMap tal,
                    const HeadsTcArgs a) {
    extern __shared__ __align__(1024) unsigned char ht_raw[];
    __shared__ uint64_t full[HT_STAGES], empty[HT_STAGES], done;
    __shared__ uint32_t tmem_base;
    __shared__ float s_bias[HT_NMAX];
    __shared__ float4 s_stat[HT_M];  // per row: this slice's max, sum of exp, sum and sum of squares
    __shared__ float4 s_half[2][HT_M];  // the same per half of the columns
    __shared__ int s_ok, s_short;
    unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(ht_raw) + 1023) & ~(uintptr_t)1023);
    TraceEnd trace_guard(a.trace);
    const int tid = threadIdx.x, warp = tid >> 5;
    const int j = blockIdx.x, head = blockIdx.y, tile = blockIdx.z;
    const int v0 = j * HT_SLICE;
    const int cnt = (j == HT_SLICES - 1 ? a.V : v0 + HT_SLICE) - v0;  // vocabulary rows of this slice
    const bool wide = cnt > HT_SLICE;
    const int N = wide ? HT_NMAX : HT_SLICE;
    // activation rows copied per stage: 32, 64 or 128 (a short batch leaves the rest of the
    // A tile stale; the MMA rows it feeds are never read)
    const uint32_t stage_bytes = 2 * (uint32_t)a.a_rows * HT_K * 2 + (uint32_t)N * HT_K * 2;
    const int wrow = head * a.V + v0;  // first weight row of the slice
    const int arow = tile * HT_M;
    const int chunks = a.k_chunks;

    if (warp == 0) {
        tmem_alloc(&tmem_base, HT_TMEM_COLS);
        tmem_relinquish();
    }
    if (tid == 32) {
        for (int s = 0; s < HT_STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(&done, 1);
        fence_barrier_init();
        s_ok = 1;
    }
    for (int c = tid; c < HT_NMAX; c += HT_THREADS) s_bias[c] = c < cnt ? a.bias[wrow + c] : 0.f;
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base;

    // weight tiles of the first stages: independent of the previous kernel
    const int pre = chunks < HT_STAGES ? chunks : HT_STAGES;
    if (tid == 0) {
        for (int c = 0; c < pre; ++c) {
            unsigned char* st = smem + (size_t)c * HT_STAGE;
            mbar_arrive_expect_tx(&full[c], stage_bytes);
            tma_load_2d(st + 2 * HT_A_BYTES, wide ? &tw144 : &tw128, c * HT_K, wrow, &full[c]);
        }
    }
    pdl_launch_dependents();
    pdl_wait();
    trace_wait(a.trace);

    if (tid == 0) {  // producer
        for (int c = 0; c < chunks; ++c) {
            const int s = c % HT_STAGES;
            unsigned char* st = smem + (size_t)s * HT_STAGE;
            if (c >= HT_STAGES) {
                if (!mbar_wait(&empty[s], (uint32_t)((c / HT_STAGES) - 1) & 1, a.err)) {
                    s_ok = 0;
                    break;
                }
                mbar_arrive_expect_tx(&full[s], stage_bytes);
                tma_load_2d(st + 2 * HT_A_BYTES, wide ? &tw144 : &tw128, c * HT_K, wrow, &full[s]);
            }
            tma_load_2d(st, &tah, c * HT_K, arow, &full[s]);
            tma_load_2d(st + HT_A_BYTES, &tal, c * HT_K, arow, &full[s]);
        }
    } else if (tid == 32) {  // MMA issuer
        const uint32_t idesc = f16_idesc(HT_M, N, false);
        int c = 0;
        for (; c < chunks; ++c) {
            const int s = c % HT_STAGES;
            if (!mbar_wait(&full[s], (uint32_t)(c / HT_STAGES) & 1, a.err)) break;
            tc_fence_after();
            const uint32_t hb = smem_addr(smem + (size_t)s * HT_STAGE), lb = hb + HT_A_BYTES, wb = lb + HT_A_BYTES;
#pragma unroll
            for (int kk = 0; kk < HT_K / 16; ++kk) {
                const uint64_t dw = sw128_desc(wb + kk * 32);
                tc_mma(tmem, sw128_desc(hb + kk * 32), dw, idesc, (c | kk) != 0);
                tc_mma(tmem, sw128_desc(lb + kk * 32), dw, idesc, 1u);
            }
            tc_commit(&empty[s]);
        }
        if (c < chunks) s_ok = 0;
        tc_commit(&done);
    }
    if (warp < 2) __syncwarp();

    const bool fin = __syncthreads_and(mbar_wait(&done, 0, a.err)) != 0;
    tc_fence_after();
    const bool ok = fin && s_ok;  // block-uniform
    trace_mark(a.trace, 0);  // accumulator complete
    // thread = (row, half of the slice's columns): warps w and w + 4 read TMEM lanes 32 (w & 3) ..
    const int lq = warp & 3, half = warp >> 2, lane = tid & 31;
    const int rt = lq * 32 + lane;  // row within the tile (TMEM lane)
    const int row = arow + rt;
    const bool row_on = ok && row < a.m;
    const bool warp_on = ok && arow + lq * 32 < a.m;  // warp-uniform: a warp of padding rows only waits
    const uint32_t taddr = tmem + ((uint32_t)(lq * 32) << 16);
    const int cbeg = half * 64, cend = half ? N : 64;  // columns of this thread: [cbeg, cend) of the slice
    float* lst = a.out_logits ? reinterpret_cast<float*>(smem + HT_LOGIT_STAGE) + (size_t)rt * HT_LOGIT_PITCH : nullptr;

    // ---- phase 1, one pass: per (row, half), max, sum of exp (rescaled when a block of 32 raises
    // the max), and sum and sum of squares of the logits ----
    float mx = -INFINITY, sm = 0.f, s1 = 0.f, s2 = 0.f;
    if (warp_on) {
#pragma unroll 1
        for (int c0 = cbeg; c0 < cend; c0 += 32) {
            float v[32];
            tmem_ld32(taddr + (uint32_t)c0, v);
            float cm = -INFINITY;
#pragma unroll
            for (int e = 0; e < 32; ++e) {
                const int c = c0 + e;
                v[e] = c < cnt ? v[e] + s_bias[c] : -INFINITY;  // the logit (-inf past the slice)
                cm = fmaxf(cm, v[e]);
                if (c < cnt) {
                    s1 += v[e];
                    s2 = fmaf(v[e], v[e], s2);
                    if (lst) lst[c] = v[e];
                }
            }
            if (cm > mx) {
                sm *= __expf(mx - cm);
                mx = cm;
            }
#pragma unroll
            for (int e = 0; e < 32; ++e) sm += __expf(v[e] - mx);
        }
    }
    s_half[half][rt] = make_float4(mx, sm, s1, s2);
    __syncthreads();
    trace_mark(a.trace, 1);  // one pass over the slice
    if (half == 0) {  // the row's two halves, in half order
        const float4 p = s_half[0][rt], q = s_half[1][rt];
        const float M = fmaxf(p.x, q.x);
        const float S = (p.x == -INFINITY ? 0.f : p.y * __expf(p.x - M)) + (q.x == -INFINITY ? 0.f : q.y * __expf(q.x - M));
        s_stat[rt] = make_float4(M, S, p.z + q.z, p.w + q.w);
    }
    if (lst && ok) {  // the staged logit rows, 16 per warp, coalesced
        const float* st = reinterpret_cast<const float*>(smem + HT_LOGIT_STAGE);
#pragma unroll 1
        for (int r = warp * 16; r < warp * 16 + 16; ++r) {
            const int grow = arow + r;
            if (grow >= a.m) break;
            float* dst = a.out_logits + (size_t)grow * a.ldl + (size_t)head * a.V + v0;
            for (int c = lane; c < cnt; c += 32) dst[c] = st[(size_t)r * HT_LOGIT_PITCH + c];
        }
    }
    trace_mark(a.trace, 2);  // logits written
    cluster_arrive_release();
    cluster_wait();

    // ---- the row's lse (the 8 slices merged in slice order: the same in every CTA) and the
    // candidate threshold T = mean + z sd of the row's logits, as logp ----
    float lse = 0.f, T = -INFINITY;
    if (warp_on) {
        float4 p[HT_SLICES];
#pragma unroll
        for (int r = 0; r < HT_SLICES; ++r) p[r] = ld_dsmem4(dsmem_addr(&s_stat[rt], r));
        float M = p[0].x, t1 = 0.f, t2 = 0.f;
#pragma unroll
        for (int r = 1; r < HT_SLICES; ++r) M = fmaxf(M, p[r].x);
        float S = 0.f;
#pragma unroll
        for (int r = 0; r < HT_SLICES; ++r) {
            S += p[r].y * __expf(p[r].x - M);
            t1 += p[r].z;
            t2 += p[r].w;
        }
        lse = M + __logf(S);
        const float mean = t1 / (float)a.V, var = fmaxf(t2 / (float)a.V - mean * mean, 0.f);
        T = __fsub_rn(mean + a.z * sqrtf(var), lse);
    }

    // ---- phase 2: each half's best KM candidates (logp >= T) by (logp desc, id asc); the two
    // halves merged into the row's slice list, pushed to the CTA that owns the row; the owner
    // merges the 8 slice lists.  T only prunes: if a row has fewer than k candidates in all, the
    // cluster runs the phase again without it (exact either way). ----
    const int owner = rt / HT_ROWS_PER_OWNER, slot = (rt % HT_ROWS_PER_OWNER) * HT_SLICES + j;
    float* stg = reinterpret_cast<float*>(smem + HT_STAGING) + (size_t)tid * 33;
    float* hv_s = reinterpret_cast<float*>(smem + HT_HALF_LISTS);  // [2][128][KM] values, then ids
    int* hi_s = reinterpret_cast<int*>(smem + HT_HALF_LISTS) + 2 * HT_M * KM;
#pragma unroll 1
    for (int round = 0; round < 2; ++round) {
        if (warp_on) {
            float val[KM];
            int ids[KM];
#pragma unroll
            for (int q = 0; q < KM; ++q) {
                val[q] = -INFINITY;
                ids[q] = 0x7fffffff;
            }
            // per 32 columns: the logp values go to this thread's staging row; the candidates that
            // beat the current last entry form a mask, and only those are inserted (a warp iterates
            // as often as its busiest lane, not once per column)
#pragma unroll 1
            for (int c0 = cbeg; c0 < cend; c0 += 32) {
                float v[32];
                tmem_ld32(taddr + (uint32_t)c0, v);
                const float thr = val[KM - 1];
                uint32_t mask = 0;
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                    const float x = c0 + e < cnt ? __fsub_rn(v[e] + s_bias[c0 + e], lse) : -INFINITY;
                    stg[e] = x;
                    if (x >= T && x > thr) mask |= 1u << e;
                }
                while (mask) {
                    const int e = __ffs(mask) - 1;
                    mask &= mask - 1;
                    const float x = stg[e];
                    if (x > val[KM - 1]) topk_insert<KM>(val, ids, x, v0 + c0 + e);
                }
                __syncwarp();  // the next tcgen05.ld is warp-collective: reconverge after the per-lane loop
            }
            float* mv = hv_s + ((size_t)half * HT_M + rt) * KM;
            int* mi = hi_s + ((size_t)half * HT_M + rt) * KM;
#pragma unroll
            for (int q = 0; q < KM; q += 4) {
                *reinterpret_cast<float4*>(mv + q) = make_float4(val[q], val[q + 1], val[q + 2], val[q + 3]);
                *reinterpret_cast<int4*>(mi + q) = make_int4(ids[q], ids[q + 1], ids[q + 2], ids[q + 3]);
            }
        }
        __syncthreads();
        if (warp_on && half == 0) {  // the row's two half lists -> its slice list at the owner
            const float* av = hv_s + (size_t)rt * KM;
            const int* ai = hi_s + (size_t)rt * KM;
            const float* bv = hv_s + ((size_t)HT_M + rt) * KM;
            const int* bi = hi_s + ((size_t)HT_M + rt) * KM;
            int pa = 0, pb = 0;
            float ov[KM];
            int oi[KM];
#pragma unroll
            for (int t = 0; t < KM; ++t) {  // the first half holds the lower ids: it wins ties
                const float x = av[pa], y = bv[pb];
                const bool takea = x >= y;
                ov[t] = takea ? x : y;
                oi[t] = takea ? ai[pa] : bi[pb];
                pa += takea;
                pb += !takea;
            }
            float* cv = reinterpret_cast<float*>(smem) + (size_t)slot * KM;
            int* ci = reinterpret_cast<int*>(smem) + (size_t)HT_ROWS_PER_OWNER * HT_SLICES * KM + (size_t)slot * KM;
            const uint32_t dv = dsmem_addr(cv, owner), di = dsmem_addr(ci, owner);
#pragma unroll
            for (int q = 0; q < KM; q += 4) {
                st_dsmem4(dv + 4 * q, make_float4(ov[q], ov[q + 1], ov[q + 2], ov[q + 3]));
                st_dsmem4(di + 4 * q, make_float4(__int_as_float(oi[q]), __int_as_float(oi[q + 1]),
                                                  __int_as_float(oi[q + 2]), __int_as_float(oi[q + 3])));
            }
        }
        trace_mark(a.trace, 3 + 2 * round);  // candidate lists pushed
        cluster_arrive_release();
        cluster_wait();

        // ---- merge: rows 16 j .. 16 j + 15 of the tile; lanes 8 r .. 8 r + 7 (threads 0..127)
        // walk the 8 sorted lists of row r (lane = slice), each step the group's best head is
        // taken (ids differ between slices, so one lane advances) ----
        bool short_row = false;
        if (ok && tid < HT_ROWS_PER_OWNER * HT_SLICES) {
            const int rl = tid >> 3, sl = tid & 7, grow = arow + j * HT_ROWS_PER_OWNER + rl;
            const float* cv = reinterpret_cast<const float*>(smem) + (size_t)(rl * HT_SLICES + sl) * KM;
            const int* ci = reinterpret_cast<const int*>(smem) + (size_t)HT_ROWS_PER_OWNER * HT_SLICES * KM +
                            (size_t)(rl * HT_SLICES + sl) * KM;
            int pos = 0;
            float hv = cv[0];
            int hid = ci[0];
            const size_t o = ((size_t)grow * a.n + head) * a.k;
            const bool writer = sl == 0 && grow < a.m;
#pragma unroll 1
            for (int t = 0; t < a.k; ++t) {
                float bv = hv;
                int bi = hid;
#pragma unroll
                for (int off = 4; off > 0; off >>= 1) {
                    const float ov = __shfl_xor_sync(FULL_MASK, bv, off);
                    const int oi = __shfl_xor_sync(FULL_MASK, bi, off);
                    if (ov > bv || (ov == bv && oi < bi)) {
                        bv = ov;
                        bi = oi;
                    }
                }
                if (hv == bv && hid == bi) {
                    ++pos;
                    hv = pos < KM ? cv[pos] : -INFINITY;
                    hid = pos < KM ? ci[pos] : 0x7fffffff;
                }
                if (writer) {
                    a.out_ids[o + t] = bi;
                    a.out_logp[o + t] = bv;
                    short_row |= bv == -INFINITY;  // fewer than k candidates: the lists ran out
                }
            }
        }
        trace_mark(a.trace, 4 + 2 * round);  // merged
        if (round == 1) break;
        const int mine = __syncthreads_or(short_row);
        if (tid == 0) s_short = mine;
        cluster_arrive_release();  // the owners are done with their lists; every CTA's verdict is written
        cluster_wait();
        int any = 0;
#pragma unroll
        for (int r = 0; r < HT_SLICES; ++r) any |= ld_dsmem_i32(dsmem_addr(&s_short, r));
        if (!any) break;
        T = -INFINITY;
    }
    if (ok && a.out_lse && row_on && j == 0 && half == 0) a.out_lse[(size_t)row * a.n + head] = lse;
    if (!fin) mbar_wait(&done, 0, nullptr);  // MMAs may still run: let them finish before TMEM is freed
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, HT_TMEM_COLS);
}

}  // namespace

bool heads_tc_supported(int V, int k) {
    // slices 0..6 of 128 rows, slice 7 of 1..137 rows (N = 144 with the first row anywhere)
    return V > (HT_SLICES - 1) * HT_SLICE && V <= (HT_SLICES - 1) * HT_SLICE + 137 && k >= 1 && k <= MAX_TOPK;
}

int heads_tc_box_rows_wide() { return HT_NMAX; }

// z with P(N(0,1) > z) = p, by bisection on the complementary error function.
float normal_upper_quantile(double p) {
    double lo = -8.0, hi = 8.0;
    for (int i = 0; i < 60; ++i) {
        const double mid = 0.5 * (lo + hi);
        if (0.5 * std::erfc(mid / std::sqrt(2.0)) > p)
            lo = mid;
        else
            hi = mid;
    }
    return (float)(0.5 * (lo + hi));
}

cudaError_t launch_heads_tc(const HeadsTc& g0, cudaStream_t s, bool pdl) {
    HeadsTc g = g0;
    HeadsTcArgs& a = g.args;
    // Candidate threshold: were a row's logits normal, about 4k + 16 of its V would lie above
    // mean + z sd.  It only prunes the top-k work; rows left with fewer than k candidates
    // run again without it.
    a.z = normal_upper_quantile(std::min(0.5, (4.0 * a.k + 16.0) / a.V));
    if (!heads_tc_supported(a.V, a.k) || a.m < 1 || a.n < 1 || a.k_chunks < 1 ||
        (a.a_rows != 32 && a.a_rows != 64 && a.a_rows != HT_M) || (a.m > a.a_rows && a.a_rows != HT_M))
        return cudaErrorInvalidValue;
    const void* kern;
    if (a.k <= 4)
        kern = reinterpret_cast<const void*>(heads_tc_kernel<4>);
    else if (a.k <= 8)
        kern = reinterpret_cast<const void*>(heads_tc_kernel<8>);
    else if (a.k <= 16)
        kern = reinterpret_cast<const void*>(heads_tc_kernel<16>);
    else
        kern = reinterpret_cast<const void*>(heads_tc_kernel<32>);
    cudaError_t e = ensure_kernel_smem(kern, HT_SMEM);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(HT_SLICES, a.n, (a.m + HT_M - 1) / HT_M);
    cfg.blockDim = dim3(HT_THREADS);
    cfg.dynamicSmemBytes = HT_SMEM;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (a.k <= 4) return cudaLaunchKernelEx(&cfg, heads_tc_kernel<4>, g.w128, g.w144, g.a_hi, g.a_lo, a);
    if (a.k <= 8) return cudaLaunchKernelEx(&cfg, heads_tc_kernel<8>, g.w128, g.w144, g.a_hi, g.a_lo, a);
    if (a.k <= 16) return cudaLaunchKernelEx(&cfg, heads_tc_kernel<16>, g.w128, g.w144, g.a_hi, g.a_lo, a);
    return cudaLaunchKernelEx(&cfg, heads_tc_kernel<32>, g.w128, g.w144, g.a_hi, g.a_lo, a);
}

}  // namespace mtp
