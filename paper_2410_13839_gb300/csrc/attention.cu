// attention.cu -- causal attention of the fed rows over the paged bf16 KV cache
// (the attention of each block, Sec. III-A), split along the key axis.
//
// Grid (split, head, group).  A group is the rows of one slot (the n tokens
// fed this step, or 8 consecutive positions of a prefill chunk).  Each CTA
// takes a contiguous range of pages of its slot and streams their keys and
// values for its head through a ring of three shared-memory slots with
// cp.async.bulk (two are in flight while one is read).  Each warp takes
// 16-key tiles on the tensor cores (mma.sync) with the keys as the M side:
// S^T = K Q^T and O^T += V^T P^T, the fed rows' Q and P entering as bf16
// hi + lo pairs (two N = 8 operands), which keeps them to fp32 accuracy, and
// its online-softmax state in registers; the warps' states are merged in
// shared memory.  Partial results (max,
// sum, unnormalised output) of the splits are merged with a log-sum-exp by
// the CTA that finishes last (an atomic counter per group and head, reset by
// that CTA), so no second kernel is needed.
//
// Under programmatic dependent launch the first pages that hold only keys
// cached by earlier steps are fetched before griddepcontrol.wait; the pages
// touched by this step's appends are read after it.
#include <math.h>

#include <cstdio>

#include "common.cuh"
#include "kernels.cuh"
#include "mtp.h"

namespace mtp {
namespace {

constexpr int ATT_THREADS = 128;  // four warps: four CTAs per SM
constexpr int ATT_STAGES = 3;    // staging slots of the key/value ring (three 64-key slots keep ~48 KB in flight)
constexpr int RPG = MAX_ROWS;    // rows per group, upper bound
constexpr int PART = 2 + HEAD_DIM;  // (max, sum, out[64]) per row and split
constexpr int MAX_SPLITS = ATTN_MAX_SPLITS;  // one warp lane per split in the merge
static_assert(MAX_SPLITS <= 32, "the merge takes one lane per split");
static_assert(HEAD_DIM == 64, "score scale 0.125 assumes 64-wide heads");



// keys per staging half: 64, or a whole page when pages are longer
__host__ __device__ constexpr int half_keys(int page_size) { return page_size > 64 ? page_size : 64; }

__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}
__device__ __forceinline__ void mma_bf16(float (&d)[4], const uint32_t (&a)[4], const uint32_t (&b)[2]) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}
// The transpose of the 8 x 8 b16 matrix whose row lane / 4, columns 2 (lane % 4) and + 1, this
// lane holds in r: returns the same elements of the transposed matrix.
__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t r) {
    uint32_t d;
    asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(r));
    return d;
}
// x0, x1 as bf16 pairs hi + lo (hi + lo = x to about 2^-16 relative; low halves hold x0)
__device__ __forceinline__ void split2(float x0, float x1, uint32_t& hi, uint32_t& lo) {
    const __nv_bfloat16 h0 = __float2bfloat16_rn(x0), h1 = __float2bfloat16_rn(x1);
    const __nv_bfloat16 l0 = __float2bfloat16_rn(x0 - __bfloat162float(h0));
    const __nv_bfloat16 l1 = __float2bfloat16_rn(x1 - __bfloat162float(h1));
    hi = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
    lo = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
}

// Bulk copies of pages [p_from, p_to) of `seq` (this head) into the half
// that starts at key `key0` of the staging arrays, completing on `bar`.
// One thread calls it; returns whether anything was requested.
__device__ __forceinline__ bool stage_pages(const AttnArgs& a, int seq, int p_from, int p_to, int slot0,
                                            __nv_bfloat16* Ks, __nv_bfloat16* Vs, long long kv_head_off,
                                            long long v_off, uint64_t* bar, const int* ids = nullptr,
                                            int id0 = 0, int n_ids = 0) {
    const int P = a.page_size;
    const uint32_t blk = (uint32_t)P * HEAD_DIM * 2;
    // page p's id: from the shared copy ids[p - id0] when it holds it, else from the block table
    auto page_id = [&](int p) {
        return (ids && p - id0 >= 0 && p - id0 < n_ids) ? ids[p - id0] : a.block_table[(size_t)seq * a.bt_stride + p];
    };
    uint32_t bytes = 0;
    for (int p = p_from; p < p_to; ++p)
        if (page_id(p) >= 0) bytes += 2 * blk;
    if (!bytes) return false;
    fence_proxy_async();  // the half was last read by this CTA's threads
    mbar_arrive_expect_tx(bar, bytes);
    for (int p = p_from; p < p_to; ++p) {
        const int phys = page_id(p);
        if (phys < 0) {  // unreserved page: report, never read
            if (a.err) atomicOr(a.err, ERR_BOUNDS);
            continue;
        }
        const __nv_bfloat16* base = a.kv_pool + (long long)phys * a.page_elems + a.layer_off + kv_head_off;
        const int slot = slot0 + (p - p_from);
        bulk_copy_g2s(Ks + (size_t)slot * P * HEAD_DIM, base, blk, bar);
        bulk_copy_g2s(Vs + (size_t)slot * P * HEAD_DIM, base + v_off, blk, bar);
    }
    return true;
}

__global__ void __launch_bounds__(ATT_THREADS, 4) attn_kernel(const AttnArgs a) {
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ uint64_t bar;         // pages staged before the dependency wait
    __shared__ uint64_t hbar[ATT_STAGES];  // the staging slots
    __shared__ int s_armed[ATT_STAGES];
    __shared__ float s_scale[ATT_THREADS / 32][RPG];
    __shared__ int s_pos[RPG];
    __shared__ int s_act[RPG];
    __shared__ int s_rseq[RPG];
    __shared__ int s_seq, s_ktot, s_pre, s_last;
    constexpr int ID_CAP = 128;
    __shared__ int s_ids[ID_CAP];  // this split's page ids (the first ID_CAP), read once

    const int sp = blockIdx.x, h = blockIdx.y, g = blockIdx.z;
    TraceEnd trace_guard(a.trace);
    const int H = a.n_heads, P = a.page_size, S = a.n_splits;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int HALF_KEYS = half_keys(P);  // keys per staging half
    __nv_bfloat16* Ks = reinterpret_cast<__nv_bfloat16*>(smem);
    __nv_bfloat16* Vs = Ks + ATT_STAGES * HALF_KEYS * HEAD_DIM;
    float* qs = reinterpret_cast<float*>(Vs + ATT_STAGES * HALF_KEYS * HEAD_DIM);  // [RPG][64], pre-scaled
    const int pages_per_batch = HALF_KEYS / P;  // pages per staging half
    const long long kv_head_off = (long long)h * P * HEAD_DIM;
    const long long v_off = (long long)H * P * HEAD_DIM;

    if (tid == 0) {
        mbar_init(&bar, 1);
        for (int i = 0; i < ATT_STAGES; ++i) mbar_init(&hbar[i], 1);
        fence_barrier_init();
        s_pre = 0;
    }
    __syncthreads();

    // ---- before the wait: slot state left by earlier steps ----
    if (tid == 0 && a.plan != PLAN_ROWS) {
        int seq, old_len, n_new;
        if (a.plan == PLAN_DEVICE) {
            seq = a.seq_base + g;
            old_len = a.seq_len[seq];
            n_new = a.seq_new[seq];
        } else {
            seq = a.val_seq;
            old_len = a.val_old;
            n_new = a.val_new;
        }
        if (n_new > 0) {
            const int n_pg = (old_len + n_new + P - 1) / P;
            const int pps = (n_pg + S - 1) / S;
            const int pg0 = sp * pps, pg1 = min(n_pg, pg0 + pps);
            int pre_end = min(min(pg1, pg0 + pages_per_batch), old_len / P);  // half 0 at most
            for (int p = pg0; p < pre_end; ++p)  // only reserved pages are fetched early
                if (a.block_table[(size_t)seq * a.bt_stride + p] < 0) pre_end = p;
            if (pre_end > pg0) {
                const uint32_t blk = (uint32_t)P * HEAD_DIM * 2;
                mbar_arrive_expect_tx(&bar, 2u * blk * (uint32_t)(pre_end - pg0));
                for (int p = pg0; p < pre_end; ++p) {
                    const int phys = a.block_table[(size_t)seq * a.bt_stride + p];
                    const __nv_bfloat16* base = a.kv_pool + (long long)phys * a.page_elems + a.layer_off + kv_head_off;
                    bulk_copy_g2s(Ks + (p - pg0) * P * HEAD_DIM, base, blk, &bar);
                    bulk_copy_g2s(Vs + (p - pg0) * P * HEAD_DIM, base + v_off, blk, &bar);
                }
                s_pre = pre_end - pg0;
            }
        }
    }

    pdl_launch_dependents();
    pdl_wait();
    trace_wait(a.trace);

    // ---- rows of this group (written by this step's embedding) ----
    const int rpg = a.rows_per_group;
    if (tid < RPG) {
        const int r = g * rpg + tid;
        const int rs = tid < rpg ? a.row_seq[r] : -1;
        const int rp = tid < rpg ? a.row_pos[r] : -1;
        s_act[tid] = rs >= 0;
        s_rseq[tid] = rs;
        s_pos[tid] = rs >= 0 ? rp : -1;
    }
    __syncthreads();
    if (tid == 0) {
        int seq = -1, kmax = 0;
        for (int j = 0; j < RPG; ++j)
            if (s_act[j]) {
                seq = s_rseq[j];
                kmax = max(kmax, s_pos[j] + 1);
            }
        s_seq = seq;
        s_ktot = kmax;
    }
    __syncthreads();
    const int seq = s_seq, K_tot = s_ktot, n_pre = s_pre;
    // output pair (2 lane, 2 lane + 1) of head h in row row_j of the group
    auto put = [&](int row_j, float v0, float v1) {
        const size_t r = (size_t)(g * rpg + row_j);
        if (a.out) {
            float* o = a.out + r * a.ldo + h * HEAD_DIM + 2 * lane;
            o[0] = v0;
            o[1] = v1;
        }
        if (a.out_hi) {
            uint32_t hi, lo;
            split2(v0, v1, hi, lo);
            *reinterpret_cast<uint32_t*>(a.out_hi + r * a.ldb + h * HEAD_DIM + 2 * lane) = hi;
            *reinterpret_cast<uint32_t*>(a.out_lo + r * a.ldb + h * HEAD_DIM + 2 * lane) = lo;
        }
    };
    if (seq < 0) {  // nothing to do for this group (no split of it counts)
        if (n_pre > 0) mbar_wait(&bar, 0, a.err);
        if (a.out_hi && sp == 0)
            for (int row_j = warp; row_j < rpg; row_j += ATT_THREADS / 32) {
                const size_t o = (size_t)(g * rpg + row_j) * a.ldb + h * HEAD_DIM + 2 * lane;
                *reinterpret_cast<uint32_t*>(a.out_hi + o) = 0u;
                *reinterpret_cast<uint32_t*>(a.out_lo + o) = 0u;
            }
        return;
    }

    const int n_pg = (K_tot + P - 1) / P;
    const int pps = (n_pg + S - 1) / S;
    const int pg0 = sp * pps, pg1 = min(n_pg, pg0 + pps);

    for (int i = tid; i < RPG * HEAD_DIM; i += ATT_THREADS) {
        const int j = i / HEAD_DIM, dd = i % HEAD_DIM;
        qs[i] = s_act[j] ? a.q[(size_t)(g * rpg + j) * a.ldq + h * HEAD_DIM + dd] * 0.125f : 0.f;  // 1/sqrt(64)
    }
    const int n_ids = min(ID_CAP, max(0, pg1 - pg0));
    for (int i = tid; i < n_ids; i += ATT_THREADS) s_ids[i] = a.block_table[(size_t)seq * a.bt_stride + pg0 + i];
    __syncthreads();
    // batches of one staging slot each: batch i = pages pg0 + i*ppb .. in slot i % ATT_STAGES
    const int n_batches = (pg1 - pg0 + pages_per_batch - 1) / pages_per_batch;
    if (tid == 0) {
        for (int i = 0; i < ATT_STAGES; ++i) s_armed[i] = 0;
        for (int i = 0; i < ATT_STAGES && i < n_batches; ++i) {
            const int b0 = pg0 + i * pages_per_batch, b1 = min(pg1, b0 + pages_per_batch);
            const int from = i == 0 ? b0 + n_pre : b0;  // batch 0's first pages came before the wait
            s_armed[i] = stage_pages(a, seq, from, b1, i * pages_per_batch + (from - b0), Ks, Vs, kv_head_off,
                                     v_off, &hbar[i], s_ids, pg0, n_ids);
        }
    }
    __syncthreads();

    // per-warp tensor-core tiles with the keys as the M side: S^T = K Q^T (16 keys x the 8 query
    // rows; the queries' bf16 hi and lo parts are two N = 8 operands) and O^T += V^T P^T (head
    // dims x query rows, P^T's hi and lo parts added into the same accumulator).  Lane (g, c2):
    // keys g, g + 8 of a tile and queries c2, c2 + 1 in S^T; head dims g, g + 8 of each 16-dim
    // block and queries c2, c2 + 1 in O^T.
    const int g8 = lane >> 2, c2 = (lane & 3) * 2;
    bool qon[2];
    int qpos[2];
#pragma unroll
    for (int j = 0; j < 2; ++j) {
        qon[j] = s_act[c2 + j] != 0;
        qpos[j] = qon[j] ? s_pos[c2 + j] : -1;
    }
    uint32_t qhi[4][2], qlo[4][2];  // B operand of S^T: query row g8, dims ks * 16 + 8 hh + c2, + 1
    {
        const bool on = s_act[g8] != 0;
#pragma unroll
        for (int ks = 0; ks < 4; ++ks)
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
                const int k = ks * 16 + hh * 8 + c2;
                split2(on ? qs[g8 * HEAD_DIM + k] : 0.f, on ? qs[g8 * HEAD_DIM + k + 1] : 0.f, qhi[ks][hh],
                       qlo[ks][hh]);
            }
    }
    float m_w[2] = {-INFINITY, -INFINITY}, l_w[2] = {0.f, 0.f};
    float o[4][4];  // O^T block dp: dims dp * 16 + g8 (0, 1) and + 8 (2, 3), queries c2 + (i & 1)
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
        for (int i = 0; i < 4; ++i) o[j][i] = 0.f;
    const int swz = a.kv_swizzled ? 7 : 0;
    bool ok = true;
    uint32_t hphase[ATT_STAGES] = {};
    for (int i = 0; i < n_batches; ++i) {
        const int half = i % ATT_STAGES;
        const int bp = pg0 + i * pages_per_batch;
        const int nk = min(pages_per_batch, pg1 - bp) * P;
        if (i == 0 && n_pre > 0) ok = mbar_wait(&bar, 0, a.err) && ok;
        if (s_armed[half]) {
            ok = mbar_wait(&hbar[half], hphase[half], a.err) && ok;
            hphase[half] ^= 1u;
        }
        const uint32_t kb = smem_addr(Ks + (size_t)half * HALF_KEYS * HEAD_DIM);
        const uint32_t vb = smem_addr(Vs + (size_t)half * HALF_KEYS * HEAD_DIM);
        for (int kt = warp * 16; kt < nk && ok; kt += (ATT_THREADS / 32) * 16) {
            float sh[4] = {0.f, 0.f, 0.f, 0.f}, sl[4] = {0.f, 0.f, 0.f, 0.f};  // hi and lo parts: own chains
            {
                // A = K rows kt..kt+15: matrices (keys 0-7 | 8-15) x (dims 0-7 | 8-15) of the k-step
                const int key = kt + (lane & 7) + (((lane >> 3) & 1) << 3), chalf = lane >> 4;
#pragma unroll
                for (int ks = 0; ks < 4; ++ks) {
                    uint32_t ka[4];
                    ldsm_x4(ka, kb + key * 128 + ((uint32_t)((2 * ks + chalf) ^ (key & swz)) << 4));
                    const uint32_t bh[2] = {qhi[ks][0], qhi[ks][1]}, bl[2] = {qlo[ks][0], qlo[ks][1]};
                    mma_bf16(sh, ka, bh);
                    mma_bf16(sl, ka, bl);
                }
            }
            // this lane's scores: keys kt + g8 (i = 0, 1) and kt + g8 + 8 (i = 2, 3), query c2 + (i & 1)
            float sv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int kp = bp * P + kt + g8 + (i >> 1) * 8, j = i & 1;
                const float v = sh[i] + sl[i];
                sv[i] = qon[j] && kp <= qpos[j] && kp < K_tot ? v : -INFINITY;
            }
            float t0 = fmaxf(sv[0], sv[2]), t1 = fmaxf(sv[1], sv[3]);  // over the tile's keys: lanes g8
#pragma unroll
            for (int off = 4; off < 32; off <<= 1) {
                t0 = fmaxf(t0, __shfl_xor_sync(FULL_MASK, t0, off));
                t1 = fmaxf(t1, __shfl_xor_sync(FULL_MASK, t1, off));
            }
            const float mn[2] = {fmaxf(m_w[0], t0), fmaxf(m_w[1], t1)};
            float corr[2];
#pragma unroll
            for (int j = 0; j < 2; ++j)
                corr[j] = mn[j] == -INFINITY ? 1.f : (m_w[j] == -INFINITY ? 0.f : expf(m_w[j] - mn[j]));
            float pv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) pv[i] = sv[i] == -INFINITY ? 0.f : expf(sv[i] - mn[i & 1]);
            l_w[0] = l_w[0] * corr[0] + (pv[0] + pv[2]);
            l_w[1] = l_w[1] * corr[1] + (pv[1] + pv[3]);
            m_w[0] = mn[0];
            m_w[1] = mn[1];
#pragma unroll
            for (int dp = 0; dp < 4; ++dp) {
                o[dp][0] *= corr[0];
                o[dp][1] *= corr[1];
                o[dp][2] *= corr[0];
                o[dp][3] *= corr[1];
            }
            // P^T as the B operand (keys x queries): this lane holds rows g8 (keys) and columns c2 (queries)
            // of each 8 x 8 block; its transpose is the operand's layout (query g8, keys c2, c2 + 1)
            uint32_t ph0, pl0, ph1, pl1;
            split2(pv[0], pv[1], ph0, pl0);  // keys g8
            split2(pv[2], pv[3], ph1, pl1);  // keys g8 + 8
            const uint32_t bph[2] = {movmatrix_trans(ph0), movmatrix_trans(ph1)};
            const uint32_t bpl[2] = {movmatrix_trans(pl0), movmatrix_trans(pl1)};
            // A = V^T: matrices (dims 0-7 | 8-15 of block dp) x (keys 0-7 | 8-15), from the key rows
            const int vkey = kt + (lane & 7) + ((lane >> 4) << 3), vhalf = (lane >> 3) & 1;
#pragma unroll
            for (int dp = 0; dp < 4; ++dp) {
                uint32_t va[4];
                ldsm_x4_t(va, vb + vkey * 128 + ((uint32_t)((2 * dp + vhalf) ^ (vkey & swz)) << 4));
                mma_bf16(o[dp], va, bph);
                mma_bf16(o[dp], va, bpl);
            }
        }
        __syncthreads();  // every warp is done with this slot
        if (tid == 0 && i + ATT_STAGES < n_batches) {
            const int b0 = pg0 + (i + ATT_STAGES) * pages_per_batch, b1 = min(pg1, b0 + pages_per_batch);
            s_armed[half] = stage_pages(a, seq, b0, b1, half * pages_per_batch, Ks, Vs, kv_head_off, v_off,
                                        &hbar[half], s_ids, pg0, n_ids);
        }
        __syncthreads();
    }
    if (!__syncthreads_and(ok)) {  // error word set; let copies in flight land before leaving
        if (n_pre > 0) mbar_wait(&bar, 0, nullptr);
        for (int hb = 0; hb < ATT_STAGES; ++hb)
            if (s_armed[hb]) mbar_wait(&hbar[hb], hphase[hb], nullptr);
        return;
    }
    // merge the warps' (max, sum, out) per row through the staging area:
    // warp j then holds row j's (m_run, l_run) and output dims 2 lane, 2 lane + 1
#pragma unroll
    for (int j = 0; j < 2; ++j)  // each lane summed its own keys; the query's keys span lanes g8
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) l_w[j] += __shfl_xor_sync(FULL_MASK, l_w[j], off);
    float* wst = reinterpret_cast<float*>(Ks);  // [warps][RPG][PART]
#pragma unroll
    for (int j = 0; j < 2; ++j) {
        float* ws = wst + ((size_t)warp * RPG + c2 + j) * PART;
        if (g8 == 0) {
            ws[0] = m_w[j];
            ws[1] = l_w[j];
        }
#pragma unroll
        for (int dp = 0; dp < 4; ++dp) {
            ws[2 + dp * 16 + g8] = o[dp][j];
            ws[2 + dp * 16 + g8 + 8] = o[dp][2 + j];
        }
    }
    __syncthreads();
    constexpr int NW = ATT_THREADS / 32;
    if (tid < NW * RPG) {
        const int w = tid / RPG, j = tid % RPG;
        float M = -INFINITY;
#pragma unroll
        for (int v = 0; v < NW; ++v) M = fmaxf(M, wst[((size_t)v * RPG + j) * PART]);
        const float mw = wst[((size_t)w * RPG + j) * PART];
        s_scale[w][j] = mw == -INFINITY ? 0.f : expf(mw - M);
    }
    __syncthreads();
    // rows warp, warp + NW, ...: (max, sum, output dims 2 lane, 2 lane + 1) over this CTA's keys
    constexpr int RPW = (RPG + NW - 1) / NW;  // rows per warp
    float m_run[RPW], l_run[RPW], acc0[RPW], acc1[RPW];
#pragma unroll
    for (int q = 0; q < RPW; ++q) {
        const int row_j = warp + q * NW;
        m_run[q] = -INFINITY;
        l_run[q] = acc0[q] = acc1[q] = 0.f;
        if (row_j >= RPG) continue;
#pragma unroll
        for (int w = 0; w < NW; ++w) {
            const float sc = s_scale[w][row_j];
            const float* ws = wst + ((size_t)w * RPG + row_j) * PART;
            m_run[q] = fmaxf(m_run[q], ws[0]);
            l_run[q] = fmaf(sc, ws[1], l_run[q]);
            acc0[q] = fmaf(sc, ws[2 + 2 * lane], acc0[q]);
            acc1[q] = fmaf(sc, ws[3 + 2 * lane], acc1[q]);
        }
    }
    if (S == 1) {
#pragma unroll
        for (int q = 0; q < RPW; ++q) {
            const int row_j = warp + q * NW;
            if (row_j < RPG && s_act[row_j]) {
                put(row_j, acc0[q] / l_run[q], acc1[q] / l_run[q]);
            } else if (row_j < rpg && a.out_hi) {
                put(row_j, 0.f, 0.f);
            }
        }
        return;
    }

    float* part = a.ws_part + (((size_t)(g * H + h) * S + sp) * RPG) * PART;
#pragma unroll
    for (int q = 0; q < RPW; ++q) {
        const int row_j = warp + q * NW;
        if (row_j >= RPG) continue;
        float* pj = part + row_j * PART;
        if (lane == 0) {
            pj[0] = m_run[q];
            pj[1] = l_run[q];
        }
        pj[2 + 2 * lane] = acc0[q];
        pj[3 + 2 * lane] = acc1[q];
    }
    __threadfence();
    __syncthreads();
    trace_mark(a.trace, 2);  // split partials written
    if (tid == 0) s_last = atomicAdd(a.ws_count + g * H + h, 1) == S - 1;
    __syncthreads();
    if (!s_last) return;
    __threadfence();

#pragma unroll 1
    for (int row_j = warp; row_j < RPG; row_j += NW) {
        if (!s_act[row_j]) {
            if (row_j < rpg && a.out_hi) put(row_j, 0.f, 0.f);
            continue;
        }
        // lane s holds split s's (max, sum); every split's output pair is
        // loaded before any is used, so the merge costs one L2 round trip
        const float* base = a.ws_part + ((size_t)(g * H + h) * S * RPG) * PART + row_j * PART;
        const size_t sstride = (size_t)RPG * PART;
        float ms = -INFINITY, ls = 0.f;
        if (lane < S) {
            ms = __ldcg(base + lane * sstride);
            ls = __ldcg(base + lane * sstride + 1);
        }
        float o0[MAX_SPLITS], o1[MAX_SPLITS];
#pragma unroll
        for (int sx = 0; sx < MAX_SPLITS; ++sx) {
            o0[sx] = sx < S ? __ldcg(base + sx * sstride + 2 + 2 * lane) : 0.f;
            o1[sx] = sx < S ? __ldcg(base + sx * sstride + 3 + 2 * lane) : 0.f;
        }
        const float M = warp_max(ms);
        const float w = (ms == -INFINITY) ? 0.f : expf(ms - M);
        const float L = warp_sum(w * ls);
        float r0 = 0.f, r1 = 0.f;
#pragma unroll
        for (int sx = 0; sx < MAX_SPLITS; ++sx) {
            const float ws = __shfl_sync(FULL_MASK, w, sx);
            r0 = fmaf(ws, o0[sx], r0);
            r1 = fmaf(ws, o1[sx], r1);
        }
        put(row_j, r0 / L, r1 / L);
    }
    if (tid == 0) a.ws_count[g * H + h] = 0;
}

}  // namespace

size_t attn_workspace_floats(int groups, int n_heads, int n_splits, int /*rows_per_group*/) {
    return (size_t)groups * n_heads * n_splits * RPG * PART;
}

size_t attn_smem_bytes(int page_size) {
    return (size_t)2 * ATT_STAGES * half_keys(page_size) * HEAD_DIM * 2 + (size_t)RPG * HEAD_DIM * 4;
}

int attn_splits_for(int groups, int n_heads, int page_size, int max_keys, int num_sms) {
    const int max_pages = (max_keys + page_size - 1) / page_size;
    int s = num_sms / max(1, groups * n_heads);
    s = max(1, min(min(s, max_pages), MAX_SPLITS));
    return s;
}

cudaError_t launch_attention(const AttnArgs& a, int groups, cudaStream_t s, bool pdl) {
    if (a.rows_per_group < 1 || a.rows_per_group > RPG || half_keys(a.page_size) % a.page_size != 0 ||
        a.n_splits < 1 || a.n_splits > MAX_SPLITS)
        return cudaErrorInvalidValue;
    const size_t smem = attn_smem_bytes(a.page_size);
    cudaError_t e = ensure_kernel_smem(reinterpret_cast<const void*>(attn_kernel), smem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.n_splits, a.n_heads, groups);
    cfg.blockDim = dim3(ATT_THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, attn_kernel, a);
}

}  // namespace mtp

// ---- allocation-free attention (mtp_attention_noalloc) ----------------------
// For callers that may not allocate GPU memory while they run (a real-time
// audio callback, where cudaMalloc/cudaFree can block or synchronise the
// device; a host that owns all GPU memory): the split-merge scratch of the
// attention kernel is this fixed array, one per GPU that loads the library,
// held until the process exits and shared by every call on that GPU.
static __device__ __align__(256) unsigned char g_attention_scratch[MTP_ATTENTION_NOALLOC_SCRATCH_BYTES];

extern "C" MTP_API int mtp_attention_noalloc(const mtp_attention_args* args, void* cuda_stream) {
    mtp::clear_error();
    mtp::AttnStandalonePlan p;
    const int r = mtp::attention_standalone_plan(args, true, &p);  // checked before anything is queued
    if (r != MTP_OK) return r;
    if (p.need > MTP_ATTENTION_NOALLOC_SCRATCH_BYTES) {
        char msg[256];
        std::snprintf(msg, sizeof(msg),
                      "attention: this call needs %zu bytes of scratch, the fixed scratch array holds %u", p.need,
                      (unsigned)MTP_ATTENTION_NOALLOC_SCRATCH_BYTES);
        return mtp::report_error(MTP_ERR_INVALID, msg);
    }
    // The array's name is only a host-side stand-in for it; its device address
    // is looked up on every call (no allocation), so it stays right after the
    // context of the device is torn down and made again.
    void* scratch = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&scratch, g_attention_scratch);
    if (e != cudaSuccess || !scratch) {
        char msg[256];
        std::snprintf(msg, sizeof(msg), "attention scratch address lookup failed: %s", cudaGetErrorString(e));
        return mtp::report_error(MTP_ERR_CUDA, msg);
    }
    const cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
    e = cudaMemsetAsync(static_cast<char*>(scratch) + p.part_bytes, 0, p.count_bytes, s);  // merge counters
    if (e != cudaSuccess) return mtp::report_error(MTP_ERR_CUDA, cudaGetErrorString(e));
    return mtp::attention_standalone_launch(args, p, scratch, s);
}
