// attention.cu -- causal attention of the fed rows over the paged bf16 KV cache
// (the attention of each block, Sec. III-A), split along the key axis.
//
// Grid (split, head, group).  A group is the rows of one slot (the n tokens
// fed this step, or 8 consecutive positions of a prefill chunk).  Each CTA
// takes a contiguous range of pages of its slot and streams their keys and
// values for its head through two halves of shared memory with
// cp.async.bulk (one half is filled while the other is read).  Each warp
// takes 16-key tiles: S = Q K^T and O += P V on the tensor cores (mma.sync;
// the fed rows are the M side, Q and P enter as bf16 hi + lo pairs, which
// keeps them to fp32 accuracy) with its online-softmax state in registers;
// the warps' states are merged in shared memory.  Partial results (max,
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

    // per-warp tensor-core tiles: fragment rows = fed rows (rows >= RPG zero)
    const int qrow = lane >> 2, c2 = (lane & 3) * 2;
    const bool qon = qrow < RPG && s_act[qrow];
    const int qpos = qon ? s_pos[qrow] : -1;
    uint32_t qhi[4][2], qlo[4][2];
#pragma unroll
    for (int ks = 0; ks < 4; ++ks)
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            const int k = ks * 16 + hh * 8 + c2;
            split2(qon ? qs[qrow * HEAD_DIM + k] : 0.f, qon ? qs[qrow * HEAD_DIM + k + 1] : 0.f, qhi[ks][hh],
                   qlo[ks][hh]);
        }
    float m_w = -INFINITY, l_w = 0.f;
    float o[8][4];
#pragma unroll
    for (int j = 0; j < 8; ++j)
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
            float sh[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
            float sl[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
            {
                const int key = kt + (lane & 7) + ((lane >> 4) << 3), chalf = (lane >> 3) & 1;
#pragma unroll
                for (int ks = 0; ks < 4; ++ks) {
                    uint32_t b[4];
                    ldsm_x4(b, kb + key * 128 + ((uint32_t)((2 * ks + chalf) ^ (key & swz)) << 4));
                    const uint32_t ah[4] = {qhi[ks][0], 0u, qhi[ks][1], 0u};
                    const uint32_t al[4] = {qlo[ks][0], 0u, qlo[ks][1], 0u};
                    const uint32_t b0[2] = {b[0], b[1]}, b1[2] = {b[2], b[3]};
                    mma_bf16(sh[0], ah, b0);
                    mma_bf16(sl[0], al, b0);
                    mma_bf16(sh[1], ah, b1);
                    mma_bf16(sl[1], al, b1);
                }
            }
            // this lane's scores: row qrow, keys kt + {c2, c2 + 1, 8 + c2, 9 + c2} of the batch
            float sv[4] = {sh[0][0] + sl[0][0], sh[0][1] + sl[0][1], sh[1][0] + sl[1][0], sh[1][1] + sl[1][1]};
            float tmax = -INFINITY;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int kp = bp * P + kt + (q >> 1) * 8 + c2 + (q & 1);
                sv[q] = qon && kp <= qpos ? sv[q] : -INFINITY;
                tmax = fmaxf(tmax, sv[q]);
            }
            tmax = fmaxf(tmax, __shfl_xor_sync(FULL_MASK, tmax, 1));
            tmax = fmaxf(tmax, __shfl_xor_sync(FULL_MASK, tmax, 2));
            const float m_new = fmaxf(m_w, tmax);
            const float corr = m_new == -INFINITY ? 1.f : (m_w == -INFINITY ? 0.f : expf(m_w - m_new));
            float pv[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) pv[q] = sv[q] == -INFINITY ? 0.f : expf(sv[q] - m_new);
            l_w = l_w * corr + ((pv[0] + pv[1]) + (pv[2] + pv[3]));
            m_w = m_new;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                o[j][0] *= corr;
                o[j][1] *= corr;
            }
            uint32_t ph[4] = {0u, 0u, 0u, 0u}, pl[4] = {0u, 0u, 0u, 0u};
            split2(pv[0], pv[1], ph[0], pl[0]);
            split2(pv[2], pv[3], ph[2], pl[2]);
            const int vkey = kt + (lane & 7) + (((lane >> 3) & 1) << 3), vhalf = lane >> 4;
#pragma unroll
            for (int dp = 0; dp < 4; ++dp) {
                uint32_t v[4];
                ldsm_x4_t(v, vb + vkey * 128 + ((uint32_t)((2 * dp + vhalf) ^ (vkey & swz)) << 4));
                const uint32_t v0[2] = {v[0], v[1]}, v1[2] = {v[2], v[3]};
                mma_bf16(o[2 * dp], ph, v0);
                mma_bf16(o[2 * dp], pl, v0);
                mma_bf16(o[2 * dp + 1], ph, v1);
                mma_bf16(o[2 * dp + 1], pl, v1);
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
    l_w += __shfl_xor_sync(FULL_MASK, l_w, 1);
    l_w += __shfl_xor_sync(FULL_MASK, l_w, 2);
    float* wst = reinterpret_cast<float*>(Ks);  // [warps][RPG][PART]
    if (qrow < RPG) {
        float* ws = wst + ((size_t)warp * RPG + qrow) * PART;
        if (c2 == 0) {
            ws[0] = m_w;
            ws[1] = l_w;
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) *reinterpret_cast<float2*>(ws + 2 + j * 8 + c2) = make_float2(o[j][0], o[j][1]);
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
