// attention_tc.cu -- causal attention of prompt rows on the tensor cores
// (tcgen05), the attention of each block during prefill (Sec. III-A: the
// concatenated phoneme + acoustic prompt runs through the blocks as one
// sequence, every position attending to itself and the positions before it).
//
// Grid (split, head, tile).  A tile is 128 rows of the pass, the MMA's M side
// and the 128 TMEM lanes; its rows may belong to several slots (a prefill pass
// packs the prompts of many slots).  Each distinct slot of the tile is a
// segment; the segment's keys 0 .. (its largest position) are cut into items
// of 128 keys, and split s takes items s, s + S, ... of every segment.  Per
// item, with the cached keys and values of the item's pages copied by
// cp.async.bulk into a two-stage ring (the cache stores chunk c of key row t
// at c ^ (t & 7): exactly the 128-byte-swizzled tile the MMA reads):
//
//   S  = (Q_hi + Q_lo) K^T       two MMAs per 16 dims, 128 x 128 fp32 in TMEM
//   P  = exp(S - m_new)          one thread per row (TMEM lane), masked to the
//                                row's own slot and keys <= its position,
//                                written to shared memory as bf16 hi + lo
//   O' = (P_hi + P_lo) V         two MMAs per 16 keys, 128 x 64 fp32 in TMEM
//                                (V read as an MN-major operand)
//   o  = o * exp(m - m_new) + O' in registers (online softmax)
//
// Q and P enter as bf16 hi + lo pairs (hi + lo = x to about 2^-16 relative),
// so the products keep fp32 accuracy; the keys and values are the cache's bf16.
// One elected thread of the fifth warp issues the copies and the MMAs; the
// four other warps own one row each per thread.  Splits leave (max, sum,
// unnormalised output) per row in the workspace and the CTA that finishes
// last merges them (an atomic counter per tile and head, reset by that CTA).
#include <math.h>

#include <algorithm>

#include "common.cuh"
#include "kernels.cuh"
#include "mtp.h"
#include "tcgen05.cuh"

namespace mtp {
namespace {

constexpr int PA_ROWS = 128;     // query rows per tile: MMA M, TMEM lanes
constexpr int PA_KEYS = 128;     // keys per item: N of Q K^T, K of P V
constexpr int PA_THREADS = 160;  // four row warps + the issuing warp
constexpr int PA_PART = 4 + HEAD_DIM;  // (max, sum, -, -, out[64]): out 16-byte aligned for float4 access
constexpr uint32_t PA_TILE = PA_ROWS * 128;  // 128 rows of 128 bytes
// shared memory (1024-byte aligned): Q hi | Q lo | P hi (keys 0-63, 64-127) |
// P lo (same) | stage 0 K | stage 0 V | stage 1 K | stage 1 V
constexpr uint32_t OFF_Q = 0, OFF_P = 2 * PA_TILE, OFF_KV = 6 * PA_TILE;
constexpr uint32_t PA_SMEM = 10 * PA_TILE + 1024;
constexpr uint32_t TM_S = 0, TM_O = 128, TM_COLS = 256;  // TMEM columns: S [128), O' double-buffered [64) x 2

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

// x0..x7 as 16 bytes of bf16 hi and 16 bytes of bf16 lo
__device__ __forceinline__ void split8(const float* x, uint4& hi, uint4& lo) {
    uint32_t h[4], l[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const __nv_bfloat16 h0 = __float2bfloat16_rn(x[2 * q]), h1 = __float2bfloat16_rn(x[2 * q + 1]);
        const __nv_bfloat16 l0 = __float2bfloat16_rn(x[2 * q] - __bfloat162float(h0));
        const __nv_bfloat16 l1 = __float2bfloat16_rn(x[2 * q + 1] - __bfloat162float(h1));
        h[q] = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
        l[q] = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
    }
    hi = make_uint4(h[0], h[1], h[2], h[3]);
    lo = make_uint4(l[0], l[1], l[2], l[3]);
}

__global__ void __launch_bounds__(PA_THREADS, 1) attn_tc_kernel(const AttnArgs a) {
    extern __shared__ __align__(1024) unsigned char pa_raw[];
    __shared__ uint64_t kv_full[2], kv_empty[2], s_full, p_full, o_full[2], done;
    __shared__ uint32_t tmem_base;
    __shared__ int s_seq[PA_ROWS], s_pos[PA_ROWS];
    __shared__ int seg_slot[PA_ROWS], seg_kmax[PA_ROWS];
    __shared__ int s_nseg, s_abort, s_last;
    unsigned char* sm = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(pa_raw) + 1023) & ~(uintptr_t)1023);
    TraceEnd trace_guard(a.trace);
    const int sp = blockIdx.x, h = blockIdx.y, tile = blockIdx.z;
    const int S = a.n_splits, H = a.n_heads, P = a.page_size;
    const int tid = threadIdx.x, warp = tid >> 5;
    const int row0 = tile * PA_ROWS;

    // ---- independent of the previous kernel ----
    if (warp == 4) {
        tmem_alloc(&tmem_base, TM_COLS);
        tmem_relinquish();
    }
    if (tid == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(&kv_full[i], 1);
            mbar_init(&kv_empty[i], 1);
            mbar_init(&o_full[i], 1);
        }
        mbar_init(&s_full, 1);
        mbar_init(&p_full, PA_ROWS);
        mbar_init(&done, 1);
        fence_barrier_init();
        s_abort = 0;
    }
    {  // keys and values past a segment's pages are read as zeros times zero weights: keep them finite
        uint4* kv = reinterpret_cast<uint4*>(sm + OFF_KV);
        for (int i = tid; i < (int)(4 * PA_TILE / 16); i += PA_THREADS) kv[i] = make_uint4(0u, 0u, 0u, 0u);
    }
    fence_proxy_async();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base;
    pdl_launch_dependents();
    pdl_wait();
    trace_wait(a.trace);

    // ---- the tile's rows, segments and this split's items ----
    if (tid < PA_ROWS) {
        const int r = row0 + tid;
        const int rs = r < a.rows ? a.row_seq[r] : -1;
        s_seq[tid] = rs;
        s_pos[tid] = rs >= 0 ? a.row_pos[r] : -1;
    }
    __syncthreads();
    if (tid == 0) {
        int nseg = 0;
        for (int r = 0; r < PA_ROWS; ++r) {
            const int q = s_seq[r];
            if (q < 0) continue;
            int g = 0;
            while (g < nseg && seg_slot[g] != q) ++g;
            if (g == nseg) {
                seg_slot[g] = q;
                seg_kmax[g] = 0;
                ++nseg;
            }
            seg_kmax[g] = max(seg_kmax[g], s_pos[r] + 1);
        }
        s_nseg = nseg;
    }
    // ---- Q of this head: rows pre-scaled by 1/sqrt(64), bf16 hi | lo, swizzled ----
    if (tid < PA_ROWS) {
        const int r = row0 + tid;
        const bool on = s_seq[tid] >= 0;
        unsigned char* qhi = sm + OFF_Q + tid * 128;
        unsigned char* qlo = qhi + PA_TILE;
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            float x[8];
            if (on) {
                const float4* src = reinterpret_cast<const float4*>(a.q + (size_t)r * a.ldq + h * HEAD_DIM + c * 8);
                const float4 u = src[0], v = src[1];
                x[0] = u.x * 0.125f; x[1] = u.y * 0.125f; x[2] = u.z * 0.125f; x[3] = u.w * 0.125f;
                x[4] = v.x * 0.125f; x[5] = v.y * 0.125f; x[6] = v.z * 0.125f; x[7] = v.w * 0.125f;
            } else {
#pragma unroll
                for (int e = 0; e < 8; ++e) x[e] = 0.f;
            }
            uint4 hi, lo;
            split8(x, hi, lo);
            const int at = (c ^ (tid & 7)) << 4;
            *reinterpret_cast<uint4*>(qhi + at) = hi;
            *reinterpret_cast<uint4*>(qlo + at) = lo;
        }
    }
    fence_proxy_async();  // Q is read by the tensor cores
    __syncthreads();
    // this split's items in order: segment g, key tiles j = sp, sp + S, ... below the segment's end
    const int nseg = s_nseg;
    auto skip_empty = [&](int2 t) {
        while (t.x < nseg && t.y * PA_KEYS >= seg_kmax[t.x]) {
            ++t.x;
            t.y = sp;
        }
        return t;
    };
    auto next_item = [&](int2 t) {
        t.y += S;
        return skip_empty(t);
    };
    const int2 first = skip_empty(make_int2(0, sp));

    const long long kv_head = (long long)h * P * HEAD_DIM, v_off = (long long)H * P * HEAD_DIM;
    // copies of item i into stage i & 1: the pages of keys [128 j, 128 j + 128) below the segment's end
    auto stage_item = [&](int i, int2 t) {
        const int g = t.x, j = t.y;
        const int seq = seg_slot[g];
        const int k0 = j * PA_KEYS, k1 = min(k0 + PA_KEYS, seg_kmax[g]);
        const uint32_t blk = (uint32_t)P * 128;
        unsigned char* ks = sm + OFF_KV + (uint32_t)(i & 1) * 2 * PA_TILE;
        // pages past the slot's table row count as unreserved
        auto page_of = [&](int p) { return p < a.bt_stride ? a.block_table[(size_t)seq * a.bt_stride + p] : -1; };
        uint32_t bytes = 0;
        for (int p = k0 / P; p * P < k1; ++p)
            if (page_of(p) >= 0) bytes += 2 * blk;
        mbar_arrive_expect_tx(&kv_full[i & 1], bytes);
        for (int p = k0 / P; p * P < k1; ++p) {
            const int phys = page_of(p);
            if (phys < 0) {  // unreserved page: report, never read
                if (a.err) atomicOr(a.err, ERR_BOUNDS);
                continue;
            }
            const __nv_bfloat16* base = a.kv_pool + (long long)phys * a.page_elems + a.layer_off + kv_head;
            const uint32_t at = (uint32_t)(p * P - k0) * 128;
            bulk_copy_g2s(ks + at, base, blk, &kv_full[i & 1]);
            bulk_copy_g2s(ks + PA_TILE + at, base + v_off, blk, &kv_full[i & 1]);
        }
    };

    float m_run = -INFINITY, l_run = 0.f, o[HEAD_DIM];
#pragma unroll
    for (int c = 0; c < HEAD_DIM; ++c) o[c] = 0.f;

    if (tid == PA_ROWS) {  // ---- the issuing thread: copies and MMAs ----
        constexpr uint32_t IDESC_S = f16_idesc(PA_ROWS, PA_KEYS, false);
        constexpr uint32_t IDESC_O = f16_idesc(PA_ROWS, HEAD_DIM, true);
        const uint32_t q_hi = smem_addr(sm + OFF_Q), q_lo = q_hi + PA_TILE;
        const uint32_t p_hi = smem_addr(sm + OFF_P), p_lo = p_hi + 2 * PA_TILE;
        bool staged[2] = {false, false};
        bool ok = true;
        if (first.x < nseg) {
            stage_item(0, first);
            staged[0] = true;
        }
        int i = 0;
        for (int2 t = first; t.x < nseg; t = next_item(t), ++i) {
            const int st = i & 1;
            const int2 t1 = next_item(t);
            if (t1.x < nseg) {  // item i - 1 held the other stage: its MMAs must be done
                if (i >= 1) ok = mbar_wait(&kv_empty[st ^ 1], (uint32_t)((i - 1) >> 1) & 1, a.err);
                if (!ok) break;
                stage_item(i + 1, t1);
                staged[st ^ 1] = true;
            }
            ok = mbar_wait(&kv_full[st], (uint32_t)(i >> 1) & 1, a.err);
            if (!ok) break;
            staged[st] = false;
            tc_fence_after();
            const uint32_t kb = smem_addr(sm + OFF_KV + (uint32_t)st * 2 * PA_TILE), vb = kb + PA_TILE;
#pragma unroll
            for (int kk = 0; kk < HEAD_DIM / 16; ++kk) {
                const uint64_t bk = sw128_desc(kb + kk * 32);
                tc_mma(tmem + TM_S, sw128_desc(q_hi + kk * 32), bk, IDESC_S, kk != 0);
                tc_mma(tmem + TM_S, sw128_desc(q_lo + kk * 32), bk, IDESC_S, 1u);
            }
            tc_commit(&s_full);
            ok = mbar_wait(&p_full, (uint32_t)i & 1, a.err);
            if (!ok) break;
            tc_fence_after();
            const uint32_t od = tmem + TM_O + (uint32_t)st * HEAD_DIM;
#pragma unroll
            for (int kk = 0; kk < PA_KEYS / 16; ++kk) {
                const uint32_t pa = (uint32_t)(kk >> 2) * PA_TILE + (uint32_t)(kk & 3) * 32;
                const uint64_t bv = sw128_mn_desc(vb + kk * 2048);
                tc_mma(od, sw128_desc(p_hi + pa), bv, IDESC_O, kk != 0);
                tc_mma(od, sw128_desc(p_lo + pa), bv, IDESC_O, 1u);
            }
            tc_commit(&o_full[st]);
            tc_commit(&kv_empty[st]);
        }
        if (!ok) s_abort = 1;
        tc_commit(&done);  // every MMA issued above has completed
        mbar_wait(&done, 0, nullptr);
        for (int st = 0; st < 2; ++st)  // copies still in flight land before the CTA leaves
            if (staged[st]) mbar_wait(&kv_full[st], (uint32_t)((i + (st != (i & 1))) >> 1) & 1, nullptr);
    } else if (tid < PA_ROWS) {  // ---- one row per thread: softmax and accumulation ----
        const int my_seq = s_seq[tid], my_pos = s_pos[tid];
        const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
        unsigned char* prow_hi = sm + OFF_P + tid * 128;
        unsigned char* prow_lo = prow_hi + 2 * PA_TILE;
        int i = 0;
        for (int2 t = first; t.x < nseg; t = next_item(t), ++i) {
            const bool in = my_seq >= 0 && seg_slot[t.x] == my_seq;
            const int k0 = t.y * PA_KEYS;
            // warp-uniform decisions: tcgen05.ld is issued by whole warps
            if (!__all_sync(FULL_MASK, mbar_wait(&s_full, (uint32_t)i & 1, a.err))) {
                s_abort = 1;
                break;
            }
            tc_fence_after();
            float sv[PA_KEYS];
#pragma unroll
            for (int c0 = 0; c0 < PA_KEYS; c0 += 32) {
                float v[32];
                tmem_ld32(tmem + lane_base + TM_S + c0, v);
#pragma unroll
                for (int e = 0; e < 32; ++e) sv[c0 + e] = (in && k0 + c0 + e <= my_pos) ? v[e] : -INFINITY;
            }
            float tmax = -INFINITY;
#pragma unroll
            for (int c = 0; c < PA_KEYS; ++c) tmax = fmaxf(tmax, sv[c]);
            const float m_new = fmaxf(m_run, tmax);
            const float corr = m_new == -INFINITY ? 1.f : (m_run == -INFINITY ? 0.f : expf(m_run - m_new));
            float psum = 0.f;
#pragma unroll
            for (int c8 = 0; c8 < PA_KEYS / 8; ++c8) {
                float pv[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const float x = sv[c8 * 8 + e];
                    pv[e] = x == -INFINITY ? 0.f : expf(x - m_new);
                }
                psum += ((pv[0] + pv[1]) + (pv[2] + pv[3])) + ((pv[4] + pv[5]) + (pv[6] + pv[7]));
                uint4 hi, lo;
                split8(pv, hi, lo);
                const uint32_t at = (uint32_t)(c8 >> 3) * PA_TILE + ((uint32_t)((c8 & 7) ^ (tid & 7)) << 4);
                *reinterpret_cast<uint4*>(prow_hi + at) = hi;
                *reinterpret_cast<uint4*>(prow_lo + at) = lo;
            }
            l_run = l_run * corr + psum;
            m_run = m_new;
            fence_proxy_async();  // P is read by the tensor cores
            tc_fence_before();
            mbar_arrive(&p_full);
            if (!__all_sync(FULL_MASK, mbar_wait(&o_full[i & 1], (uint32_t)(i >> 1) & 1, a.err))) {
                s_abort = 1;
                break;
            }
            tc_fence_after();
#pragma unroll
            for (int c0 = 0; c0 < HEAD_DIM; c0 += 32) {
                float v[32];
                tmem_ld32(tmem + lane_base + TM_O + (uint32_t)(i & 1) * HEAD_DIM + c0, v);
#pragma unroll
                for (int e = 0; e < 32; ++e) o[c0 + e] = o[c0 + e] * corr + v[e];
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 4) tmem_dealloc(tmem, TM_COLS);
    if (s_abort) return;  // error word set

    // ---- results: rows of this tile ----
    const int r = row0 + tid;
    auto put = [&](const float* v) {  // 64 outputs of this row and head
        if (a.out) {
            float4* dst = reinterpret_cast<float4*>(a.out + (size_t)r * a.ldo + h * HEAD_DIM);
#pragma unroll
            for (int c = 0; c < HEAD_DIM / 4; ++c) dst[c] = make_float4(v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
        }
        if (a.out_hi) {
            uint4* dh = reinterpret_cast<uint4*>(a.out_hi + (size_t)r * a.ldb + h * HEAD_DIM);
            uint4* dl = reinterpret_cast<uint4*>(a.out_lo + (size_t)r * a.ldb + h * HEAD_DIM);
#pragma unroll
            for (int c = 0; c < HEAD_DIM / 8; ++c) split8(v + 8 * c, dh[c], dl[c]);
        }
    };
    const bool row_on = tid < PA_ROWS && r < a.rows;
    const bool active = row_on && s_seq[tid] >= 0;
    if (S == 1) {
        if (active) {
#pragma unroll
            for (int c = 0; c < HEAD_DIM; ++c) o[c] /= l_run;
            put(o);
        } else if (row_on && a.out_hi) {
#pragma unroll
            for (int c = 0; c < HEAD_DIM; ++c) o[c] = 0.f;
            put(o);
        }
        return;
    }
    float* part = a.ws_part + (((size_t)(tile * H + h) * S + sp) * PA_ROWS) * PA_PART;
    if (tid < PA_ROWS) {
        float* pj = part + (size_t)tid * PA_PART;
        pj[0] = m_run;
        pj[1] = l_run;
#pragma unroll
        for (int c = 0; c < HEAD_DIM; c += 4)
            *reinterpret_cast<float4*>(pj + 4 + c) = make_float4(o[c], o[c + 1], o[c + 2], o[c + 3]);
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) s_last = atomicAdd(a.ws_count + tile * H + h, 1) == S - 1;
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    if (tid == 0) a.ws_count[tile * H + h] = 0;
    if (!row_on) return;
    if (!active) {
        if (a.out_hi) {
#pragma unroll
            for (int c = 0; c < HEAD_DIM; ++c) o[c] = 0.f;
            put(o);
        }
        return;
    }
    // merge the splits in split order: M = max m_s, L = sum exp(m_s - M) l_s, out = sum exp(m_s - M) o_s / L
    const float* base = a.ws_part + ((size_t)(tile * H + h) * S * PA_ROWS + tid) * PA_PART;
    const size_t sstride = (size_t)PA_ROWS * PA_PART;
    float M = -INFINITY;
    for (int s = 0; s < S; ++s) M = fmaxf(M, __ldcg(base + s * sstride));
    float L = 0.f;
#pragma unroll
    for (int c = 0; c < HEAD_DIM; ++c) o[c] = 0.f;
    for (int s = 0; s < S; ++s) {
        const float* ps = base + s * sstride;
        const float ms = __ldcg(ps);
        const float w = ms == -INFINITY ? 0.f : expf(ms - M);
        L = fmaf(w, __ldcg(ps + 1), L);
#pragma unroll
        for (int c = 0; c < HEAD_DIM; c += 4) {
            const float4 v = __ldcg(reinterpret_cast<const float4*>(ps + 4 + c));
            o[c] = fmaf(w, v.x, o[c]);
            o[c + 1] = fmaf(w, v.y, o[c + 1]);
            o[c + 2] = fmaf(w, v.z, o[c + 2]);
            o[c + 3] = fmaf(w, v.w, o[c + 3]);
        }
    }
#pragma unroll
    for (int c = 0; c < HEAD_DIM; ++c) o[c] /= L;
    put(o);
}

}  // namespace

size_t attn_tc_workspace_floats(int tiles, int n_heads, int n_splits) {
    return (size_t)tiles * n_heads * n_splits * PA_ROWS * PA_PART;
}

int attn_tc_tiles(int rows) { return (rows + PA_ROWS - 1) / PA_ROWS; }

int attn_tc_splits_for(int tiles, int n_heads, int max_keys, int num_sms) {
    const int key_tiles = (max_keys + PA_KEYS - 1) / PA_KEYS;
    int s = num_sms / std::max(1, tiles * n_heads);
    return std::max(1, std::min(s, key_tiles));
}

cudaError_t launch_attention_tc(const AttnArgs& a, cudaStream_t s, bool pdl) {
    if (a.rows < 1 || a.n_splits < 1 || a.n_splits > 0xffff || !a.kv_swizzled || (a.page_size & 7) ||
        PA_KEYS % a.page_size || (a.ldq & 3) || (a.out && (a.ldo & 3)) || (a.out_hi && (a.ldb & 7)) ||
        (reinterpret_cast<uintptr_t>(a.q) & 15))
        return cudaErrorInvalidValue;
    cudaError_t e = ensure_kernel_smem(reinterpret_cast<const void*>(attn_tc_kernel), PA_SMEM);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.n_splits, a.n_heads, attn_tc_tiles(a.rows));
    cfg.blockDim = dim3(PA_THREADS);
    cfg.dynamicSmemBytes = PA_SMEM;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, attn_tc_kernel, a);
}

}  // namespace mtp
