// attention.cu -- causal attention of the fed rows over the paged bf16 KV cache
// (the attention of each block, Sec. III-A), split along the key axis.
//
// Grid (split, head, group).  A group is the rows of one slot (the n tokens
// fed this step, or a prefill chunk).  Each CTA takes a contiguous range of
// pages of its slot, stages their keys and values for its head in shared
// memory, and runs a per-row online softmax over them; partial results
// (max, sum, unnormalised output) of the splits are merged with a log-sum-exp
// by the CTA that finishes last (an atomic counter per group and head, reset
// by that CTA), so no second kernel is needed.
//
// Under programmatic dependent launch the pages that hold only keys cached by
// earlier steps are fetched with cp.async.bulk before griddepcontrol.wait;
// the pages touched by this step's appends are read after it.
#include <math.h>

#include <cstdio>
#include <mutex>

#include "common.cuh"
#include "kernels.cuh"
#include "mtp.h"

namespace mtp {
namespace {

constexpr int ATT_THREADS = 256;
constexpr int ATT_KEYS = 256;    // keys staged per batch: 32 KB of keys + 32 KB of values
constexpr int RPG = MAX_ROWS;    // rows per group, upper bound
constexpr int PART = 2 + HEAD_DIM;  // (max, sum, out[64]) per row and split
constexpr int MAX_SPLITS = 32;     // one warp lane per split in the merge
static_assert(HEAD_DIM == 64, "score scale 0.125 assumes 64-wide heads");

__device__ __forceinline__ void load_page_block(__nv_bfloat16* dst, const __nv_bfloat16* src, int elems) {
    const uint4* s = reinterpret_cast<const uint4*>(src);
    uint4* d = reinterpret_cast<uint4*>(dst);
    for (int i = threadIdx.x; i < elems / 8; i += ATT_THREADS) d[i] = s[i];
}

__global__ void __launch_bounds__(ATT_THREADS, 2) attn_kernel(const AttnArgs a) {
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ uint64_t bar;
    __shared__ int s_pos[RPG];
    __shared__ int s_act[RPG];
    __shared__ int s_rseq[RPG];
    __shared__ int s_seq, s_ktot, s_pre, s_last;

    const int sp = blockIdx.x, h = blockIdx.y, g = blockIdx.z;
    TraceEnd trace_guard(a.trace);
    const int H = a.n_heads, P = a.page_size, S = a.n_splits;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    __nv_bfloat16* Ks = reinterpret_cast<__nv_bfloat16*>(smem);
    __nv_bfloat16* Vs = Ks + ATT_KEYS * HEAD_DIM;
    float* qs = reinterpret_cast<float*>(Vs + ATT_KEYS * HEAD_DIM);  // [RPG][64], pre-scaled
    float* Ps = qs + RPG * HEAD_DIM;                                  // [RPG][ATT_KEYS]
    const int pages_per_batch = ATT_KEYS / P;
    const long long kv_head_off = (long long)h * P * HEAD_DIM;
    const long long v_off = (long long)H * P * HEAD_DIM;

    if (tid == 0) {
        mbar_init(&bar, 1);
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
            int pre_end = min(min(pg1, pg0 + pages_per_batch), old_len / P);
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
    if (seq < 0) {  // nothing to do for this group (no split of it counts)
        if (n_pre > 0) mbar_wait(&bar, 0, a.err);
        return;
    }

    const int n_pg = (K_tot + P - 1) / P;
    const int pps = (n_pg + S - 1) / S;
    const int pg0 = sp * pps, pg1 = min(n_pg, pg0 + pps);

    for (int i = tid; i < RPG * HEAD_DIM; i += ATT_THREADS) {
        const int j = i / HEAD_DIM, dd = i % HEAD_DIM;
        qs[i] = s_act[j] ? a.q[(size_t)(g * rpg + j) * a.ldq + h * HEAD_DIM + dd] * 0.125f : 0.f;  // 1/sqrt(64)
    }

    float m_run = -INFINITY, l_run = 0.f, acc0 = 0.f, acc1 = 0.f;  // warp j = row j, lane: dims 2l, 2l+1
    const int row_j = warp;
    const bool row_on = warp < RPG && s_act[min(warp, RPG - 1)];
    const int pos_j = row_on ? s_pos[warp] : -1;

    for (int bp = pg0; bp < pg1; bp += pages_per_batch) {
        const int nb = min(pages_per_batch, pg1 - bp);
        const int nk = nb * P;
        const int first_plain = (bp == pg0) ? n_pre : 0;
        for (int p = first_plain; p < nb; ++p) {
            const int phys = a.block_table[(size_t)seq * a.bt_stride + bp + p];
            if (phys < 0) {  // unreserved page: report, never read
                if (tid == 0 && a.err) atomicOr(a.err, ERR_BOUNDS);
                continue;
            }
            const __nv_bfloat16* base = a.kv_pool + (long long)phys * a.page_elems + a.layer_off + kv_head_off;
            load_page_block(Ks + p * P * HEAD_DIM, base, P * HEAD_DIM);
            load_page_block(Vs + p * P * HEAD_DIM, base + v_off, P * HEAD_DIM);
        }
        if (bp == pg0 && n_pre > 0) {
            bool ok = mbar_wait(&bar, 0, a.err);
            ok = __syncthreads_and(ok) != 0;
            if (!ok) {  // error word set; let copies in flight land before leaving
                mbar_wait(&bar, 0, nullptr);
                return;
            }
        }
        __syncthreads();

        // scores: thread t = key t of the batch
        for (int t = tid; t < nk; t += ATT_THREADS) {
            float sc[RPG];
#pragma unroll
            for (int j = 0; j < RPG; ++j) sc[j] = 0.f;
            const int swz = a.kv_swizzled ? (t & 7) : 0;
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                // logical chunk cc of row t; consecutive rows hit different banks either by the
                // rotation (plain pages) or by the stored swizzle (physical chunk cc ^ (t & 7))
                const int cc = a.kv_swizzled ? c : (c + t) & 7;
                const uint4 kr = *reinterpret_cast<const uint4*>(Ks + t * HEAD_DIM + ((cc ^ swz) << 3));
                const float kf[8] = {bf16_lo(kr.x), bf16_hi(kr.x), bf16_lo(kr.y), bf16_hi(kr.y),
                                     bf16_lo(kr.z), bf16_hi(kr.z), bf16_lo(kr.w), bf16_hi(kr.w)};
#pragma unroll
                for (int j = 0; j < RPG; ++j) {
                    const float4 q0 = *reinterpret_cast<const float4*>(qs + j * HEAD_DIM + cc * 8);
                    const float4 q1 = *reinterpret_cast<const float4*>(qs + j * HEAD_DIM + cc * 8 + 4);
                    float s = sc[j];
                    s = fmaf(q0.x, kf[0], s); s = fmaf(q0.y, kf[1], s);
                    s = fmaf(q0.z, kf[2], s); s = fmaf(q0.w, kf[3], s);
                    s = fmaf(q1.x, kf[4], s); s = fmaf(q1.y, kf[5], s);
                    s = fmaf(q1.z, kf[6], s); s = fmaf(q1.w, kf[7], s);
                    sc[j] = s;
                }
            }
            const int kp = bp * P + t;
#pragma unroll
            for (int j = 0; j < RPG; ++j)
                Ps[j * ATT_KEYS + t] = (s_act[j] && kp <= s_pos[j]) ? sc[j] : -INFINITY;
        }
        __syncthreads();

        if (row_on) {
            float* pr = Ps + row_j * ATT_KEYS;
            float bmax = -INFINITY;
            for (int t = lane; t < nk; t += 32) bmax = fmaxf(bmax, pr[t]);
            bmax = warp_max(bmax);
            const float m_new = fmaxf(m_run, bmax);
            if (m_new != -INFINITY) {
                const float corr = expf(m_run - m_new);  // 0 when m_run = -inf
                float lsum = 0.f;
                for (int t = lane; t < nk; t += 32) {
                    const float p = expf(pr[t] - m_new);
                    pr[t] = p;
                    lsum += p;
                }
                lsum = warp_sum(lsum);
                l_run = l_run * corr + lsum;
                acc0 *= corr;
                acc1 *= corr;
                m_run = m_new;
                __syncwarp();
                const int kend = min(nk, pos_j - bp * P + 1);  // keys past the row's position weigh 0
                // dims 2 lane, 2 lane + 1: chunk lane / 4 of the row, stored at (lane / 4) ^ (t & 7) if swizzled
                const int vch = lane >> 2, vin = (2 * lane) & 7;
                float a0[4] = {0.f, 0.f, 0.f, 0.f}, a1[4] = {0.f, 0.f, 0.f, 0.f};
                int t = 0;
                for (; t + 4 <= kend; t += 4) {  // four independent chains
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const float p = pr[t + u];
                        const int tt = t + u;
                        const int col = a.kv_swizzled ? (((vch ^ (tt & 7)) << 3) | vin) : 2 * lane;
                        const uint32_t v2 = *reinterpret_cast<const uint32_t*>(Vs + tt * HEAD_DIM + col);
                        a0[u] = fmaf(p, bf16_lo(v2), a0[u]);
                        a1[u] = fmaf(p, bf16_hi(v2), a1[u]);
                    }
                }
                for (; t < kend; ++t) {
                    const float p = pr[t];
                    const int col = a.kv_swizzled ? (((vch ^ (t & 7)) << 3) | vin) : 2 * lane;
                    const uint32_t v2 = *reinterpret_cast<const uint32_t*>(Vs + t * HEAD_DIM + col);
                    a0[0] = fmaf(p, bf16_lo(v2), a0[0]);
                    a1[0] = fmaf(p, bf16_hi(v2), a1[0]);
                }
                acc0 += (a0[0] + a0[1]) + (a0[2] + a0[3]);
                acc1 += (a1[0] + a1[1]) + (a1[2] + a1[3]);
            }
        }
        __syncthreads();
    }

    float* out_row = a.out + (size_t)(g * rpg + row_j) * a.ldo + h * HEAD_DIM + 2 * lane;
    if (S == 1) {
        if (row_on) {
            out_row[0] = acc0 / l_run;
            out_row[1] = acc1 / l_run;
        }
        return;
    }

    float* part = a.ws_part + (((size_t)(g * H + h) * S + sp) * RPG) * PART;
    if (warp < RPG) {
        float* pj = part + warp * PART;
        if (lane == 0) {
            pj[0] = m_run;
            pj[1] = l_run;
        }
        pj[2 + 2 * lane] = acc0;
        pj[3 + 2 * lane] = acc1;
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) s_last = atomicAdd(a.ws_count + g * H + h, 1) == S - 1;
    __syncthreads();
    if (!s_last) return;
    __threadfence();

    if (row_on) {
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
        for (int s = 0; s < MAX_SPLITS; ++s) {
            o0[s] = s < S ? __ldcg(base + s * sstride + 2 + 2 * lane) : 0.f;
            o1[s] = s < S ? __ldcg(base + s * sstride + 3 + 2 * lane) : 0.f;
        }
        const float M = warp_max(ms);
        const float w = (ms == -INFINITY) ? 0.f : expf(ms - M);
        const float L = warp_sum(w * ls);
        float r0 = 0.f, r1 = 0.f;
#pragma unroll
        for (int s = 0; s < MAX_SPLITS; ++s) {
            const float ws = __shfl_sync(FULL_MASK, w, s);
            r0 = fmaf(ws, o0[s], r0);
            r1 = fmaf(ws, o1[s], r1);
        }
        out_row[0] = r0 / L;
        out_row[1] = r1 / L;
    }
    if (tid == 0) a.ws_count[g * H + h] = 0;
}

}  // namespace

size_t attn_workspace_floats(int groups, int n_heads, int n_splits, int /*rows_per_group*/) {
    return (size_t)groups * n_heads * n_splits * RPG * PART;
}

size_t attn_smem_bytes(int /*page_size*/) {
    return (size_t)2 * ATT_KEYS * HEAD_DIM * 2 + (size_t)RPG * HEAD_DIM * 4 + (size_t)RPG * ATT_KEYS * 4;
}

int attn_splits_for(int groups, int n_heads, int page_size, int max_keys, int num_sms) {
    const int max_pages = (max_keys + page_size - 1) / page_size;
    int s = num_sms / max(1, groups * n_heads);
    s = max(1, min(min(s, max_pages), MAX_SPLITS));
    return s;
}

cudaError_t launch_attention(const AttnArgs& a, int groups, cudaStream_t s, bool pdl) {
    if (a.rows_per_group < 1 || a.rows_per_group > RPG || ATT_KEYS % a.page_size != 0 || a.n_splits < 1)
        return cudaErrorInvalidValue;
    static bool configured = false;
    const size_t smem = attn_smem_bytes(a.page_size);
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        configured = true;
    }
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

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mutex;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device.  The array's
// name is only a host-side stand-in, so the address is looked up once per
// device (with that device current) and remembered.
int scratch_address(void** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return mtp::report_error(MTP_ERR_CUDA, cudaGetErrorString(e));
    if (dev < 0 || dev >= kMaxDevices) return mtp::report_error(MTP_ERR_INVALID, "device index out of range");
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_attention_scratch);
        if (e != cudaSuccess || !p) {
            char msg[256];
            std::snprintf(msg, sizeof(msg), "attention scratch address lookup failed: %s", cudaGetErrorString(e));
            return mtp::report_error(MTP_ERR_CUDA, msg);
        }
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return MTP_OK;
}

}  // namespace

extern "C" MTP_API int mtp_attention_noalloc(const mtp_attention_args* args, void* cuda_stream) {
    mtp::clear_error();
    if (!args) return mtp::report_error(MTP_ERR_INVALID, "attention: null arguments");
    const size_t need = mtp_attention_workspace_bytes(args);
    if (need == 0) return mtp::report_error(MTP_ERR_INVALID, "attention: invalid sizes");
    if (need > MTP_ATTENTION_NOALLOC_SCRATCH_BYTES) {
        char msg[256];
        std::snprintf(msg, sizeof(msg),
                      "attention: this call needs %zu bytes of scratch, the fixed scratch array holds %u", need,
                      (unsigned)MTP_ATTENTION_NOALLOC_SCRATCH_BYTES);
        return mtp::report_error(MTP_ERR_INVALID, msg);
    }
    void* scratch = nullptr;
    const int r = scratch_address(&scratch);
    if (r != MTP_OK) return r;
    // the merge counters follow the 256-byte-aligned partials and must start at zero
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return mtp::report_error(MTP_ERR_CUDA, cudaGetErrorString(e));
    const int groups = (args->rows + args->rows_per_group - 1) / args->rows_per_group;
    const int splits = mtp::attn_splits_for(groups, args->n_heads, args->page_size, args->max_keys, sms);
    const size_t part = (mtp::attn_workspace_floats(groups, args->n_heads, splits, args->rows_per_group) * 4 + 255) &
                        ~(size_t)255;
    e = cudaMemsetAsync(static_cast<char*>(scratch) + part, 0, need - part, static_cast<cudaStream_t>(cuda_stream));
    if (e != cudaSuccess) return mtp::report_error(MTP_ERR_CUDA, cudaGetErrorString(e));
    return mtp_attention(args, scratch, MTP_ATTENTION_NOALLOC_SCRATCH_BYTES, cuda_stream);
}
