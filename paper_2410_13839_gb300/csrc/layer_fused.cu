// layer_fused.cu -- one pre-LN transformer block (Sec. III-A) over <= 8 fed
// rows as two thread-block-cluster kernels.
//
// Kernel A (attention half), grid (CA, H): the CA = 8 CTAs of a cluster serve
// one attention head.
//   1. before the dependency wait: cp.async.bulk of the CTA's 24 of the
//      head's 192 q|k|v weight rows, its d/CA rows of the head's W_o column
//      block, and the cached key/value pages of its key split;
//   2. LN1 + its 24 projection rows -> shared memory; key/value rows are
//      appended to the paged cache (bf16);
//   3. cluster barrier; every CTA gathers the head's q, k, v of the fed rows
//      from its peers' shared memory (DSMEM);
//   4. attention of the fed rows over its split of the keys (online softmax);
//      the keys fed this step come from the gathered rows, the older ones
//      from the cache;
//   5. cluster barrier; the CA partial (max, sum, output) triples are merged
//      (log-sum-exp) from DSMEM, and the CTA applies its rows of W_o to the
//      head's output, adding the result (plus residual and bias, head 0) into
//      the next residual buffer with float atomics.
// Kernel B (MLP), grid = clusters of CB CTAs over the FFN width: each CTA
// takes a slice of FFN rows, computes u = GELU(LN2(x) W1^T + b1) for them and
// the partial u W2^T over all d outputs; the cluster sums its partials in
// DSMEM and adds them (plus residual and bias, cluster 0) into the layer's
// output buffer with float atomics.
//
// Residual buffers rotate in threes so that every atomic target was zeroed
// by the previous kernel: A(l) zeroes B(l)'s target and B(l) zeroes the
// target of A(l + 1).
#include <cooperative_groups.h>
#include <math.h>

#include "common.cuh"
#include "frag.cuh"
#include "kernels.cuh"

namespace cg = cooperative_groups;

namespace mtp {
namespace {

constexpr int CA = 8;                    // CTAs per head (cluster of kernel A)
constexpr int QROWS = 3 * HEAD_DIM / CA;  // projection rows per CTA (24)
constexpr int MAX_PRE_KEYS = 192;         // cached keys per CTA staged before the dependency wait
// dynamic shared memory of kernel A: small enough for two CTAs per SM (16
// clusters of 8 fit at once only so), and for one CTA beside one CTA of kernel B
// (at d = 1024, 4 fed rows: 88.75 + 133.25 KB of the SM's 228), so that under
// programmatic launch each kernel's CTAs start, and copy their weights, while
// the previous kernel still runs
constexpr size_t A_SMEM_CAP = 91136;
constexpr int PARTW = 2 + HEAD_DIM;       // (max, sum, out[64])
using frag::NTHREADS;
using frag::NWARPS;
using namespace frag;

__host__ __device__ inline size_t al128(size_t x) { return (x + 127) & ~(size_t)127; }

// ---- shared-memory layouts (host and device compute the same offsets) ----
struct ALayout {
    size_t wqkv, ks, wo, qkvp, qkvf, part, attn, uni, total;
    size_t xb, red, attn_b, ytile;  // xb and red share W_o's space; attn_b, ytile the union
    int tile;  // keys of the dedicated staging slots (filled before the dependency wait)
    __host__ __device__ ALayout(int d, int wbytes, int mt, int page) {
        const size_t wq_bytes = (size_t)QROWS * d * wbytes, slot_bytes = (size_t)2 * page * HEAD_DIM * 2;
        // dedicated page slots: as many whole pages as keep two CTAs per SM (at most
        // MAX_PRE_KEYS keys), and one at least when the weight area holds no page
        place(d, wbytes, mt, wq_bytes, 0);
        int pages = total < A_SMEM_CAP ? (int)((A_SMEM_CAP - total) / slot_bytes) : 0;
        pages = min(pages, max(1, MAX_PRE_KEYS / page));
        if (wq_bytes < slot_bytes) pages = max(pages, 1);
        tile = pages * page;
        // the q|k|v slice and the dedicated slots are adjacent: after the attention
        // they hold the warps' softmax states [NWARPS][mt][PARTW]
        size_t ks_bytes = (size_t)pages * slot_bytes;
        const size_t merge_bytes = (size_t)NWARPS * mt * PARTW * 4;
        if (wq_bytes + ks_bytes < merge_bytes) ks_bytes = merge_bytes - wq_bytes;
        place(d, wbytes, mt, wq_bytes, ks_bytes);
    }
    __host__ __device__ void place(int d, int wbytes, int mt, size_t wq_bytes, size_t ks_bytes) {
        const int groups = (QROWS * mt + 31) / 32;
        wqkv = 0;
        ks = al128(wqkv + wq_bytes);  // page slots: [keys | values] each
        // W_o's slice arrives after the projection; until then its space holds the
        // bf16 hi/lo inputs and then the warps' tile sums (tensor cores), or the
        // reduce-scatter scratch (fp32)
        wo = al128(ks + ks_bytes);
        xb = wo;
        red = wo;
        size_t xbytes = (size_t)(d / CA) * HEAD_DIM * wbytes;
        const size_t ibytes = (size_t)2 * mt * (d + 8) * 2;
        const size_t rbytes = wbytes == 2 ? (size_t)NWARPS * QROWS * 8 * 4 : (size_t)NWARPS * groups * 32 * 4;
        if (ibytes > xbytes) xbytes = ibytes;
        if (rbytes > xbytes) xbytes = rbytes;
        qkvp = al128(wo + xbytes);
        qkvf = al128(qkvp + (size_t)QROWS * mt * 4);
        part = al128(qkvf + (size_t)3 * HEAD_DIM * mt * 4);
        attn = al128(part + (size_t)mt * PARTW * 4);
        uni = al128(attn + (size_t)mt * HEAD_DIM * 4);
        // output projection: bf16 hi/lo head output, projected rows
        attn_b = uni;
        ytile = al128(attn_b + (size_t)2 * mt * (HEAD_DIM + 8) * 2);
        total = al128(ytile + (size_t)mt * (d / CA) * 4);
    }
};

struct BLayout {
    size_t w1, w2, xb, accs, ub, u, red, ypart, total;
    int rpad;  // FFN rows rounded up to the 16-row MMA step
    __host__ __device__ BLayout(int d, int rows, int wbytes, int mt, int cb) {
        (void)cb;
        const int groups = (rows * mt + 31) / 32;
        rpad = (rows + 15) / 16 * 16;
        w1 = 0;
        w2 = al128(w1 + (size_t)rows * d * wbytes);
        // bf16 hi/lo inputs, then (same space) the warps' tile sums; fp32: the reduce-scatter scratch
        xb = al128(w2 + (size_t)rows * d * wbytes);
        red = xb;
        size_t xbytes = wbytes == 2 ? (size_t)2 * mt * (d + 8) * 2 : 0;
        const size_t rbytes = wbytes == 2 ? (size_t)NWARPS * rows * 8 * 4 : (size_t)NWARPS * groups * 32 * 4;
        if (rbytes > xbytes) xbytes = rbytes;
        accs = al128(xb + xbytes);                      // [rows][mt] FFN pre-activations
        ub = al128(accs + (size_t)rows * mt * 4);        // bf16 hi/lo GELU outputs
        u = al128(ub + (size_t)2 * mt * (rpad + 8) * 2);  // fp32 GELU outputs
        size_t end = al128(u + (wbytes == 2 ? 0 : (size_t)rows * mt * 4));
        const size_t ybytes = (size_t)mt * d * 4;
        // the partial outputs reuse W1's space once u is known, when it fits
        if ((size_t)rows * d * wbytes >= ybytes) {
            ypart = w1;
        } else {
            ypart = end;
            end = al128(end + ybytes);
        }
        total = end;
    }
};

// out[row][n] = sum_k W[row][k] x[n][k] ([R][MT]) for the R (<= 64) rows of a weight
// slice in shared memory (rows keyed key0 + row), K split across the 8
// warps.  x is given as bf16 hi and lo parts ([MT][K + 8] each, lo right
// after hi), one MMA each, so the product keeps x to fp32 accuracy.  Each
// warp stores its tile sums in wpart [NWARPS][R][8] (which may overlap x)
// and a second pass adds the warps' partials (no shared-memory atomics).
template <int MT>
__device__ __forceinline__ void mma_rows_ksplit(const void* w, int R, int K, int key0, const __nv_bfloat16* xb,
                                                float* wpart, float* out) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int tiles = (R + 15) / 16;
    const int kslice = K / NWARPS;
    const uint32_t wb = smem_addr(w), xbase = smem_addr(xb);
    const int xstride = (K + 8) * 2, row_bytes = K * 2;
    const int brow = (lane & 7) < MT ? (lane & 7) : 0;  // tokens past MT repeat token 0 (ignored)
    const int bhalf = (lane >> 3) & 1;
    const int arow = lane & 15, ahalf = lane >> 4;
    float acc[4][4], accl[4][4];  // hi and lo products in separate chains
#pragma unroll
    for (int t = 0; t < 4; ++t)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[t][i] = accl[t][i] = 0.f;
    const uint32_t xlo = (uint32_t)MT * xstride;
#pragma unroll 2
    for (int k0 = warp * kslice; k0 < (warp + 1) * kslice; k0 += 16) {
        uint32_t bh[2], bl[2];
        ldsm_x2(bh, xbase + brow * xstride + (k0 + bhalf * 8) * 2);
        ldsm_x2(bl, xbase + xlo + brow * xstride + (k0 + bhalf * 8) * 2);
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            if (t < tiles) {
                const int row = min(t * 16 + arow, R - 1);
                uint32_t a[4];
                ldsm_x4(a, wchunk(wb, row, row_bytes, (k0 >> 3) + ahalf, key0 + row));
                mma_bf16(acc[t], a, bh);
                mma_bf16(accl[t], a, bl);
            }
        }
    }
#pragma unroll
    for (int t = 0; t < 4; ++t)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[t][i] += accl[t][i];
    __syncthreads();  // every warp is done with x
    const int g = lane >> 2, c2 = (lane & 3) * 2;
    float* mine = wpart + (size_t)warp * R * 8;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
        if (t >= tiles) continue;
        const int r0 = t * 16 + g, r1 = r0 + 8;
        if (r0 < R) *reinterpret_cast<float2*>(mine + r0 * 8 + c2) = make_float2(acc[t][0], acc[t][1]);
        if (r1 < R) *reinterpret_cast<float2*>(mine + r1 * 8 + c2) = make_float2(acc[t][2], acc[t][3]);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < R * MT; i += NTHREADS) {
        const int j = (i / MT) * 8 + i % MT;
        float y = 0.f;
#pragma unroll
        for (int w2 = 0; w2 < NWARPS; ++w2) y += wpart[(size_t)w2 * R * 8 + j];
        out[i] = y;
    }
}

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

// out[n * R + row] = sum_k W[row][k] x[n][k] for the R rows (R / 16 tiles, one
// warp per tile at a time) of a weight slice with short K (whole K per warp).
// x: bf16 hi and lo parts [MT][K + 8] each (lo right after hi); rows keyed key0 + row.
template <int MT>
__device__ __forceinline__ void mma_rows_tiles(const void* w, int R, int K, int key0, const __nv_bfloat16* xb,
                                               float* out) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t wb = smem_addr(w), xbase = smem_addr(xb);
    const int xstride = (K + 8) * 2, row_bytes = K * 2;
    const int brow = (lane & 7) < MT ? (lane & 7) : 0;
    const int bhalf = (lane >> 3) & 1;
    const int arow = lane & 15, ahalf = lane >> 4;
    const int g = lane >> 2, c2 = (lane & 3) * 2;
    for (int t = warp; t * 16 < R; t += NWARPS) {
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
        const int row = min(t * 16 + arow, R - 1);
        for (int k0 = 0; k0 < K; k0 += 16) {
            uint32_t a[4], bh[2], bl[2];
            ldsm_x2(bh, xbase + brow * xstride + (k0 + bhalf * 8) * 2);
            ldsm_x2(bl, xbase + MT * xstride + brow * xstride + (k0 + bhalf * 8) * 2);
            ldsm_x4(a, wchunk(wb, row, row_bytes, (k0 >> 3) + ahalf, key0 + row));
            mma_bf16(acc, a, bh);
            mma_bf16(acc, a, bl);
        }
        const int r0 = t * 16 + g, r1 = r0 + 8;
        if (c2 < MT) {
            if (r0 < R) out[c2 * R + r0] = acc[0];
            if (r1 < R) out[c2 * R + r1] = acc[2];
        }
        if (c2 + 1 < MT) {
            if (r0 < R) out[(c2 + 1) * R + r0] = acc[1];
            if (r1 < R) out[(c2 + 1) * R + r1] = acc[3];
        }
    }
}

// y[n * C + col] = sum_f W[f][col] u[n][f] over the R FFN rows f of a slice
// stored [R][C] (rows keyed key0 + f): the MMA's A operand is W transposed,
// loaded with ldmatrix.trans.  u: bf16 hi and lo parts [MT][rpad + 8] each
// (lo right after hi), zero for f >= R.
template <int MT>
__device__ __forceinline__ void mma_cols_trans(const void* w, int R, int rpad, int C, int key0, const __nv_bfloat16* ub,
                                               float* y) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t wb = smem_addr(w), ubase = smem_addr(ub);
    const int ustride = (rpad + 8) * 2, row_bytes = C * 2;
    const int brow = (lane & 7) < MT ? (lane & 7) : 0;
    const int bhalf = (lane >> 3) & 1;
    const int g = lane >> 2, c2 = (lane & 3) * 2;
    const int ksteps = rpad / 16;  // <= 4
    uint32_t bh[4][2], bl[4][2];
#pragma unroll
    for (int ks = 0; ks < 4; ++ks)
        if (ks < ksteps) {
            ldsm_x2(bh[ks], ubase + brow * ustride + (ks * 16 + bhalf * 8) * 2);
            ldsm_x2(bl[ks], ubase + MT * ustride + brow * ustride + (ks * 16 + bhalf * 8) * 2);
        }
    // ldmatrix.trans lanes: f row = k0 + (lane & 7) + 8 * (lane >> 4), column chunk + ((lane >> 3) & 1)
    const int fl = (lane & 7) + ((lane >> 4) << 3), chalf = (lane >> 3) & 1;
    for (int t = warp; t * 16 < C; t += NWARPS) {
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
            if (ks >= ksteps) continue;
            const int f = min(ks * 16 + fl, R - 1);
            uint32_t a[4];
            ldsm_x4_t(a, wchunk(wb, f, row_bytes, t * 2 + chalf, key0 + f));
            mma_bf16(acc, a, bh[ks]);
            mma_bf16(acc, a, bl[ks]);
        }
        const int col0 = t * 16 + g, col1 = col0 + 8;
        if (c2 < MT) {
            y[c2 * C + col0] = acc[0];
            y[c2 * C + col1] = acc[2];
        }
        if (c2 + 1 < MT) {
            y[(c2 + 1) * C + col0] = acc[1];
            y[(c2 + 1) * C + col1] = acc[3];
        }
    }
}

// out[row * MT + m] = sum_k W[row, k] x[m, k] for rows < R of the weight
// slice in shared memory (row-major, K columns); red = NWARPS x groups x 32.
template <typename WT, int MT>
__device__ __forceinline__ void project_rows(const WT* wsm, int R, int K, const RowRegs<MT>& x, float* red,
                                             float* out) {
    constexpr int G = 32 / MT;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int Kw = K / NWARPS;
    const int ngroups = (R + G - 1) / G;
    const bool valid = lane * 4 < Kw;
    const int k = warp * Kw + lane * 4;
    for (int g = 0; g < ngroups; ++g) {
        float acc[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) acc[i] = 0.f;
        if (valid) {
#pragma unroll
            for (int r = 0; r < G; ++r) {
                const int row = g * G + r;
                if (row < R) {
                    float w[4];
                    load4(wsm + (size_t)row * K + k, w);
#pragma unroll
                    for (int m = 0; m < MT; ++m) {
                        float t = acc[r * MT + m];
                        t = fmaf(w[0], x.v[m][0], t);
                        t = fmaf(w[1], x.v[m][1], t);
                        t = fmaf(w[2], x.v[m][2], t);
                        t = fmaf(w[3], x.v[m][3], t);
                        acc[r * MT + m] = t;
                    }
                }
            }
        }
        red[(warp * ngroups + g) * 32 + lane] = reduce_scatter32(acc, lane);
    }
    __syncthreads();
    for (int o = threadIdx.x; o < R * MT; o += NTHREADS) {
        const int g = o / 32, l = o % 32;
        float y = 0.f;
#pragma unroll
        for (int w = 0; w < NWARPS; ++w) y += red[(w * ngroups + g) * 32 + l];
        out[o] = y;
    }
    __syncthreads();
}

__device__ __forceinline__ void zero_slice(float* buf, size_t n, int part, int parts) {
    if (!buf) return;
    const size_t per = (n + parts - 1) / parts;
    const size_t b = (size_t)part * per, e = min(n, b + per);
    for (size_t i = b + threadIdx.x; i < e; i += NTHREADS) buf[i] = 0.f;
}

// Slot and position of fed row r of this pass, from state left by earlier
// steps only (the same rule the embedding applies), so it is known before
// the dependency wait.
__device__ __forceinline__ void plan_row(const LayerArgs& a, int r, int& seq, int& pos) {
    seq = -1;
    pos = -1;
    if (r >= a.M) return;
    if (a.plan == PLAN_DEVICE) {
        const int g = r / a.rows_per_group, j = r % a.rows_per_group;
        const int b = a.seq_base + g;
        if (b < a.slots) {  // one round of independent loads
            const int act = a.active[b], dn = a.done[b], nw = a.seq_new[b], len = a.seq_len[b];
            if (act && !dn && j < nw) {
                seq = b;
                pos = len + j;
            }
        }
    } else if (r < a.val_new) {
        seq = a.val_seq;
        pos = a.val_old + r;
    }
}

// Bulk copies of cached pages bp + first .. bp + nb - 1 of sequence seq into
// slots first .. nb - 1 (the first n_ded slots in the dedicated area, the
// rest in the free weight area), on barrier `bar`.  One thread calls it;
// returns whether anything was requested.
__device__ __forceinline__ int issue_pages(const LayerArgs& a, int seq, int bp, int first, int nb, int slot_elems,
                                           long long kv_head, long long v_off, __nv_bfloat16* ks,
                                           __nv_bfloat16* wq_slots, int n_ded, uint64_t* bar) {
    const int P = a.page_size;
    uint32_t bytes = 0;
    for (int p = first; p < nb; ++p)
        if (a.block_table[(size_t)seq * a.bt_stride + bp + p] >= 0) bytes += (uint32_t)slot_elems * 2;
    if (!bytes) return 0;
    fence_proxy_async();  // the slots were last read by this CTA's threads
    mbar_arrive_expect_tx(bar, bytes);
    for (int p = first; p < nb; ++p) {
        const int phys = a.block_table[(size_t)seq * a.bt_stride + bp + p];
        if (phys < 0) {
            atomicOr(a.err, ERR_BOUNDS);
            continue;
        }
        __nv_bfloat16* dst = p < n_ded ? ks + (size_t)p * slot_elems : wq_slots + (size_t)(p - n_ded) * slot_elems;
        const __nv_bfloat16* base = a.kv_pool + (long long)phys * a.page_elems + a.layer_off + kv_head;
        bulk_copy_g2s(dst, base, (uint32_t)P * HEAD_DIM * 2, bar);
        bulk_copy_g2s(dst + P * HEAD_DIM, base + v_off, (uint32_t)P * HEAD_DIM * 2, bar);
    }
    return 1;
}

// ============================================================ kernel A ====

template <typename WT, int MT>
__global__ void __cluster_dims__(CA, 1, 1) __launch_bounds__(NTHREADS, 2) attn_block_kernel(const LayerArgs a) {
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ uint64_t bar;
    __shared__ float ln_part[2 * NWARPS][MT];
    __shared__ float ln_stat[2][MT];
    __shared__ int s_seq[MT], s_pos[MT], s_page[MT];
    __shared__ int s_gseq[MT], s_gold[MT], s_gktot[MT];
    __shared__ int s_pre, s_armed;
    __shared__ uint64_t bar_o;  // W_o slice, requested after the projection
    __shared__ float s_scale[NWARPS][MT];
    TraceEnd trace_guard(a.trace);
    cg::cluster_group cluster = cg::this_cluster();

    const int s = blockIdx.x, h = blockIdx.y;  // split (cluster rank) and head
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int d = a.d, H = a.n_heads, P = a.page_size;
    const int orows = d / CA;  // W_o rows of this CTA
    const ALayout L(d, sizeof(WT), MT, P);
    const int ATT_TILE = L.tile;
    WT* wqkv = reinterpret_cast<WT*>(smem + L.wqkv);
    WT* wo = reinterpret_cast<WT*>(smem + L.wo);
    __nv_bfloat16* Ks = reinterpret_cast<__nv_bfloat16*>(smem + L.ks);
    float* qkvp = reinterpret_cast<float*>(smem + L.qkvp);  // [QROWS][MT]
    float* qkvf = reinterpret_cast<float*>(smem + L.qkvf);  // [192][MT]
    float* part = reinterpret_cast<float*>(smem + L.part);  // [MT][PARTW]
    float* attn = reinterpret_cast<float*>(smem + L.attn);  // [MT][64]
    float* red = reinterpret_cast<float*>(smem + L.red);
    constexpr bool BF = sizeof(WT) == 2;                    // bf16 weights: tensor-core projections
    __nv_bfloat16* xb = reinterpret_cast<__nv_bfloat16*>(smem + L.xb);
    const long long kv_head = (long long)h * P * HEAD_DIM;
    const long long v_off = (long long)H * P * HEAD_DIM;
    const int rpg = a.rows_per_group;
    // page slots: the dedicated staging area, then the q|k|v weight area, free after the projection
    const int slot_elems = 2 * P * HEAD_DIM;  // keys then values of one page
    const int n_ded = ATT_TILE / P;
    const int n_slots = n_ded + (int)((size_t)QROWS * d * sizeof(WT) / ((size_t)slot_elems * 2));
    __nv_bfloat16* const wq_slots = reinterpret_cast<__nv_bfloat16*>(smem + L.wqkv);

    // ---- 1. before the wait: fed rows, weights, cached keys/values ----
    if (tid < MT) {
        int seq, pos;
        plan_row(a, tid, seq, pos);
        s_seq[tid] = seq;
        s_pos[tid] = pos;
        s_page[tid] = seq >= 0 ? a.block_table[(size_t)seq * a.bt_stride + pos / P] : -1;
    }
    if (tid == 0) {
        mbar_init(&bar, 1);
        mbar_init(&bar_o, 1);
        fence_barrier_init();
        s_pre = 0;
    }
    __syncthreads();
    if (tid < MT) {  // per group: slot, first fed position (= cached length) and key count
        const int g = tid;
        int seq = -1, kmin = 1 << 30, kmax = 0;
        for (int j = 0; j < rpg && g * rpg + j < MT; ++j) {
            const int r = g * rpg + j;
            if (s_seq[r] >= 0) {
                seq = s_seq[r];
                kmin = min(kmin, s_pos[r]);
                kmax = max(kmax, s_pos[r] + 1);
            }
        }
        s_gseq[g] = seq;
        s_gold[g] = seq >= 0 ? kmin : 0;
        s_gktot[g] = kmax;
    }
    __syncthreads();
    if (tid == 0) {
        const uint32_t wq = (uint32_t)QROWS * d * sizeof(WT);
        uint32_t kvb = 0;
        int n_pre = 0, pg0 = 0;
        const int seq = s_gseq[0];
        if (seq >= 0) {  // group 0: pages of this split holding only keys of earlier steps
            const int old_len = s_gold[0];
            const int n_pg = (s_gktot[0] + P - 1) / P;
            const int pps = (n_pg + CA - 1) / CA;
            pg0 = s * pps;
            const int pg1 = min(n_pg, pg0 + pps);
            (void)old_len;  // rows of the fed keys are filled in shared memory after the copy
            int pre_end = min(pg1, pg0 + ATT_TILE / P);
            for (int p = pg0; p < pre_end; ++p)
                if (a.block_table[(size_t)seq * a.bt_stride + p] < 0) pre_end = p;
            n_pre = max(0, pre_end - pg0);
            kvb = 2u * (uint32_t)n_pre * P * HEAD_DIM * 2;
        }
        mbar_arrive_expect_tx(&bar, wq + kvb);
        const char* srcq = reinterpret_cast<const char*>(a.wqkv) + ((size_t)h * 3 * HEAD_DIM + s * QROWS) * d * sizeof(WT);
        const uint64_t pol = l2_evict_first_policy();
        for (uint32_t off = 0; off < wq; off += 32768)
            bulk_copy_g2s_hint(smem + L.wqkv + off, srcq + off, min(32768u, wq - off), &bar, pol);
        for (int i = 0; i < n_pre; ++i) {
            const int phys = a.block_table[(size_t)seq * a.bt_stride + pg0 + i];
            const __nv_bfloat16* base = a.kv_pool + (long long)phys * a.page_elems + a.layer_off + kv_head;
            bulk_copy_g2s(Ks + (size_t)i * 2 * P * HEAD_DIM, base, (uint32_t)P * HEAD_DIM * 2, &bar);
            bulk_copy_g2s(Ks + (size_t)i * 2 * P * HEAD_DIM + P * HEAD_DIM, base + v_off, (uint32_t)P * HEAD_DIM * 2,
                          &bar);
        }
        s_pre = n_pre;
    } else if (tid == 32) {  // L2 prefetches, issued beside the copies above
        const uint32_t wq = (uint32_t)QROWS * d * sizeof(WT);
        const uint32_t wob = (uint32_t)orows * HEAD_DIM * sizeof(WT);
        const size_t offq = ((size_t)h * 3 * HEAD_DIM + s * QROWS) * d * sizeof(WT);
        const size_t offo = ((size_t)h * d + s * orows) * HEAD_DIM * sizeof(WT);
        prefetch_l2(reinterpret_cast<const char*>(a.wo) + offo, wob);  // copied after the projection
        const int seq = s_gseq[0];
        if (seq >= 0) {  // the split's cached pages past the staged ones (copied to shared memory later)
            const int n_pg = (s_gktot[0] + P - 1) / P;
            const int pps = (n_pg + CA - 1) / CA;
            const int pg0 = s * pps, pg1 = min(n_pg, pg0 + pps);
            for (int p = pg0 + ATT_TILE / P; p < pg1; ++p) {
                const int phys = a.block_table[(size_t)seq * a.bt_stride + p];
                if (phys < 0) continue;
                const __nv_bfloat16* base = a.kv_pool + (long long)phys * a.page_elems + a.layer_off + kv_head;
                prefetch_l2(base, (uint32_t)P * HEAD_DIM * 2);
                prefetch_l2(base + v_off, (uint32_t)P * HEAD_DIM * 2);
            }
        }
        if (a.next_w_a) {  // the next layer's slices of the same weights, into L2
            prefetch_l2(reinterpret_cast<const char*>(a.next_w_a) + offq, wq);
            prefetch_l2(reinterpret_cast<const char*>(a.next_w_b) + offo, wob);
        }
    }
    float gam[4], bet[4], bq[1] = {0.f};
    {
        const int Kw = d / NWARPS;
        if (lane * 4 < Kw) {
            load4(a.ln_g + warp * Kw + lane * 4, gam);
            load4(a.ln_b + warp * Kw + lane * 4, bet);
        } else {
#pragma unroll
            for (int i = 0; i < 4; ++i) gam[i] = bet[i] = 0.f;
        }
        if (tid < QROWS * MT) bq[0] = __ldg(a.bqkv + h * 3 * HEAD_DIM + s * QROWS + tid / MT);
    }

    pdl_launch_dependents();
    pdl_wait();
    trace_wait(a.trace);

    // ---- 2. inputs: LN1, projection ----
    RowRegs<MT> xr;
    load_rows<MT>(a.x_in, d, a.M, d, xr);
    constexpr int RES_N = (MT * (1024 / CA) + NTHREADS - 1) / NTHREADS;  // W_o outputs per thread
    float resr[RES_N];  // residual + bias of this thread's W_o outputs (head 0 adds them)
#pragma unroll
    for (int k = 0; k < RES_N; ++k) {
        const int o = tid + k * NTHREADS, m = o / orows, f = s * orows + o % orows;
        resr[k] = h == 0 && o < orows * MT && m < a.M ? a.x_in[(size_t)m * d + f] + a.bo[f] : 0.f;
    }
    zero_slice(a.x_zero, (size_t)MAX_ROWS * d, h * CA + s, H * CA);
    layer_norm_rows<MT>(xr, d, gam, bet, a.ln_eps, ln_part, ln_stat);
    if (BF) {
        store_rows_split<MT>(xr, d, xb);
    }
    trace_mark(a.trace, 0);  // inputs loaded, LN1 done
    bool ok = mbar_wait(&bar, 0, a.err);
    ok = __syncthreads_and(ok) != 0;
    if (!ok) {
        mbar_wait(&bar, 0, nullptr);
        cluster.sync();
        cluster.sync();
        cluster.sync();
        return;
    }
    trace_mark(a.trace, 1);  // weights and cached keys in shared memory
    if (BF) {
        mma_rows_ksplit<MT>(wqkv, QROWS, d, 0, xb, red, qkvp);
        __syncthreads();
    } else {
        project_rows<WT, MT>(wqkv, QROWS, d, xr, red, qkvp);
    }
    // q|k|v rows with bias (QROWS * MT <= NTHREADS: one per thread), released to the cluster
    const bool has_row = tid < QROWS * MT;
    const float yrow = has_row ? qkvp[tid] + bq[0] : 0.f;
    if (has_row) qkvp[tid] = yrow;
    cluster_arrive_release();
    if (has_row) {
        const int row = s * QROWS + tid / MT, m = tid % MT;  // row within the head's q|k|v
        if (row >= HEAD_DIM && s_seq[m] >= 0) {               // key or value: append to the cache
            const int sec = row / HEAD_DIM, dd = row % HEAD_DIM;
            const int page = s_page[m];
            if (page < 0) {
                atomicOr(a.err, ERR_BOUNDS);
            } else {
                const int t = s_pos[m] % P;  // key row of the page; its 16-byte chunks are stored swizzled
                const long long idx = (long long)page * a.page_elems + a.layer_off + (sec - 1) * v_off + kv_head +
                                      (long long)t * HEAD_DIM + kv_col(t, dd);
                reinterpret_cast<uint16_t*>(a.kv_pool)[idx] = f32_to_bf16_bits(yrow);
            }
        }
    }
    if (tid == 0) {  // W_o's slice, and group 0's first batch of cached pages, while the cluster gathers
        fence_proxy_async();  // the spaces were last written and read by this CTA's threads
        const uint32_t wob = (uint32_t)orows * HEAD_DIM * sizeof(WT);
        mbar_arrive_expect_tx(&bar_o, wob);
        bulk_copy_g2s_hint(smem + L.wo,
                           reinterpret_cast<const char*>(a.wo) + ((size_t)h * d + s * orows) * HEAD_DIM * sizeof(WT),
                           wob, &bar_o, l2_evict_first_policy());
        s_armed = 0;
        const int seq = s_gseq[0];
        if (seq >= 0) {
            const int n_pg = (s_gktot[0] + P - 1) / P, pps = (n_pg + CA - 1) / CA;
            const int pg0 = s * pps, pg1 = min(n_pg, pg0 + pps);
            if (pg0 < pg1)
                s_armed = issue_pages(a, seq, pg0, s_pre, min(n_slots, pg1 - pg0), slot_elems, kv_head, v_off, Ks,
                                      wq_slots, n_ded, &bar);
        }
    }
    trace_mark(a.trace, 2);  // projection rows done
    // ---- 3. gather the head's q, k, v of the fed rows from the cluster ----
    cluster_wait();
    trace_mark(a.trace, 3);
    {
        constexpr int PER = (3 * HEAD_DIM * MT + NTHREADS - 1) / NTHREADS;
        float v[PER];
#pragma unroll
        for (int u = 0; u < PER; ++u) {  // issue every remote load before using any
            const int i = tid + u * NTHREADS;
            v[u] = 0.f;
            if (i < 3 * HEAD_DIM * MT) {
                const int row = i / MT;
                v[u] = ld_dsmem(dsmem_addr(qkvp + (row % QROWS) * MT + i % MT, row / QROWS));
            }
        }
#pragma unroll
        for (int u = 0; u < PER; ++u) {
            const int i = tid + u * NTHREADS;
            if (i < 3 * HEAD_DIM * MT)
                qkvf[i] = i / MT >= HEAD_DIM ? __bfloat162float(__float2bfloat16_rn(v[u])) : v[u];  // keys/values as cached
        }
    }
    __syncthreads();

    trace_mark(a.trace, 4);  // gathered
    // ---- 4. attention over this CTA's split of each group's keys ----
    // Flash-attention style on the tensor cores: each warp takes 16-key tiles
    // of a batch with online-softmax state in registers; Q and P enter as
    // bf16 hi + lo pairs (two MMAs), which keeps them to fp32 accuracy.
    // Keys as the MMA's M side: S^T = K Q^T over 16-key tiles (the fed rows' bf16 hi and lo parts
    // as two N = 8 operands) and O^T += V^T P^T (head dims x fed rows; P^T's hi and lo parts into
    // one accumulator).  Lane (g8, c2): keys g8, g8 + 8 of a tile and rows c2, c2 + 1 in S^T; head
    // dims g8, g8 + 8 of each 16-dim block and rows c2, c2 + 1 in O^T.
    const int g8 = lane >> 2, c2 = (lane & 3) * 2;
    bool qon[2];
    int qpos[2], qgrp[2];
#pragma unroll
    for (int j = 0; j < 2; ++j) {
        const int r = c2 + j;
        qon[j] = r < MT && r < a.M && s_seq[min(r, MT - 1)] >= 0;
        qpos[j] = qon[j] ? s_pos[min(r, MT - 1)] : -1;
        qgrp[j] = r / rpg;
    }
    uint32_t qhi[4][2], qlo[4][2];  // B operand of S^T: fed row g8, dims ks * 16 + 8 hh + c2, + 1
    {
        const bool on = g8 < MT && g8 < a.M && s_seq[min(g8, MT - 1)] >= 0;
#pragma unroll
        for (int ks = 0; ks < 4; ++ks)
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
                const int k = ks * 16 + hh * 8 + c2;
                // the query scaled by 1/sqrt(64) (exact in binary)
                const float q0 = on ? qkvf[k * MT + g8] * 0.125f : 0.f;
                const float q1 = on ? qkvf[(k + 1) * MT + g8] * 0.125f : 0.f;
                split_bf16x2(q0, q1, qhi[ks][hh], qlo[ks][hh]);
            }
    }
    float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
    float o[4][4];  // O^T block dp: dims dp * 16 + g8 (0, 1) and + 8 (2, 3), fed rows c2 + (i & 1)
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
        for (int i = 0; i < 4; ++i) o[j][i] = 0.f;
    const int G = (a.M + rpg - 1) / rpg;
    auto slot_keys = [&](int i) -> __nv_bfloat16* {
        return i < n_ded ? Ks + (size_t)i * slot_elems : wq_slots + (size_t)(i - n_ded) * slot_elems;
    };
    uint32_t phase = 1;  // phase 0 of the barrier brought the weights
    bool first_batch = true;
    for (int g = 0; g < G; ++g) {
        const int seq = s_gseq[g], old_len = s_gold[g], K_tot = s_gktot[g];
        if (seq < 0) continue;
        const int n_pg = (K_tot + P - 1) / P;
        const int pps = (n_pg + CA - 1) / CA;
        const int pg0 = s * pps, pg1 = min(n_pg, pg0 + pps);
        for (int bp = pg0; bp < pg1; bp += n_slots) {
            const int nb = min(n_slots, pg1 - bp);
            const int nk = nb * P;
            __syncthreads();  // every reader of the slots is done with the previous batch
            if (!(first_batch && g == 0)) {  // group 0's first batch was requested after the projection
                if (tid == 0) s_armed = issue_pages(a, seq, bp, 0, nb, slot_elems, kv_head, v_off, Ks, wq_slots,
                                                    n_ded, &bar);
                __syncthreads();
            }
            first_batch = false;
            if (s_armed) {
                if (!mbar_wait(&bar, phase & 1, a.err)) mbar_wait(&bar, phase & 1, nullptr);
                ++phase;
            }
            {  // keys fed this step (positions old_len .. K_tot-1 inside this batch), from the gather
                const int k0 = max(old_len, bp * P), k1 = min(K_tot, bp * P + nk);
                for (int i = tid; i < (k1 - k0) * HEAD_DIM; i += NTHREADS) {
                    const int key = k0 + i / HEAD_DIM, dd = i % HEAD_DIM;
                    const int m = g * rpg + (key - old_len);
                    const int t = (key - bp * P) % P;
                    __nv_bfloat16* kp = slot_keys((key - bp * P) / P) + t * HEAD_DIM + kv_col(t, dd);
                    kp[0] = __float2bfloat16_rn(qkvf[(HEAD_DIM + dd) * MT + m]);
                    kp[P * HEAD_DIM] = __float2bfloat16_rn(qkvf[(2 * HEAD_DIM + dd) * MT + m]);
                }
            }
            __syncthreads();
            for (int kt = warp * 16; kt < nk; kt += NWARPS * 16) {
                const int r0 = kt % P;  // first key row of the tile in its page
                const uint32_t kb = smem_addr(slot_keys(kt / P)), vb = kb + P * HEAD_DIM * 2;
                float sh[4] = {0.f, 0.f, 0.f, 0.f}, sl[4] = {0.f, 0.f, 0.f, 0.f};  // hi and lo parts: own chains
                {
                    // A = K rows: matrices (keys 0-7 | 8-15) x (dims 0-7 | 8-15) of the k-step
                    const int key = r0 + (lane & 7) + (((lane >> 3) & 1) << 3), chalf = lane >> 4;
#pragma unroll
                    for (int ks = 0; ks < 4; ++ks) {
                        uint32_t ka[4];
                        ldsm_x4(ka, kb + key * 128 + ((uint32_t)((2 * ks + chalf) ^ (key & 7)) << 4));
                        const uint32_t bh[2] = {qhi[ks][0], qhi[ks][1]}, bl[2] = {qlo[ks][0], qlo[ks][1]};
                        mma_bf16(sh, ka, bh);
                        mma_bf16(sl, ka, bl);
                    }
                }
                // this lane's scores: keys kt + g8 (i = 0, 1) and kt + g8 + 8 (i = 2, 3), fed row c2 + (i & 1)
                float sv[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int kp = bp * P + kt + g8 + (i >> 1) * 8, j = i & 1;
                    const bool vis = qon[j] && qgrp[j] == g && kp <= qpos[j] && kp < K_tot;
                    sv[i] = vis ? sh[i] + sl[i] : -INFINITY;
                }
                float t0 = fmaxf(sv[0], sv[2]), t1 = fmaxf(sv[1], sv[3]);  // over the tile's keys: lanes g8
#pragma unroll
                for (int off = 4; off < 32; off <<= 1) {
                    t0 = fmaxf(t0, __shfl_xor_sync(FULL_MASK, t0, off));
                    t1 = fmaxf(t1, __shfl_xor_sync(FULL_MASK, t1, off));
                }
                const float mn[2] = {fmaxf(m_run[0], t0), fmaxf(m_run[1], t1)};
                float corr[2];
#pragma unroll
                for (int j = 0; j < 2; ++j)
                    corr[j] = mn[j] == -INFINITY ? 1.f : (m_run[j] == -INFINITY ? 0.f : expf(m_run[j] - mn[j]));
                float pv[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) pv[i] = sv[i] == -INFINITY ? 0.f : expf(sv[i] - mn[i & 1]);
                l_run[0] = l_run[0] * corr[0] + (pv[0] + pv[2]);
                l_run[1] = l_run[1] * corr[1] + (pv[1] + pv[3]);
                m_run[0] = mn[0];
                m_run[1] = mn[1];
#pragma unroll
                for (int dp = 0; dp < 4; ++dp) {
                    o[dp][0] *= corr[0];
                    o[dp][1] *= corr[1];
                    o[dp][2] *= corr[0];
                    o[dp][3] *= corr[1];
                }
                // P^T as the B operand: this lane holds rows g8 (keys), columns c2 (fed rows) of each
                // 8 x 8 block; its transpose is the operand's layout (fed row g8, keys c2, c2 + 1)
                uint32_t ph0, pl0, ph1, pl1;
                split_bf16x2(pv[0], pv[1], ph0, pl0);  // keys g8
                split_bf16x2(pv[2], pv[3], ph1, pl1);  // keys g8 + 8
                const uint32_t bph[2] = {movmatrix_trans(ph0), movmatrix_trans(ph1)};
                const uint32_t bpl[2] = {movmatrix_trans(pl0), movmatrix_trans(pl1)};
                // A = V^T: matrices (dims 0-7 | 8-15 of block dp) x (keys 0-7 | 8-15), from the key rows
                const int vkey = r0 + (lane & 7) + ((lane >> 4) << 3), vhalf = (lane >> 3) & 1;
#pragma unroll
                for (int dp = 0; dp < 4; ++dp) {
                    uint32_t va[4];
                    ldsm_x4_t(va, vb + vkey * 128 + ((uint32_t)((2 * dp + vhalf) ^ (vkey & 7)) << 4));
                    mma_bf16(o[dp], va, bph);
                    mma_bf16(o[dp], va, bpl);
                }
            }
        }
    }
    // merge the warps' (max, sum, out) states into part through the weight
    // area (free once every warp is past its last tile): [NWARPS][MT][PARTW]
#pragma unroll
    for (int j = 0; j < 2; ++j)  // each lane summed its own keys; a row's keys span lanes g8
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) l_run[j] += __shfl_xor_sync(FULL_MASK, l_run[j], off);
    __syncthreads();
    float* wst = reinterpret_cast<float*>(smem + L.wqkv);
#pragma unroll
    for (int j = 0; j < 2; ++j) {
        if (c2 + j >= MT) continue;
        float* ws = wst + ((size_t)warp * MT + c2 + j) * PARTW;
        if (g8 == 0) {
            ws[0] = m_run[j];
            ws[1] = l_run[j];
        }
#pragma unroll
        for (int dp = 0; dp < 4; ++dp) {
            ws[2 + dp * 16 + g8] = o[dp][j];
            ws[2 + dp * 16 + g8 + 8] = o[dp][2 + j];
        }
    }
    __syncthreads();
    if (tid < NWARPS * MT) {  // weight of warp w's state in row m: exp(max_w - common max)
        const int w = tid / MT, m = tid % MT;
        float M = -INFINITY;
#pragma unroll
        for (int v = 0; v < NWARPS; ++v) M = fmaxf(M, wst[((size_t)v * MT + m) * PARTW]);
        const float mw = wst[((size_t)w * MT + m) * PARTW];
        s_scale[w][m] = mw == -INFINITY ? 0.f : expf(mw - M);
        if (w == 0) part[m * PARTW] = M;
    }
    __syncthreads();
    for (int i = tid; i < MT * (1 + HEAD_DIM); i += NTHREADS) {
        const int m = i / (1 + HEAD_DIM), c = 1 + i % (1 + HEAD_DIM);
        float y = 0.f;
#pragma unroll
        for (int w = 0; w < NWARPS; ++w) y = fmaf(s_scale[w][m], wst[((size_t)w * MT + m) * PARTW + c], y);
        part[m * PARTW + c] = y;
    }
    __syncthreads();

    trace_mark(a.trace, 5);  // attention partials done
    // ---- 5. merge the splits (DSMEM) and apply this CTA's W_o rows ----
    cluster.sync();
    trace_mark(a.trace, 6);
    const int row_j = warp;  // warp m merges fed row m
    const bool row_on = row_j < MT && row_j < a.M && s_seq[min(row_j, MT - 1)] >= 0;
    if (row_on) {
        float ms = -INFINITY, ls = 0.f, o0[CA], o1[CA];
        const float* mine = part + row_j * PARTW;
        float2 st = make_float2(-INFINITY, 0.f);
        if (lane < CA) st = ld_dsmem2(dsmem_addr(mine, lane));  // (max, sum) of split `lane`
#pragma unroll
        for (int r = 0; r < CA; ++r) {
            const float2 ov = ld_dsmem2(dsmem_addr(mine + 2 + 2 * lane, r));
            o0[r] = ov.x;
            o1[r] = ov.y;
        }
        ms = st.x;
        ls = st.y;
        const float M = warp_max(ms);
        const float w = (ms == -INFINITY) ? 0.f : expf(ms - M);
        const float Lsum = warp_sum(lane < CA ? w * ls : 0.f);
        float r0 = 0.f, r1 = 0.f;
#pragma unroll
        for (int r = 0; r < CA; ++r) {
            const float wr = __shfl_sync(FULL_MASK, w, r);
            r0 = fmaf(wr, o0[r], r0);
            r1 = fmaf(wr, o1[r], r1);
        }
        attn[row_j * HEAD_DIM + 2 * lane] = r0 / Lsum;
        attn[row_j * HEAD_DIM + 2 * lane + 1] = r1 / Lsum;
    } else if (row_j < MT) {
        attn[row_j * HEAD_DIM + 2 * lane] = 0.f;
        attn[row_j * HEAD_DIM + 2 * lane + 1] = 0.f;
    }
    cluster_arrive_relaxed();  // done reading the peers' partials (waited for before exiting)
    __syncthreads();
    bool okw = mbar_wait(&bar_o, 0, a.err);
    okw = __syncthreads_and(okw) != 0;
    if (!okw) {
        mbar_wait(&bar_o, 0, nullptr);
    } else if (BF) {  // head output as bf16 hi/lo, then W_o rows on the tensor cores
        __nv_bfloat16* ab = reinterpret_cast<__nv_bfloat16*>(smem + L.attn_b);  // [MT][64 + 8]
        float* ytile = reinterpret_cast<float*>(smem + L.ytile);                  // [MT][orows]
        for (int i = tid; i < MT * HEAD_DIM; i += NTHREADS) {
            const __nv_bfloat16 hi = __float2bfloat16_rn(attn[i]);
            const int at = (i / HEAD_DIM) * (HEAD_DIM + 8) + i % HEAD_DIM;
            ab[at] = hi;
            ab[MT * (HEAD_DIM + 8) + at] = __float2bfloat16_rn(attn[i] - __bfloat162float(hi));
        }
        __syncthreads();
        mma_rows_tiles<MT>(wo, orows, HEAD_DIM, 0, ab, ytile);
        __syncthreads();
#pragma unroll
        for (int k = 0; k < RES_N; ++k) {
            const int o = tid + k * NTHREADS;
            const int m = o / orows, t = o % orows;  // a warp adds 32 consecutive floats
            if (o >= orows * MT || m >= a.M || s_seq[m] < 0) continue;
            atomicAdd(a.x_out + (size_t)m * d + s * orows + t, ytile[o] + resr[k]);
        }
    } else {
#pragma unroll
        for (int k = 0; k < RES_N; ++k) {
            const int o = tid + k * NTHREADS;
            const int m = o / orows, t = o % orows;  // fed row m, W_o row t: a warp adds 32 consecutive floats
            if (o >= orows * MT || m >= a.M || s_seq[m] < 0) continue;
            const WT* wr = wo + (size_t)t * HEAD_DIM;
            float acc[4] = {0.f, 0.f, 0.f, 0.f};  // four independent chains
#pragma unroll
            for (int c = 0; c < HEAD_DIM / 4; ++c) {
                const int cc = (c + t) & (HEAD_DIM / 4 - 1);  // rotate to spread banks
                float w4[4];
                load4(wr + cc * 4, w4);
                const float4 av = *reinterpret_cast<const float4*>(attn + m * HEAD_DIM + cc * 4);
                float v = acc[c & 3];
                v = fmaf(w4[0], av.x, v);
                v = fmaf(w4[1], av.y, v);
                v = fmaf(w4[2], av.z, v);
                v = fmaf(w4[3], av.w, v);
                acc[c & 3] = v;
            }
            const float y = (acc[0] + acc[1]) + (acc[2] + acc[3]) + resr[k];
            atomicAdd(a.x_out + (size_t)m * d + s * orows + t, y);
        }
    }
    trace_mark(a.trace, 7);  // output projection added
    cluster_wait();  // peers may still read this CTA's shared memory
}

// ============================================================ kernel B ====

template <typename WT, int MT, int CB>
__global__ void __launch_bounds__(NTHREADS, 2) mlp_kernel(const LayerArgs a) {
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ uint64_t bar;
    __shared__ float ln_part[2 * NWARPS][MT];
    __shared__ float ln_stat[2][MT];
    __shared__ int s_act[MT];
    TraceEnd trace_guard(a.trace);
    cg::cluster_group cluster = cg::this_cluster();

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int d = a.d, F = a.d_ffn;
    const int rpc = a.ffn_rows_per_cta;
    const int f0 = blockIdx.x * rpc;
    const int R = max(0, min(rpc, F - f0));
    const int rank = (int)cluster.block_rank();
    const int cols = d / CB;  // output columns this CTA reduces
    const BLayout L(d, rpc, sizeof(WT), MT, CB);
    WT* w1 = reinterpret_cast<WT*>(smem + L.w1);
    WT* w2 = reinterpret_cast<WT*>(smem + L.w2);
    float* u = reinterpret_cast<float*>(smem + L.u);          // [R][MT] (fp32 weights)
    constexpr bool BF = sizeof(WT) == 2;                      // bf16 weights: tensor-core projections
    const int rpad = L.rpad;
    __nv_bfloat16* xb = reinterpret_cast<__nv_bfloat16*>(smem + L.xb);
    float* accs = reinterpret_cast<float*>(smem + L.accs);
    __nv_bfloat16* ub = reinterpret_cast<__nv_bfloat16*>(smem + L.ub);  // hi, lo: [MT][rpad + 8] each
    float* ypart = reinterpret_cast<float*>(smem + L.ypart);  // [MT][d]
    float* red = reinterpret_cast<float*>(smem + L.red);
    const bool first_cluster = blockIdx.x < CB;

    if (tid < MT) {
        int seq, pos;
        plan_row(a, tid, seq, pos);
        s_act[tid] = seq >= 0;
    }
    if (tid == 0) {
        mbar_init(&bar, 1);
        fence_barrier_init();
    }
    __syncthreads();
    if (tid == 0 && R > 0) {
        const uint32_t wb = (uint32_t)R * d * sizeof(WT);
        mbar_arrive_expect_tx(&bar, 2 * wb);
        const size_t off0 = (size_t)f0 * d * sizeof(WT);
        const char* s1 = reinterpret_cast<const char*>(a.w1) + off0;
        const char* s2 = reinterpret_cast<const char*>(a.w2t) + off0;
        const uint64_t pol = l2_evict_first_policy();
        for (uint32_t off = 0; off < wb; off += 32768) {
            bulk_copy_g2s_hint(smem + L.w1 + off, s1 + off, min(32768u, wb - off), &bar, pol);
            bulk_copy_g2s_hint(smem + L.w2 + off, s2 + off, min(32768u, wb - off), &bar, pol);
        }
    } else if (tid == 32 && R > 0 && a.next_w_a) {  // the next layer's slices, into L2
        const uint32_t wb = (uint32_t)R * d * sizeof(WT);
        const size_t off0 = (size_t)f0 * d * sizeof(WT);
        prefetch_l2(reinterpret_cast<const char*>(a.next_w_a) + off0, wb);
        prefetch_l2(reinterpret_cast<const char*>(a.next_w_b) + off0, wb);
    }
    float gam[4], bet[4], b1v[2] = {0.f, 0.f};
    {
        const int Kw = d / NWARPS;
        if (lane * 4 < Kw) {
            load4(a.ln_g + warp * Kw + lane * 4, gam);
            load4(a.ln_b + warp * Kw + lane * 4, bet);
        } else {
#pragma unroll
            for (int i = 0; i < 4; ++i) gam[i] = bet[i] = 0.f;
        }
        for (int k = 0; k < 2; ++k) {
            const int o = tid + k * NTHREADS;
            if (BF) {  // item o = (m, f) of the bf16 GELU output
                const int f = o % rpad;
                if (o < MT * rpad && f < R) b1v[k] = __ldg(a.b1 + f0 + f);
            } else if (o < R * MT) {
                b1v[k] = __ldg(a.b1 + f0 + o / MT);
            }
        }
    }

    pdl_launch_dependents();
    pdl_wait();
    trace_wait(a.trace);

    RowRegs<MT> xr;
    load_rows<MT>(a.x_in, d, a.M, d, xr);
    constexpr int RES_PER = 2;  // residual items per thread kept in registers (MT * cols / 4 <= 512)
    float4 resv[RES_PER];
#pragma unroll
    for (int k = 0; k < RES_PER; ++k) {  // residual and bias of the columns this CTA reduces
        const int i = tid + k * NTHREADS;
        resv[k] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (first_cluster && i < MT * cols / 4) {
            const int m = i / (cols / 4), c = rank * cols + (i % (cols / 4)) * 4;
            if (m < a.M) {
                const float4 xv = *reinterpret_cast<const float4*>(a.x_in + (size_t)m * d + c);
                const float4 bv = *reinterpret_cast<const float4*>(a.b2 + c);
                resv[k] = make_float4(xv.x + bv.x, xv.y + bv.y, xv.z + bv.z, xv.w + bv.w);
            }
        }
    }
    zero_slice(a.x_zero, (size_t)MAX_ROWS * d, blockIdx.x, gridDim.x);
    layer_norm_rows<MT>(xr, d, gam, bet, a.ln_eps, ln_part, ln_stat);
    if (BF) {
        store_rows_split<MT>(xr, d, xb);
    }

    trace_mark(a.trace, 0);  // inputs loaded, LN2 done
    bool ok = R == 0 || mbar_wait(&bar, 0, a.err);
    ok = __syncthreads_and(ok) != 0;
    if (!ok) {
        if (R > 0) mbar_wait(&bar, 0, nullptr);
        cluster.sync();
        cluster.sync();
        return;
    }
    trace_mark(a.trace, 1);  // weights in shared memory
    if (BF) {
        // u = GELU(LN2(x) W1^T + b1) for this CTA's FFN rows, as bf16 [MT][rpad]
        if (R > 0) mma_rows_ksplit<MT>(w1, R, d, f0, xb, red, accs);
        __syncthreads();
        for (int k = 0; k < 2; ++k) {
            const int o = tid + k * NTHREADS;
            if (o >= MT * rpad) continue;
            const int m = o / rpad, f = o % rpad;
            const float v = f < R ? gelu_erf(accs[f * MT + m] + b1v[k]) : 0.f;
            const __nv_bfloat16 hi = __float2bfloat16_rn(v);
            ub[m * (rpad + 8) + f] = hi;
            ub[(MT + m) * (rpad + 8) + f] = __float2bfloat16_rn(v - __bfloat162float(hi));
        }
        __syncthreads();
        trace_mark(a.trace, 2);  // u done
        // partial u W2^T over all d columns (W2 stored transposed: row f = column f of W2)
        if (R > 0) {
            mma_cols_trans<MT>(w2, R, rpad, d, f0, ub, ypart);
        } else {
            for (int i = tid; i < MT * d; i += NTHREADS) ypart[i] = 0.f;
        }
    } else {
        // u = GELU(LN2(x) W1^T + b1) for this CTA's FFN rows
        if (R > 0) project_rows<WT, MT>(w1, R, d, xr, red, u);
        for (int o = tid; o < R * MT; o += NTHREADS) u[o] = gelu_erf(u[o] + (o < NTHREADS ? b1v[0] : b1v[1]));
        __syncthreads();
        trace_mark(a.trace, 2);  // u done
        // partial u W2^T over all d columns (W2 stored transposed: row f = column f of W2)
        for (int c = tid * 4; c < d; c += NTHREADS * 4) {
            float acc[MT][4];
#pragma unroll
            for (int m = 0; m < MT; ++m)
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[m][i] = 0.f;
            for (int f = 0; f < R; ++f) {
                float w4[4];
                load4(w2 + (size_t)f * d + c, w4);
#pragma unroll
                for (int m = 0; m < MT; ++m) {
                    const float uf = u[f * MT + m];
#pragma unroll
                    for (int i = 0; i < 4; ++i) acc[m][i] = fmaf(uf, w4[i], acc[m][i]);
                }
            }
#pragma unroll
            for (int m = 0; m < MT; ++m)
                *reinterpret_cast<float4*>(ypart + (size_t)m * d + c) =
                    make_float4(acc[m][0], acc[m][1], acc[m][2], acc[m][3]);
        }
    }
    trace_mark(a.trace, 3);  // partial outputs done
    cluster.sync();
    trace_mark(a.trace, 4);
    // this CTA sums columns [rank * cols, +cols) over the cluster and adds them to the output
#pragma unroll
    for (int k = 0; k < RES_PER; ++k) {
        const int i = tid + k * NTHREADS;
        if (i >= MT * cols / 4) continue;
        const int m = i / (cols / 4), c = rank * cols + (i % (cols / 4)) * 4;
        if (!s_act[m]) continue;
        float4 y = resv[k];
#pragma unroll
        for (int r = 0; r < CB; ++r) {
            const float4 p = ld_dsmem4(dsmem_addr(ypart + (size_t)m * d + c, r));
            y.x += p.x;
            y.y += p.y;
            y.z += p.z;
            y.w += p.w;
        }
        atomicAdd(reinterpret_cast<float4*>(a.x_out + (size_t)m * d + c), y);
    }
    trace_mark(a.trace, 5);  // cluster sums added
    cluster_arrive_relaxed();  // done reading the peers' partials
    cluster_wait();            // peers may still read this CTA's shared memory
}

// the whole unified L1 as shared memory, so CTAs of the two block kernels can share an SM
template <typename T>
cudaError_t set_smem(T kern, size_t bytes) {
    return ensure_kernel_smem(reinterpret_cast<const void*>(kern), bytes, true);
}

template <typename WT, int MT>
cudaError_t launch_attn_block_t(const LayerArgs& a, cudaStream_t s, bool pdl) {
    const ALayout L(a.d, sizeof(WT), MT, a.page_size);
    auto kern = attn_block_kernel<WT, MT>;
    cudaError_t e = set_smem(kern, L.total);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(CA, a.n_heads);
    cfg.blockDim = dim3(NTHREADS);
    cfg.dynamicSmemBytes = L.total;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, a);
}

template <typename WT, int MT>
cudaError_t launch_mlp_t(const LayerArgs& a, int grid, cudaStream_t s, bool pdl) {
    const BLayout L(a.d, a.ffn_rows_per_cta, sizeof(WT), MT, MLP_CLUSTER);
    auto kern = mlp_kernel<WT, MT, MLP_CLUSTER>;
    cudaError_t e = set_smem(kern, L.total);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(NTHREADS);
    cfg.dynamicSmemBytes = L.total;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = MLP_CLUSTER;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kern, a);
}

template <int MT>
cudaError_t dispatch_layer(const LayerArgs& a, int which, bool bf, int grid, cudaStream_t s, bool pdl) {
    if (which == 0) return bf ? launch_attn_block_t<__nv_bfloat16, MT>(a, s, pdl) : launch_attn_block_t<float, MT>(a, s, pdl);
    return bf ? launch_mlp_t<__nv_bfloat16, MT>(a, grid, s, pdl) : launch_mlp_t<float, MT>(a, grid, s, pdl);
}

cudaError_t dispatch_rows(const LayerArgs& a, int which, bool bf, int grid, cudaStream_t s, bool pdl) {
    if (a.M < 1 || a.M > MAX_ROWS) return cudaErrorInvalidValue;
    if (a.M <= 1) return dispatch_layer<1>(a, which, bf, grid, s, pdl);
    if (a.M <= 2) return dispatch_layer<2>(a, which, bf, grid, s, pdl);
    if (a.M <= 4) return dispatch_layer<4>(a, which, bf, grid, s, pdl);
    return dispatch_layer<8>(a, which, bf, grid, s, pdl);
}

}  // namespace

size_t attn_block_smem_bytes(int d, int wbytes, int page) { return ALayout(d, wbytes, MAX_ROWS, page).total; }

size_t mlp_smem_bytes(int d, int rows_per_cta, int wbytes) {
    return BLayout(d, rows_per_cta, wbytes, MAX_ROWS, MLP_CLUSTER).total;
}

cudaError_t mlp_max_clusters(int d, int num_sms, int wbytes, int d_ffn, int* clusters) {
    // the most clusters C of MLP_CLUSTER CTAs, each with ceil(d_ffn / (C * MLP_CLUSTER))
    // FFN rows, that the GPU can hold at once
    auto kern = wbytes == 2 ? mlp_kernel<__nv_bfloat16, MAX_ROWS, MLP_CLUSTER> : mlp_kernel<float, MAX_ROWS, MLP_CLUSTER>;
    *clusters = 0;
    for (int C = num_sms / MLP_CLUSTER; C >= 1; --C) {  // one CTA per SM at most
        const int rpc = (d_ffn + C * MLP_CLUSTER - 1) / (C * MLP_CLUSTER);
        const BLayout L(d, rpc, wbytes, MAX_ROWS, MLP_CLUSTER);
        if (L.total > 200 * 1024) break;  // fewer clusters only need more shared memory
        cudaError_t e = set_smem(kern, L.total);
        if (e != cudaSuccess) return e;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(C * MLP_CLUSTER);
        cfg.blockDim = dim3(NTHREADS);
        cfg.dynamicSmemBytes = L.total;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = MLP_CLUSTER;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int fit = 0;
        e = cudaOccupancyMaxActiveClusters(&fit, kern, &cfg);
        if (e != cudaSuccess) return e;
        if (fit >= C) {
            *clusters = C;
            return cudaSuccess;
        }
    }
    return cudaSuccess;
}

cudaError_t launch_attn_block(const LayerArgs& a, bool w_bf16, cudaStream_t s, bool pdl) {
    if (a.d % CA || a.d > 1024 || a.rows_per_group < 1 || a.page_size < 1) return cudaErrorInvalidValue;
    return dispatch_rows(a, 0, w_bf16, 0, s, pdl);
}

cudaError_t launch_mlp(const LayerArgs& a, bool w_bf16, int grid, cudaStream_t s, bool pdl) {
    if (a.d % (4 * MLP_CLUSTER) || a.d > 1024 || grid % MLP_CLUSTER) return cudaErrorInvalidValue;
    return dispatch_rows(a, 1, w_bf16, grid, s, pdl);
}

}  // namespace mtp
