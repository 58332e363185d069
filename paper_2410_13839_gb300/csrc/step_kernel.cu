// step_kernel.cu -- the transformer stack of one decode pass (Sec. III-A:
// embedding of the fed codec tokens, then every pre-LN block) as ONE
// persistent kernel, for bf16 weights and at most 8 fed rows.
//
// Why one kernel: at batch 1 a layer streams 25 MB of weights (3.7 us at the
// HBM peak) but is a chain of dependent phases; launched as two kernels per
// layer the step pays launch gaps and cold instruction caches 24 times.  Here
// every CTA (one per SM, clusters of 4) owns a shared-memory ring of 16 KB
// stages that a producer warp keeps filled with cp.async.bulk copies of the
// CTA's weight slices and cached keys/values in the order the CTA consumes
// them, for the whole pass -- weights never wait for activations, so the next
// phases' bytes stream while the current phase computes and while the grid
// waits at a barrier.
//
// Work of a layer l (x(l): the fed rows' residual stream):
//   phase A, clusters 0..H-1 (cluster h = attention head h, CTA rank r):
//     LN1(x(l)) -> this CTA's 48 of head h's 192 q|k|v rows (mma.sync,
//     bf16 hi + lo activations); keys/values of the fed rows appended to the
//     paged cache; the head's q|k|v rows exchanged in the cluster through
//     distributed shared memory (mbarrier arrive.release.cluster); attention
//     of the fed rows over split r of the cached keys (rank 3 also over the
//     keys fed this step, from the exchanged rows); the 4 splits merged
//     (log-sum-exp) over DSMEM; this CTA's d/4 rows of W_o applied and added
//     into x_mid(l) with float atomics (head 0 adds x(l) + b_o).
//   grid barrier (bounded); phase F, every CTA with FFN units:
//     LN2(x_mid(l)) -> u = GELU(W1 rows + b1) for its FFN rows -> partial
//     u W2^T over all d outputs; the cluster sums its 4 partials over DSMEM
//     and adds them into x(l+1) (cluster 0 adds x_mid(l) + b2).
//   grid barrier (bounded).
// Layer 0's x(0) = E_codec[token] + PE(position) is computed in registers by
// the attention CTAs (no embedding kernel, no barrier).
//
// Residual buffers: T_0 (x_mid(0)) is a dedicated buffer Z that must be zero
// at entry; T_p (p >= 1) rotates over three buffers, T_p = B[(p - 1) % 3].
// Phase p zeroes T_{p+1}, whose old contents were last read in phase p - 1
// (before the barrier that opened phase p); phase 2 re-zeroes Z for the next
// launch.  The pass's final rows are T_{2L-1}.  Grid barriers count arrivals
// in a device word that the last CTA to leave resets.
//
// Every wait is bounded (ring stages, cluster exchanges, grid barriers); on
// time-out the kernel sets the device error word, skips the rest of its work
// and still meets the final cluster barrier, so no CTA leaves while a peer
// may read its shared memory.
#include <math.h>

#include "common.cuh"
#include "frag.cuh"
#include "kernels.cuh"

namespace mtp {
namespace {

using namespace frag;

constexpr int CL = SK_CLUSTER;               // CTAs per cluster = key splits of a head
constexpr int THREADS = NTHREADS + 32;        // 8 consumer warps + 1 producer warp
constexpr int STAGE = SK_STAGE_BYTES;         // bytes per ring stage
constexpr int STAGE_KEYS = 64;                // cached positions per key/value stage (K 8 KB | V 8 KB)
constexpr int KV_CHUNK = 4;                   // key/value stages waited for together
constexpr int QR = 3 * HEAD_DIM / CL;         // q|k|v rows per attention CTA (48)
constexpr int PARTW = 2 + HEAD_DIM;           // (max, sum, out[64])
constexpr uint32_t GRID_MAX_POLLS = 1u << 21;  // grid-barrier polls before giving up (about a second)

__host__ __device__ inline size_t al128(size_t x) { return (x + 127) & ~(size_t)127; }

// Dynamic shared memory (host and device compute the same offsets):
//   ring   stages of weights / cached keys and values
//   x      the fed rows' LayerNorm as bf16 hi | lo; then the K-split partials
//          and the projection result; the warps' softmax states; W_o outputs;
//          the GELU rows as bf16 hi | lo (all local to the CTA)
//   u      phase A: q|k|v rows received from the cluster, the keys/values fed
//          this step, the attention partials sent and received (then the merged
//          head output); phase F: the FFN partial outputs received from the
//          cluster.  Peers write u only after the grid barrier that ends the
//          other phase, so the two uses never overlap in time.
struct SkLayout {
    size_t ring, x, accs, qkvf, newkv, part, parts, yrecv, total;
    __host__ __device__ SkLayout(int d, int mt, int nst) {
        ring = 0;
        x = (size_t)nst * STAGE;
        const size_t xb = (size_t)2 * mt * (d + 8) * 2;                 // LN rows, bf16 hi | lo
        const size_t red = (size_t)NWARPS * 64 * 8 * 4;                 // K-split partials (<= 64 rows)
        const size_t wst = (size_t)NWARPS * mt * PARTW * 4;             // warps' softmax states
        const size_t yt = (size_t)mt * (d / CL) * 4;                    // W_o outputs of this CTA
        size_t xs = xb > red + (size_t)64 * mt * 4 ? xb : red + (size_t)64 * mt * 4;
        xs = xs > wst ? xs : wst;
        xs = xs > yt ? xs : yt;
        accs = x + red;                                                  // [64][MT] after the partials
        const size_t u = al128(x + xs);
        qkvf = u;                                                        // [192][MT] (then the head output)
        newkv = al128(qkvf + (size_t)3 * HEAD_DIM * mt * 4);            // [2][MT + 16][64] bf16 (then W_o's operand)
        part = al128(newkv + (size_t)2 * (mt + 16) * HEAD_DIM * 2);     // [MT][PARTW]
        parts = al128(part + (size_t)mt * PARTW * 4);                   // [CL][MT][PARTW]
        const size_t a_end = al128(parts + (size_t)CL * mt * PARTW * 4);
        yrecv = u;                                                       // [CL][MT][d / CL]
        const size_t f_end = al128(u + (size_t)mt * d * 4);
        total = a_end > f_end ? a_end : f_end;
    }
};

// ---- synchronisation -------------------------------------------------------

__device__ __forceinline__ void consumer_sync() { ConsumerSync()(); }

// AND of v over the 256 consumer threads (named barrier 1; the producer warp takes no part).
__device__ __forceinline__ bool consumer_all(bool v) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.and.pred q, 1, 256, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)v)
        : "memory");
    return r != 0;
}

__device__ __forceinline__ uint32_t ld_acquire_gpu(const unsigned* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Bounded wait on phase `parity` of a local mbarrier with cluster-scope acquire
// (peers' shared-memory writes released by their arrive become visible).
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t* bar, uint32_t parity, int* err) {
    for (uint32_t i = 0; i < MBAR_MAX_POLLS; ++i) {
        uint32_t done;
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(done)
            : "r"(smem_addr(bar)), "r"(parity)
            : "memory");
        if (done) return true;
    }
    atomicOr(err, ERR_WAIT_TIMEOUT);
    return false;
}

// One fp32 into the shared memory of cluster CTA `rank` (addresses mapped with
// dsmem_addr), completing `bytes` 4 of that CTA's transaction barrier: no
// fence, the barrier's phase completes once every expected byte has landed.
__device__ __forceinline__ void push_f32(uint32_t remote, float v, uint32_t remote_bar) {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.f32 [%0], %1, [%2];" ::"r"(remote), "f"(v),
                 "r"(remote_bar)
                 : "memory");
}

// Grid barrier of the 256 consumer threads of every CTA: arrive, then wait
// until `target` arrivals are counted.  Bounded: on time-out sets the error
// word and the abort flag.  Returns false when the CTA must stop.
__device__ __forceinline__ bool grid_sync(unsigned* ctr, unsigned target, int* err, volatile int* s_abort) {
    consumer_sync();
    if (threadIdx.x == 0 && !*s_abort) {
        __threadfence();
        atomicAdd(ctr, 1u);
        uint32_t polls = 0;
        while (ld_acquire_gpu(ctr) < target) {
            if (++polls > GRID_MAX_POLLS) {
                atomicOr(err, ERR_WAIT_TIMEOUT);
                *s_abort = 1;
                break;
            }
        }
        __threadfence();
    }
    consumer_sync();
    return *s_abort == 0;
}

// ---- phase timeline (tracing) ----------------------------------------------
// With tracing on, a.trace is followed by one record per phase (A then F of
// each layer): earliest CTA start of the phase, latest CTA start, latest CTA
// end (arrival at the next barrier) and up to 8 marks (latest CTA past each);
// then, for the middle layer, one record per CTA and phase with the same
// fields for that CTA alone (its index in the second word).
__device__ __forceinline__ unsigned long long* phase_rec(const StepArgs& a, int p) {
    return a.trace ? a.trace + (size_t)TRACE_WORDS * (1 + p) : nullptr;
}
__device__ __forceinline__ unsigned long long* cta_rec(const StepArgs& a, int p) {
    if (!a.trace || p / 2 != a.L / 2) return nullptr;
    return a.trace + (size_t)TRACE_WORDS * (1 + 2 * a.L + 2 * blockIdx.x + (p & 1));
}
__device__ __forceinline__ void phase_start(const StepArgs& a, int p) {
    unsigned long long* r = phase_rec(a, p);
    if (r && threadIdx.x == 0) {
        const unsigned long long t = globaltimer();
        atomicMin(r, t);
        atomicMax(r + 1, t);
        if (unsigned long long* c = cta_rec(a, p)) {
            c[0] = t;
            c[1] = blockIdx.x;
        }
    }
}
__device__ __forceinline__ void phase_mark(const StepArgs& a, int p, int i) {
    unsigned long long* r = phase_rec(a, p);
    if (r && threadIdx.x == 0) {
        const unsigned long long t = globaltimer();
        atomicMax(r + 3 + i, t);
        if (unsigned long long* c = cta_rec(a, p)) c[3 + i] = t;
    }
}
__device__ __forceinline__ void phase_end(const StepArgs& a, int p) {
    unsigned long long* r = phase_rec(a, p);
    if (r && threadIdx.x == 0) {
        const unsigned long long t = globaltimer();
        atomicMax(r + 2, t);
        if (unsigned long long* c = cta_rec(a, p)) c[2] = t;
    }
}

// ---- the stage ring --------------------------------------------------------
// Items (stage fills) are produced and consumed in one fixed order per CTA.
// full[s]: the producer's expect_tx + the copies' bytes; empty[s]: one arrive
// per consumer warp.  Consumers wait for "full" of every item in order before
// releasing it, so no warp can release a use of a slot before its fill.

struct Ring {
    uint64_t* full;
    uint64_t* empty;
    uint32_t base;  // shared address of stage 0
    int nst;
};

__device__ __forceinline__ int ring_slot(int item, int nst) { return item % nst; }
__device__ __forceinline__ uint32_t ring_parity(int item, int nst) { return (uint32_t)(item / nst) & 1u; }

__device__ __forceinline__ bool ring_wait_full(const Ring& R, int item, int* err) {
    return mbar_wait(&R.full[ring_slot(item, R.nst)], ring_parity(item, R.nst), err);
}
// Rows of a weight slice spread over consecutive ring stages, `rps` rows per stage.
struct RingRows {
    uint32_t base;
    int first, nst, rps_shift, row_bytes;
    __device__ __forceinline__ uint32_t row(int r) const {
        int s = first + (r >> rps_shift);
        if (s >= nst) s -= nst;
        return base + (uint32_t)s * STAGE + (uint32_t)(r & ((1 << rps_shift) - 1)) * row_bytes;
    }
};

// ---- row plan --------------------------------------------------------------

struct Plan {
    int seq[MAX_ROWS], pos[MAX_ROWS], tok[MAX_ROWS];
    int gseq[MAX_ROWS], gold[MAX_ROWS], gnew[MAX_ROWS];  // per group: slot, cached length, fed count
};

// Row r of the pass is fed token j = r % rpg of slot seq_base + r / rpg.
__device__ __forceinline__ void plan_rows(const StepArgs& a, int* seq, int* pos, int* tok, int* gseq, int* gold,
                                          int* gnew) {
    const int groups = (a.rows + a.rpg - 1) / a.rpg;
    for (int g = 0; g < MAX_ROWS; ++g) {
        gseq[g] = -1;
        gold[g] = 0;
        gnew[g] = 0;
    }
    for (int r = 0; r < MAX_ROWS; ++r) {
        seq[r] = -1;
        pos[r] = -1;
        tok[r] = 0;
        if (r >= a.rows) continue;
        const int g = r / a.rpg, j = r % a.rpg, b = a.seq_base + g;
        if (b >= a.slots) continue;
        const int act = a.active[b], dn = a.done[b], np = a.n_pending[b], len = a.seq_len[b];
        if (!act || dn || j >= np) continue;
        const int t = a.pending[b * a.n_max + j];
        if (len + j >= a.max_pos || t < 0 || t >= a.codec_vocab) {
            atomicOr(a.err, ERR_BOUNDS);
            continue;
        }
        seq[r] = b;
        pos[r] = len + j;
        tok[r] = t;
        gseq[g] = b;
        gold[g] = len;
        gnew[g] = max(gnew[g], j + 1);
    }
    (void)groups;
}

// Cached-key stages [s0, s1) of split `rank` for a group with `old` cached keys.
__device__ __forceinline__ void split_stages(int old, int rank, int& s0, int& s1) {
    const int ns = (old + STAGE_KEYS - 1) / STAGE_KEYS;
    const int per = (ns + CL - 1) / CL;
    s0 = min(ns, rank * per);
    s1 = min(ns, s0 + per);
}

// ---- producer --------------------------------------------------------------

struct Producer {
    const StepArgs& a;
    const Ring& R;
    int item;
    uint64_t pol;
    bool ok;

    // Wait for the next slot to be free and arm it for `bytes`; returns its shared address.
    __device__ __forceinline__ uint32_t begin(uint32_t bytes, uint64_t** full) {
        const int s = ring_slot(item, R.nst);
        // first use of a slot: parity 1 of a fresh barrier counts as completed
        if (!mbar_wait(&R.empty[s], ring_parity(item, R.nst) ^ 1u, a.err)) {
            ok = false;
            return 0;
        }
        *full = &R.full[s];
        mbar_arrive_expect_tx(*full, bytes);
        return R.base + (uint32_t)s * STAGE;
    }
    __device__ __forceinline__ void copy(uint32_t dst, const void* src, uint32_t bytes, uint64_t* full, bool hint) {
        if (hint)
            asm volatile(
                "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], "
                "%4;" ::"r"(dst),
                "l"(src), "r"(bytes), "r"(smem_addr(full)), "l"(pol)
                : "memory");
        else
            asm volatile(
                "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                "l"(src), "r"(bytes), "r"(smem_addr(full))
                : "memory");
    }
    // `total` contiguous weight bytes from src, in stages of at most STAGE bytes
    __device__ __forceinline__ void weights(const void* src, uint32_t total) {
        const char* p = static_cast<const char*>(src);
        for (uint32_t off = 0; off < total && ok; off += STAGE) {
            const uint32_t n = min((uint32_t)STAGE, total - off);
            uint64_t* full;
            const uint32_t dst = begin(n, &full);
            if (!ok) return;
            copy(dst, p + off, n, full, true);
            ++item;
        }
    }
    // cached keys/values of positions [s * 64, s * 64 + 64) of `seq`, layer l, head h
    __device__ __forceinline__ void kv_stage(int seq, int s, int l, int h) {
        const int P = a.page_size;
        const long long layer_off = (long long)l * 2 * a.H * P * HEAD_DIM;
        const long long head = (long long)h * P * HEAD_DIM, v_off = (long long)a.H * P * HEAD_DIM;
        uint64_t* full;
        const uint32_t dst = begin(STAGE, &full);
        if (!ok) return;
        const int* bt = a.block_table + (size_t)seq * a.bt_stride;
        const int key0 = s * STAGE_KEYS;
        if (P >= STAGE_KEYS) {
            int phys = bt[key0 / P];
            if (phys < 0) {
                atomicOr(a.err, ERR_BOUNDS);
                phys = 0;
            }
            const __nv_bfloat16* k = a.kv_pool + (long long)phys * a.page_elems + layer_off + head +
                                     (long long)(key0 % P) * HEAD_DIM;
            copy(dst, k, STAGE / 2, full, false);
            copy(dst + STAGE / 2, k + v_off, STAGE / 2, full, false);
        } else {
            const int per = STAGE_KEYS / P;  // pages per stage
            int first = bt[key0 / P];
            if (first < 0) {
                atomicOr(a.err, ERR_BOUNDS);
                first = 0;
            }
            for (int q = 0; q < per; ++q) {
                const int idx = key0 / P + q;
                int phys = idx < a.bt_stride ? bt[idx] : -1;
                if (phys < 0) phys = first;  // past the slot's pages: any valid page (those keys are masked)
                const __nv_bfloat16* k = a.kv_pool + (long long)phys * a.page_elems + layer_off + head;
                const uint32_t bytes = (uint32_t)P * HEAD_DIM * 2;
                copy(dst + q * bytes, k, bytes, full, false);
                copy(dst + STAGE / 2 + q * bytes, k + v_off, bytes, full, false);
            }
        }
        ++item;
    }
};

__device__ __noinline__ int run_producer(const StepArgs& a, const Ring& R, bool att, int head, int rank,
                                         int2 ffn) {
    Producer p{a, R, 0, l2_evict_first_policy(), true};
    const int d = a.d;
    const size_t lw = (size_t)a.layer_stride;
    const uint32_t qkv_bytes = (uint32_t)QR * d * 2, wo_bytes = (uint32_t)(d / CL) * HEAD_DIM * 2;
    const uint32_t unit_bytes = (uint32_t)a.ffn_unit_rows * d * 2;
    auto qkv_src = [&](int l) {
        return reinterpret_cast<const char*>(a.wqkv) + l * lw + ((size_t)head * 3 * HEAD_DIM + rank * QR) * d * 2;
    };
    auto ffn_units = [&](int l) {
        const char* w1 = reinterpret_cast<const char*>(a.w1) + l * lw + (size_t)ffn.x * unit_bytes;
        const char* w2 = reinterpret_cast<const char*>(a.w2t) + l * lw + (size_t)ffn.x * unit_bytes;
        p.weights(w1, (uint32_t)ffn.y * unit_bytes);  // one stage per unit
        p.weights(w2, (uint32_t)ffn.y * unit_bytes);
    };
    // before the dependency wait: what needs no state from the previous kernel
    if (att) p.weights(qkv_src(0), qkv_bytes);
    pdl_wait();
    Plan pl;
    plan_rows(a, pl.seq, pl.pos, pl.tok, pl.gseq, pl.gold, pl.gnew);
    const int groups = (a.rows + a.rpg - 1) / a.rpg;
    for (int l = 0; l < a.L && p.ok; ++l) {
        if (att) {
            if (l > 0) p.weights(qkv_src(l), qkv_bytes);
            for (int g = 0; g < groups && p.ok; ++g) {
                if (pl.gseq[g] < 0) continue;
                int s0, s1;
                split_stages(pl.gold[g], rank, s0, s1);
                for (int s = s0; s < s1 && p.ok; ++s) p.kv_stage(pl.gseq[g], s, l, head);
            }
            p.weights(reinterpret_cast<const char*>(a.wo) + l * lw + ((size_t)head * d + rank * (d / CL)) * HEAD_DIM * 2,
                      wo_bytes);
        }
        if (ffn.y > 0) ffn_units(l);
    }
    return p.item;  // items issued
}

// ---- consumer building blocks ---------------------------------------------

// out[row][m] = sum_k W[row][k] x[m][k] for R <= 64 rows spread over ring stages,
// K split across the 8 warps; x as bf16 hi and lo parts [MT][K + 8] each.
// wpart [NWARPS][R][8] may overlap x.
template <int MT>
__device__ __forceinline__ void ring_rows_ksplit(const RingRows& w, int R, int K, const __nv_bfloat16* xb,
                                                 float* wpart, float* out) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int tiles = (R + 15) / 16;
    const int kslice = K / NWARPS;
    const uint32_t xbase = smem_addr(xb);
    const int xstride = (K + 8) * 2;
    const int brow = (lane & 7) < MT ? (lane & 7) : 0;
    const int bhalf = (lane >> 3) & 1;
    const int arow = lane & 15, ahalf = lane >> 4;
    uint32_t ra[4];
    int rk[4];
#pragma unroll
    for (int t = 0; t < 4; ++t) {
        const int row = min(t * 16 + arow, R - 1);
        ra[t] = w.row(row);
        rk[t] = row & 7;
    }
    float acc[4][4], accl[4][4];
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
        const int chunk = (k0 >> 3) + ahalf;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            if (t < tiles) {
                uint32_t af[4];
                ldsm_x4(af, ra[t] + ((uint32_t)(chunk ^ rk[t]) << 4));
                mma_bf16(acc[t], af, bh);
                mma_bf16(accl[t], af, bl);
            }
        }
    }
#pragma unroll
    for (int t = 0; t < 4; ++t)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[t][i] += accl[t][i];
    consumer_sync();  // every warp is done with x
    const int g = lane >> 2, c2 = (lane & 3) * 2;
    float* mine = wpart + (size_t)warp * R * 8;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
        if (t >= tiles) continue;
        const int r0 = t * 16 + g, r1 = r0 + 8;
        if (r0 < R) *reinterpret_cast<float2*>(mine + r0 * 8 + c2) = make_float2(acc[t][0], acc[t][1]);
        if (r1 < R) *reinterpret_cast<float2*>(mine + r1 * 8 + c2) = make_float2(acc[t][2], acc[t][3]);
    }
    consumer_sync();
    for (int i = threadIdx.x; i < R * MT; i += NTHREADS) {
        const int j = (i / MT) * 8 + i % MT;
        float y = 0.f;
#pragma unroll
        for (int w2 = 0; w2 < NWARPS; ++w2) y += wpart[(size_t)w2 * R * 8 + j];
        out[i] = y;
    }
    consumer_sync();
}

// out[m * R + row] = sum_k W[row][k] x[m][k] for R rows over ring stages with
// short K (one warp per 16-row tile, whole K); x: bf16 hi | lo [MT][K + 8].
template <int MT>
__device__ __forceinline__ void ring_rows_tiles(const RingRows& w, int R, int K, const __nv_bfloat16* xb,
                                                float* out) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t xbase = smem_addr(xb);
    const int xstride = (K + 8) * 2;
    const int brow = (lane & 7) < MT ? (lane & 7) : 0;
    const int bhalf = (lane >> 3) & 1;
    const int arow = lane & 15, ahalf = lane >> 4;
    const int g = lane >> 2, c2 = (lane & 3) * 2;
    for (int t = warp; t * 16 < R; t += NWARPS) {
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
        const int row = min(t * 16 + arow, R - 1);
        const uint32_t ra = w.row(row);
        const int rk = row & 7;
        for (int k0 = 0; k0 < K; k0 += 16) {
            uint32_t af[4], bh[2], bl[2];
            ldsm_x2(bh, xbase + brow * xstride + (k0 + bhalf * 8) * 2);
            ldsm_x2(bl, xbase + MT * xstride + brow * xstride + (k0 + bhalf * 8) * 2);
            ldsm_x4(af, ra + ((uint32_t)(((k0 >> 3) + ahalf) ^ rk) << 4));
            mma_bf16(acc, af, bh);
            mma_bf16(acc, af, bl);
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

// y[m * C + col] = sum_f W2[col][f] u[m][f] over the R <= 64 FFN rows f whose
// W2^T rows (C columns each) are spread over ring stages; the MMA's A operand
// is W2 read with ldmatrix.trans.  u: bf16 hi | lo [MT][rpad + 8], zero for f >= R.
template <int MT>
__device__ __forceinline__ void ring_cols_trans(const RingRows& w, int R, int rpad, int C, const __nv_bfloat16* ub,
                                                float* y) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t ubase = smem_addr(ub);
    const int ustride = (rpad + 8) * 2;
    const int brow = (lane & 7) < MT ? (lane & 7) : 0;
    const int bhalf = (lane >> 3) & 1;
    const int g = lane >> 2, c2 = (lane & 3) * 2;
    const int ksteps = rpad / 16;  // <= 4
    uint32_t bh[4][2], bl[4][2], fa[4];
    int fk[4];
    const int fl = (lane & 7) + ((lane >> 4) << 3), chalf = (lane >> 3) & 1;
#pragma unroll
    for (int ks = 0; ks < 4; ++ks)
        if (ks < ksteps) {
            ldsm_x2(bh[ks], ubase + brow * ustride + (ks * 16 + bhalf * 8) * 2);
            ldsm_x2(bl[ks], ubase + MT * ustride + brow * ustride + (ks * 16 + bhalf * 8) * 2);
            const int f = min(ks * 16 + fl, R - 1);
            fa[ks] = w.row(f);
            fk[ks] = f & 7;
        }
    for (int t = warp; t * 16 < C; t += NWARPS) {
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
            if (ks >= ksteps) continue;
            uint32_t af[4];
            ldsm_x4_t(af, fa[ks] + ((uint32_t)((t * 2 + chalf) ^ fk[ks]) << 4));
            mma_bf16(acc, af, bh[ks]);
            mma_bf16(acc, af, bl[ks]);
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

// ring_cols_trans, with each output y[m][col] sent to the cluster CTA that
// reduces column col (dest = col / (C / CL)) at yrecv[rank][m][col % (C / CL)]
// of that CTA (st.async on its barrier xf) instead of being stored locally.
template <int MT>
__device__ __forceinline__ void ring_cols_trans_push(const RingRows& w, int R, int rpad, int C, const __nv_bfloat16* ub,
                                                     const float* yrecv, uint64_t* xf, int rank) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t ubase = smem_addr(ub);
    const int ustride = (rpad + 8) * 2;
    const int brow = (lane & 7) < MT ? (lane & 7) : 0;
    const int bhalf = (lane >> 3) & 1;
    const int g = lane >> 2, c2 = (lane & 3) * 2;
    const int ksteps = rpad / 16;  // <= 4
    const int cols = C / CL;
    uint32_t bh[4][2], bl[4][2], fa[4];
    int fk[4];
    const int fl = (lane & 7) + ((lane >> 4) << 3), chalf = (lane >> 3) & 1;
#pragma unroll
    for (int ks = 0; ks < 4; ++ks)
        if (ks < ksteps) {
            ldsm_x2(bh[ks], ubase + brow * ustride + (ks * 16 + bhalf * 8) * 2);
            ldsm_x2(bl[ks], ubase + MT * ustride + brow * ustride + (ks * 16 + bhalf * 8) * 2);
            const int f = min(ks * 16 + fl, R - 1);
            fa[ks] = w.row(f);
            fk[ks] = f & 7;
        }
    // two 16-column tiles per warp at a time (independent accumulator chains)
    const int ntiles = C / 16;
    for (int t0 = warp; t0 < ntiles; t0 += 2 * NWARPS) {
        float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
            if (ks >= ksteps) continue;
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int t = min(t0 + u * NWARPS, ntiles - 1);
                uint32_t af[4];
                ldsm_x4_t(af, fa[ks] + ((uint32_t)((t * 2 + chalf) ^ fk[ks]) << 4));
                mma_bf16(acc[u], af, bh[ks]);
                mma_bf16(acc[u], af, bl[ks]);
            }
        }
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int t = t0 + u * NWARPS;
            if (t >= ntiles) continue;
            const int col0 = t * 16 + g;
            const int dest = col0 / cols, lc = col0 % cols;  // a 16-column tile never straddles two CTAs' columns
            const uint32_t ybase = dsmem_addr(yrecv, dest), bar = dsmem_addr(xf, dest);
            if (c2 < MT) {
                push_f32(ybase + (uint32_t)(((rank * MT + c2) * cols + lc) * 4), acc[u][0], bar);
                push_f32(ybase + (uint32_t)(((rank * MT + c2) * cols + lc + 8) * 4), acc[u][2], bar);
            }
            if (c2 + 1 < MT) {
                push_f32(ybase + (uint32_t)(((rank * MT + c2 + 1) * cols + lc) * 4), acc[u][1], bar);
                push_f32(ybase + (uint32_t)(((rank * MT + c2 + 1) * cols + lc + 8) * 4), acc[u][3], bar);
            }
        }
    }
}

// Attention state of one warp: rows qrow = lane / 4 (< MT), online softmax.
struct AttnState {
    float m_run, l_run;
    float o[8][4];
};

// One 16-key tile: keys at shared address kb (rows key*128, 16-byte chunks
// swizzled by key & 7 when swz), values at vb likewise; key position of row i
// is kp0 + i, visible to the lane's query row when vis(i).
template <class Vis>
__device__ __forceinline__ void attn_tile(AttnState& st, const uint32_t (&qhi)[4][2], const uint32_t (&qlo)[4][2],
                                          uint32_t kb, uint32_t vb, int r0, bool swz, Vis vis) {
    const int lane = threadIdx.x & 31;
    const int c2 = (lane & 3) * 2;
    float sfr[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
    float sfl[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
    {
        const int key = r0 + (lane & 7) + ((lane >> 4) << 3), chalf = (lane >> 3) & 1;
        const int kx = swz ? (key & 7) : 0;
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
            uint32_t b[4];
            ldsm_x4(b, kb + key * 128 + ((uint32_t)((2 * ks + chalf) ^ kx) << 4));
            const uint32_t ah[4] = {qhi[ks][0], 0u, qhi[ks][1], 0u};
            const uint32_t al[4] = {qlo[ks][0], 0u, qlo[ks][1], 0u};
            const uint32_t b0[2] = {b[0], b[1]}, b1[2] = {b[2], b[3]};
            mma_bf16(sfr[0], ah, b0);
            mma_bf16(sfl[0], al, b0);
            mma_bf16(sfr[1], ah, b1);
            mma_bf16(sfl[1], al, b1);
        }
    }
    float sv[4] = {sfr[0][0] + sfl[0][0], sfr[0][1] + sfl[0][1], sfr[1][0] + sfl[1][0], sfr[1][1] + sfl[1][1]};
    float tmax = -INFINITY;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int kr = (i >> 1) * 8 + c2 + (i & 1);  // key row within the tile
        sv[i] = vis(kr) ? sv[i] : -INFINITY;
        tmax = fmaxf(tmax, sv[i]);
    }
    tmax = fmaxf(tmax, __shfl_xor_sync(FULL_MASK, tmax, 1));
    tmax = fmaxf(tmax, __shfl_xor_sync(FULL_MASK, tmax, 2));
    const float m_new = fmaxf(st.m_run, tmax);
    const float corr = m_new == -INFINITY ? 1.f : (st.m_run == -INFINITY ? 0.f : expf(st.m_run - m_new));
    float pv[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) pv[i] = sv[i] == -INFINITY ? 0.f : expf(sv[i] - m_new);
    st.l_run = st.l_run * corr + ((pv[0] + pv[1]) + (pv[2] + pv[3]));
    st.m_run = m_new;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        st.o[j][0] *= corr;
        st.o[j][1] *= corr;
    }
    uint32_t ph[4] = {0u, 0u, 0u, 0u}, pl[4] = {0u, 0u, 0u, 0u};
    split_bf16x2(pv[0], pv[1], ph[0], pl[0]);
    split_bf16x2(pv[2], pv[3], ph[2], pl[2]);
    const int vkey = r0 + (lane & 7) + (((lane >> 3) & 1) << 3), vhalf = lane >> 4;
    const int vx = swz ? (vkey & 7) : 0;
#pragma unroll
    for (int dp = 0; dp < 4; ++dp) {
        uint32_t v[4];
        ldsm_x4_t(v, vb + vkey * 128 + ((uint32_t)((2 * dp + vhalf) ^ vx) << 4));
        const uint32_t v0[2] = {v[0], v[1]}, v1[2] = {v[2], v[3]};
        mma_bf16(st.o[2 * dp], ph, v0);
        mma_bf16(st.o[2 * dp], pl, v0);
        mma_bf16(st.o[2 * dp + 1], ph, v1);
        mma_bf16(st.o[2 * dp + 1], pl, v1);
    }
}

// ---- the kernel ------------------------------------------------------------

template <int MT>
__global__ void __cluster_dims__(CL, 1, 1) __launch_bounds__(THREADS, 1) step_kernel(const StepArgs a) {
    extern __shared__ __align__(1024) unsigned char smem[];
    __shared__ uint64_t full_bar[SK_MAX_STAGES], empty_bar[SK_MAX_STAGES];
    // cluster exchanges (transaction barriers: one local arrival + the bytes the peers push):
    // q|k|v rows, attention partials, FFN partial outputs
    __shared__ uint64_t xq_bar, xa_bar, xf_bar;
    __shared__ uint64_t xr_bar;  // the phase's input rows, multicast into every CTA of the cluster
    __shared__ int s_seq[MAX_ROWS], s_pos[MAX_ROWS], s_tok[MAX_ROWS];
    __shared__ int s_gseq[MAX_ROWS], s_gold[MAX_ROWS], s_gnew[MAX_ROWS];
    __shared__ float ln_part[2 * NWARPS][MT];
    __shared__ float ln_stat[2][MT];
    __shared__ float s_scale[NWARPS][MT];
    __shared__ volatile int s_abort;
    __shared__ int s_issued, s_consumed;
    TraceEnd trace_guard(a.trace);

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int G = gridDim.x;
    uint32_t rank_u;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(rank_u));
    const int rank = (int)rank_u, cl = blockIdx.x / CL;
    const int d = a.d, H = a.H;
    const bool att = cl < H;                      // attention cluster of head cl
    const int head = att ? cl : 0;
    const int2 ffn = a.ffn_range[blockIdx.x];
    int f_senders = 0;                            // CTAs of this cluster with FFN rows
    for (int r = 0; r < CL; ++r) f_senders += a.ffn_range[cl * CL + r].y > 0;
    const bool fcl = f_senders > 0;               // the cluster reduces FFN outputs
    const bool res_cl = cl == a.res_cluster;      // ... and adds x_mid + b2
    const SkLayout Lo(d, MT, a.ring_stages);
    const Ring R{full_bar, empty_bar, smem_addr(smem + Lo.ring), a.ring_stages};
    const int rps_shift = 31 - __clz(a.ffn_unit_rows);  // weight rows per stage (power of two)
    const int orows = d / CL;                      // W_o rows and reduced FFN columns of this CTA
    const uint32_t xq_bytes = (uint32_t)3 * HEAD_DIM * MT * 4;
    const uint32_t xa_bytes = (uint32_t)CL * MT * PARTW * 4;
    const uint32_t xf_bytes = (uint32_t)f_senders * MT * orows * 4;
    const uint32_t xr_bytes = (uint32_t)MT * d * 4;
    const int xr_total = (att ? a.L - 1 : 0) + (fcl ? a.L : 0);  // multicast row copies this CTA receives

    if (tid == 0) {
        for (int s = 0; s < a.ring_stages; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], NWARPS);
        }
        mbar_init(&xq_bar, 1);
        mbar_init(&xa_bar, 1);
        mbar_init(&xf_bar, 1);
        mbar_init(&xr_bar, 1);
        fence_barrier_init();
        if (xr_total > 0) mbar_arrive_expect_tx(&xr_bar, xr_bytes);
        // armed for layer 0's exchanges before any peer can push
        if (att) {
            mbar_arrive_expect_tx(&xq_bar, xq_bytes);
            mbar_arrive_expect_tx(&xa_bar, xa_bytes);
        }
        if (fcl) mbar_arrive_expect_tx(&xf_bar, xf_bytes);
        s_abort = 0;
    }
    // every CTA's barriers are initialised and armed before any peer pushes to them
    cluster_arrive_release();
    cluster_wait();

    if (warp == NWARPS) {  // producer warp
        if (lane == 0) s_issued = run_producer(a, R, att, head, rank, ffn);
        __syncwarp();
        pdl_launch_dependents();
    } else {
        // ---------------------------------------------------------- consumers
        const int Kw = d / NWARPS;
        float* xs = reinterpret_cast<float*>(smem + Lo.x);
        __nv_bfloat16* xb = reinterpret_cast<__nv_bfloat16*>(smem + Lo.x);   // LN rows hi | lo
        __nv_bfloat16* ub = xb;                                               // GELU rows hi | lo [MT][rpad + 8]
        float* accs = reinterpret_cast<float*>(smem + Lo.accs);              // [64][MT] (q|k|v: [QR][MT])
        float* qkvf = reinterpret_cast<float*>(smem + Lo.qkvf);              // [192][MT]
        float* attn = qkvf;                                                   // [MT][64], after the attention
        __nv_bfloat16* newk = reinterpret_cast<__nv_bfloat16*>(smem + Lo.newkv);  // [MT + 16][64]
        __nv_bfloat16* newv = newk + (MT + 16) * HEAD_DIM;
        __nv_bfloat16* attnb = newk;                                          // hi | lo [MT][72], after
        float* part = reinterpret_cast<float*>(smem + Lo.part);              // [MT][PARTW]
        float* parts = reinterpret_cast<float*>(smem + Lo.parts);            // [CL][MT][PARTW]
        float* yrecv = reinterpret_cast<float*>(smem + Lo.yrecv);            // [CL][MT][orows]
        const int groups = (a.rows + a.rpg - 1) / a.rpg;
        const int rps = a.ffn_unit_rows;
        const int n_qkv_st = (QR + rps - 1) / rps;
        const int n_wo_st = (orows * HEAD_DIM * 2 + STAGE - 1) / STAGE;
        const int fr = ffn.y * rps;                                 // FFN rows of this CTA
        const int rpad = (fr + 15) / 16 * 16;
        int item = 0;                                               // next ring item
        unsigned target = 0;                                        // grid-barrier arrivals awaited
        bool ok = true;
        const size_t lw = (size_t)a.layer_stride;
        auto lp = [&](const float* p, int l) {
            return reinterpret_cast<const float*>(reinterpret_cast<const char*>(p) + l * lw);
        };

        // ---- per-phase parameters, loaded into registers before the phase's barrier
        constexpr int QITEMS = (QR * MT + NTHREADS - 1) / NTHREADS;       // (q|k|v row, fed row) per thread
        constexpr int RES_N = (MT * (1024 / CL) + NTHREADS - 1) / NTHREADS;  // W_o outputs per thread
        constexpr int RES_PER = 2;                                         // FFN output float4s per thread
        float g1[4], be1[4], bq[QITEMS], bo[RES_N];                        // phase A
        float g2[4], be2[4], b1v[2];                                       // phase F
        float4 b2v[RES_PER];
        auto load_a_params = [&](int l) {
            if (!att) return;
            if (lane * 4 < Kw) {
                load4(lp(a.ln1_g, l) + warp * Kw + lane * 4, g1);
                load4(lp(a.ln1_b, l) + warp * Kw + lane * 4, be1);
            }
#pragma unroll
            for (int k = 0; k < QITEMS; ++k) {
                const int i = tid + k * NTHREADS;
                bq[k] = i < QR * MT ? lp(a.bqkv, l)[head * 3 * HEAD_DIM + rank * QR + i / MT] : 0.f;
            }
#pragma unroll
            for (int k = 0; k < RES_N; ++k) {
                const int o = tid + k * NTHREADS;
                bo[k] = head == 0 && o < orows * MT ? lp(a.bo, l)[rank * orows + o % orows] : 0.f;
            }
        };
        auto load_f_params = [&](int l) {
            if (!fcl) return;
            if (fr > 0 && lane * 4 < Kw) {
                load4(lp(a.ln2_g, l) + warp * Kw + lane * 4, g2);
                load4(lp(a.ln2_b, l) + warp * Kw + lane * 4, be2);
            }
            for (int k = 0; k < 2; ++k) {
                const int o = tid + k * NTHREADS, f = o % max(rpad, 1);
                b1v[k] = fr > 0 && o < MT * rpad && f < fr ? lp(a.b1, l)[ffn.x * rps + f] : 0.f;
            }
#pragma unroll
            for (int k = 0; k < RES_PER; ++k) {
                const int i = tid + k * NTHREADS;
                b2v[k] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (res_cl && i < MT * orows / 4)
                    b2v[k] = *reinterpret_cast<const float4*>(lp(a.b2, l) + rank * orows + (i % (orows / 4)) * 4);
            }
        };
#pragma unroll
        for (int i = 0; i < 4; ++i) g1[i] = be1[i] = g2[i] = be2[i] = 0.f;
        load_a_params(0);

        pdl_wait();
        trace_wait(a.trace);
        if (tid == 0) {
            int seq[MAX_ROWS], pos[MAX_ROWS], tok[MAX_ROWS], gs[MAX_ROWS], go[MAX_ROWS], gn[MAX_ROWS];
            plan_rows(a, seq, pos, tok, gs, go, gn);
            for (int r = 0; r < MAX_ROWS; ++r) {
                s_seq[r] = seq[r];
                s_pos[r] = pos[r];
                s_tok[r] = tok[r];
                s_gseq[r] = gs[r];
                s_gold[r] = go[r];
                s_gnew[r] = gn[r];
            }
            if (blockIdx.x == 0)
                for (int r = 0; r < MAX_ROWS; ++r) {  // a slot's last fed row: the next row is another slot's or idle
                    const bool next_same = r + 1 < a.rows && (r + 1) % a.rpg != 0 && seq[r + 1] >= 0;
                    a.row_seq[r] = seq[r];
                    a.row_pos[r] = pos[r];
                    a.row_last[r] = seq[r] >= 0 && !next_same;
                }
        }
        consumer_sync();
        trace_mark(a.trace, 0);

        // The rows a phase starts from ([MT][d] fp32) come from global memory once per cluster:
        // rank 0 copies them with one multicast bulk copy into the x area of all four CTAs (a
        // quarter of the L2 requests of every CTA loading them), each waiting on its xr_bar.
        int xr_left = xr_total;
        auto issue_rows = [&](const float* src) {
            if (rank == 0 && tid == 0) {
                // the rows were written by other CTAs (generic proxy) and are read by the copy engine
                asm volatile("fence.proxy.async.global;" ::: "memory");
                asm volatile(
                    "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.multicast::cluster "
                    "[%0], [%1], %2, [%3], %4;" ::"r"(smem_addr(xs)),
                    "l"(src), "r"(xr_bytes), "r"(smem_addr(&xr_bar)), "h"((uint16_t)((1u << CL) - 1))
                    : "memory");
            }
        };
        auto wait_rows = [&]() -> bool {
            const bool r = mbar_wait(&xr_bar, (uint32_t)(xr_total - xr_left) & 1u, a.err);
            --xr_left;
            if (tid == 0 && xr_left > 0) mbar_arrive_expect_tx(&xr_bar, xr_bytes);  // the next copy
            return r;
        };
        auto tbuf = [&](int p) -> float* {  // residual buffer T_p
            return p == 0 ? a.xbuf + (size_t)3 * MAX_ROWS * d : a.xbuf + (size_t)((p - 1) % 3) * MAX_ROWS * d;
        };
        auto zero_part = [&](float* buf) {  // this CTA's share of a [MAX_ROWS][d] buffer
            const size_t n4 = (size_t)MAX_ROWS * d / 4, per = (n4 + G - 1) / G;
            const size_t b = (size_t)blockIdx.x * per, e = min(n4, b + per);
            for (size_t i = b + tid; i < e; i += NTHREADS) reinterpret_cast<float4*>(buf)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
        };
        // Ring waits and releases are issued in parallel, thread i (lane i) for item first + i: an
        // mbarrier wait or arrive takes a few hundred ns even when the phase is complete.  A
        // wait's result reaches the other threads through the consumer_all that follows it.
        auto wait_items = [&](int first, int count) -> bool {
            return tid >= count || ring_wait_full(R, first + tid, a.err);
        };
        auto release_items = [&](int first, int count) {
            __syncwarp();
            if (lane < count) {
                uint64_t* b = &R.empty[ring_slot(first + lane, R.nst)];
                asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(b)) : "memory");
            }
        };
        // register rows -> LN -> bf16 hi | lo in xb
        auto ln_rows = [&](RowRegs<MT>& xr, const float (&g)[4], const float (&b)[4]) {
            layer_norm_rows<MT, ConsumerSync>(xr, d, g, b, a.ln_eps, ln_part, ln_stat);
            store_rows_split<MT>(xr, d, xb);
            consumer_sync();
        };
        // rows [MT][d] fp32 in shared memory (the cluster's multicast copy) -> registers
        auto load_resid = [&](RowRegs<MT>& xr, const float* x) {
#pragma unroll
            for (int m = 0; m < MT; ++m) {
                if (lane * 4 < Kw) {
                    const float4 v = *reinterpret_cast<const float4*>(x + (size_t)m * d + warp * Kw + lane * 4);
                    xr.v[m][0] = v.x; xr.v[m][1] = v.y; xr.v[m][2] = v.z; xr.v[m][3] = v.w;
                } else {
#pragma unroll
                    for (int i = 0; i < 4; ++i) xr.v[m][i] = 0.f;
                }
            }
        };
        // x(0) = E_codec[token] + PE(position) for active rows, 0 otherwise
        auto embed_val = [&](int m, int c) -> float {
            if (s_seq[m] < 0) return 0.f;
            const uint16_t bits = reinterpret_cast<const uint16_t*>(a.tok_codec)[(size_t)s_tok[m] * d + c];
            return __uint_as_float((uint32_t)bits << 16) + a.pe[(size_t)s_pos[m] * d + c];
        };

        for (int l = 0; l < a.L && ok; ++l) {
            float* x_in = l == 0 ? nullptr : tbuf(2 * l - 1);
            float* x_mid = tbuf(2 * l);
            float* x_out = tbuf(2 * l + 1);
            const uint32_t par = (uint32_t)l & 1u;
            // ======================================================= phase A
            phase_start(a, 2 * l);
            if (att && l > 0) issue_rows(x_in);
            zero_part(tbuf(2 * l + 1));
            if (l == 1) zero_part(tbuf(0));
            if (att) {
                RowRegs<MT> xr;
                float resr[RES_N];  // head 0: x(l) + b_o of this CTA's W_o outputs
                if (l == 0) {
#pragma unroll
                    for (int m = 0; m < MT; ++m)
#pragma unroll
                        for (int i = 0; i < 4; ++i)
                            xr.v[m][i] = lane * 4 < Kw ? embed_val(m, warp * Kw + lane * 4 + i) : 0.f;
                } else {
                    ok = consumer_all(wait_rows());
                    if (!ok) break;
                    load_resid(xr, xs);  // x(l), multicast into this CTA's x area
                }
#pragma unroll
                for (int k = 0; k < RES_N; ++k) {
                    const int o = tid + k * NTHREADS, m = o / orows, f = rank * orows + o % orows;
                    float v = 0.f;
                    if (head == 0 && o < orows * MT && s_seq[m] >= 0)
                        v = (l == 0 ? embed_val(m, f) : xs[(size_t)m * d + f]) + bo[k];
                    resr[k] = v;
                }
                consumer_sync();  // every thread holds its rows before LN overwrites the x area
                ln_rows(xr, g1, be1);
                phase_mark(a, 2 * l, 0);
                // ---- this CTA's q|k|v rows, pushed to every CTA of the cluster
                ok = consumer_all(wait_items(item, n_qkv_st));
                phase_mark(a, 2 * l, 1);
                if (ok) {
                    const RingRows w{R.base, ring_slot(item, R.nst), R.nst, rps_shift, d * 2};
                    ring_rows_ksplit<MT>(w, QR, d, xb, xs, accs);
                }
                release_items(item, n_qkv_st);
                item += n_qkv_st;
                if (!ok) break;
                phase_mark(a, 2 * l, 2);
                float yq[QITEMS];
#pragma unroll
                for (int k = 0; k < QITEMS; ++k) {
                    const int i = tid + k * NTHREADS;
                    yq[k] = 0.f;
                    if (i >= QR * MT) continue;
                    const int row = rank * QR + i / MT;  // within the head's q | k | v
                    const float y = accs[i] + bq[k];
                    yq[k] = y;
                    const float sent = row >= HEAD_DIM ? __bfloat162float(__float2bfloat16_rn(y)) : y;  // k, v as cached
                    const uint32_t off = (uint32_t)(row * MT + i % MT) * 4;
#pragma unroll
                    for (int r = 0; r < CL; ++r) push_f32(dsmem_addr(qkvf, r) + off, sent, dsmem_addr(&xq_bar, r));
                }
                // keys and values of the fed rows into the cache (read by later steps only)
#pragma unroll
                for (int k = 0; k < QITEMS; ++k) {
                    const int i = tid + k * NTHREADS;
                    if (i >= QR * MT) continue;
                    const int row = rank * QR + i / MT, m = i % MT;
                    if (row < HEAD_DIM || s_seq[m] < 0) continue;
                    const int P = a.page_size, sec = row / HEAD_DIM, dd = row % HEAD_DIM;
                    const int page = a.block_table[(size_t)s_seq[m] * a.bt_stride + s_pos[m] / P];
                    if (page < 0) {
                        atomicOr(a.err, ERR_BOUNDS);
                        continue;
                    }
                    const int t = s_pos[m] % P;
                    const long long idx = (long long)page * a.page_elems + (long long)l * 2 * H * P * HEAD_DIM +
                                          (long long)(sec - 1) * H * P * HEAD_DIM + (long long)head * P * HEAD_DIM +
                                          (long long)t * HEAD_DIM + kv_col(t, dd);
                    reinterpret_cast<uint16_t*>(a.kv_pool)[idx] = f32_to_bf16_bits(yq[k]);
                }
                ok = consumer_all(mbar_wait_cluster(&xq_bar, par, a.err));
                if (!ok) break;
                if (tid == 0) mbar_arrive_expect_tx(&xq_bar, xq_bytes);  // armed for the next layer
                // keys/values fed this step as bf16 rows [MT + 16][64] (zero past the fed rows)
                for (int i = tid; i < (MT + 16) * HEAD_DIM; i += NTHREADS) {
                    const int r = i / HEAD_DIM, dd = i % HEAD_DIM;
                    const bool on = r < MT && s_seq[r] >= 0;
                    newk[i] = __float2bfloat16_rn(on ? qkvf[(HEAD_DIM + dd) * MT + r] : 0.f);
                    newv[i] = __float2bfloat16_rn(on ? qkvf[(2 * HEAD_DIM + dd) * MT + r] : 0.f);
                }
                const int qrow = lane >> 2, c2 = (lane & 3) * 2;
                const bool qon = qrow < MT && s_seq[min(qrow, MT - 1)] >= 0;
                const int qpos = qon ? s_pos[qrow] : -1;
                const int qgrp = qrow / a.rpg;
                uint32_t qhi[4][2], qlo[4][2];
#pragma unroll
                for (int ks = 0; ks < 4; ++ks)
#pragma unroll
                    for (int hh = 0; hh < 2; ++hh) {
                        const int k = ks * 16 + hh * 8 + c2;
                        const float q0 = qon ? qkvf[k * MT + qrow] * 0.125f : 0.f;  // 1/sqrt(64), exact
                        const float q1 = qon ? qkvf[(k + 1) * MT + qrow] * 0.125f : 0.f;
                        split_bf16x2(q0, q1, qhi[ks][hh], qlo[ks][hh]);
                    }
                consumer_sync();
                phase_mark(a, 2 * l, 3);
                // ---- attention of the fed rows over split `rank` of each group's keys
                AttnState st;
                st.m_run = -INFINITY;
                st.l_run = 0.f;
#pragma unroll
                for (int j = 0; j < 8; ++j)
#pragma unroll
                    for (int i = 0; i < 4; ++i) st.o[j][i] = 0.f;
                int tc = 0;  // tile counter: warp w takes tiles tc = w mod 8
                for (int g = 0; g < groups && ok; ++g) {
                    if (s_gseq[g] < 0) continue;
                    const int old = s_gold[g];
                    int s0, s1;
                    split_stages(old, rank, s0, s1);
                    for (int c0 = s0; c0 < s1 && ok; c0 += KV_CHUNK) {  // stages waited for and released a chunk at a time
                        const int cn = min(KV_CHUNK, s1 - c0);
                        ok = consumer_all(wait_items(item, cn));
                        if (ok) {
                            for (int j = 0; j < cn; ++j) {
                                const uint32_t kb = R.base + (uint32_t)ring_slot(item + j, R.nst) * STAGE;
                                for (int i = 0; i < 4; ++i, ++tc) {
                                    if ((tc & (NWARPS - 1)) != warp) continue;
                                    const int kp0 = (c0 + j) * STAGE_KEYS + i * 16;
                                    if (kp0 >= old) continue;  // no cached key in this tile
                                    attn_tile(st, qhi, qlo, kb, kb + STAGE / 2, i * 16, true,
                                              [&](int kr) { return qon && qgrp == g && kp0 + kr < old; });
                                }
                            }
                        }
                        release_items(item, cn);
                        item += cn;
                    }
                    if (rank == CL - 1) {  // the keys fed this step
                        const int nn = s_gnew[g];
                        if ((tc & (NWARPS - 1)) == warp) {
                            const uint32_t kb = smem_addr(newk + (size_t)g * a.rpg * HEAD_DIM);
                            const uint32_t vb = smem_addr(newv + (size_t)g * a.rpg * HEAD_DIM);
                            attn_tile(st, qhi, qlo, kb, vb, 0, false,
                                      [&](int kr) { return qon && qgrp == g && kr < nn && old + kr <= qpos; });
                        }
                        ++tc;
                    }
                }
                ok = consumer_all(ok);
                if (!ok) break;
                // merge the warps' states: [NWARPS][MT][PARTW] in the x area
                st.l_run += __shfl_xor_sync(FULL_MASK, st.l_run, 1);
                st.l_run += __shfl_xor_sync(FULL_MASK, st.l_run, 2);
                float* wst = xs;
                if (qrow < MT) {
                    float* ws = wst + ((size_t)warp * MT + qrow) * PARTW;
                    if (c2 == 0) {
                        ws[0] = st.m_run;
                        ws[1] = st.l_run;
                    }
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        *reinterpret_cast<float2*>(ws + 2 + j * 8 + c2) = make_float2(st.o[j][0], st.o[j][1]);
                }
                consumer_sync();
                if (tid < NWARPS * MT) {
                    const int w = tid / MT, m = tid % MT;
                    float Mx = -INFINITY;
#pragma unroll
                    for (int v = 0; v < NWARPS; ++v) Mx = fmaxf(Mx, wst[((size_t)v * MT + m) * PARTW]);
                    const float mw = wst[((size_t)w * MT + m) * PARTW];
                    s_scale[w][m] = mw == -INFINITY ? 0.f : expf(mw - Mx);
                    if (w == 0) part[m * PARTW] = Mx;
                }
                consumer_sync();
                for (int i = tid; i < MT * (1 + HEAD_DIM); i += NTHREADS) {
                    const int m = i / (1 + HEAD_DIM), c = 1 + i % (1 + HEAD_DIM);
                    float y = 0.f;
#pragma unroll
                    for (int w = 0; w < NWARPS; ++w) y = fmaf(s_scale[w][m], wst[((size_t)w * MT + m) * PARTW + c], y);
                    part[m * PARTW + c] = y;
                }
                consumer_sync();
                // this CTA's (max, sum, out) per fed row to every CTA of the cluster: parts[rank]
                for (int i = tid; i < MT * PARTW; i += NTHREADS) {
                    const float v = part[i];
                    const uint32_t off = (uint32_t)(rank * MT * PARTW + i) * 4;
#pragma unroll
                    for (int r = 0; r < CL; ++r) push_f32(dsmem_addr(parts, r) + off, v, dsmem_addr(&xa_bar, r));
                }
                phase_mark(a, 2 * l, 4);
                ok = consumer_all(mbar_wait_cluster(&xa_bar, par, a.err));
                if (!ok) break;
                if (tid == 0) mbar_arrive_expect_tx(&xa_bar, xa_bytes);  // armed for the next layer
                {  // merge the cluster's 4 splits (log-sum-exp) into the head output
                    const int row_j = warp;
                    const bool row_on = row_j < MT && s_seq[min(row_j, MT - 1)] >= 0;
                    if (row_on) {
                        float Mx = -INFINITY;
#pragma unroll
                        for (int r = 0; r < CL; ++r) Mx = fmaxf(Mx, parts[(r * MT + row_j) * PARTW]);
                        float r0 = 0.f, r1 = 0.f, Lsum = 0.f;
#pragma unroll
                        for (int r = 0; r < CL; ++r) {
                            const float* pr = parts + (r * MT + row_j) * PARTW;
                            const float wgt = pr[0] == -INFINITY ? 0.f : expf(pr[0] - Mx);
                            Lsum = fmaf(wgt, pr[1], Lsum);
                            r0 = fmaf(wgt, pr[2 + 2 * lane], r0);
                            r1 = fmaf(wgt, pr[3 + 2 * lane], r1);
                        }
                        attn[row_j * HEAD_DIM + 2 * lane] = r0 / Lsum;
                        attn[row_j * HEAD_DIM + 2 * lane + 1] = r1 / Lsum;
                    } else if (row_j < MT) {
                        attn[row_j * HEAD_DIM + 2 * lane] = 0.f;
                        attn[row_j * HEAD_DIM + 2 * lane + 1] = 0.f;
                    }
                }
                consumer_sync();
                for (int i = tid; i < MT * HEAD_DIM; i += NTHREADS) {
                    const __nv_bfloat16 hi = __float2bfloat16_rn(attn[i]);
                    const int at = (i / HEAD_DIM) * (HEAD_DIM + 8) + i % HEAD_DIM;
                    attnb[at] = hi;
                    attnb[MT * (HEAD_DIM + 8) + at] = __float2bfloat16_rn(attn[i] - __bfloat162float(hi));
                }
                consumer_sync();
                phase_mark(a, 2 * l, 5);
                ok = consumer_all(wait_items(item, n_wo_st));
                phase_mark(a, 2 * l, 6);
                float* ytile = xs;  // [MT][orows]
                if (ok) {
                    const RingRows w{R.base, ring_slot(item, R.nst), R.nst, 7, HEAD_DIM * 2};  // 128 rows per stage
                    ring_rows_tiles<MT>(w, orows, HEAD_DIM, attnb, ytile);
                }
                release_items(item, n_wo_st);
                item += n_wo_st;
                ok = consumer_all(ok);
                if (!ok) break;
                phase_mark(a, 2 * l, 7);
#pragma unroll
                for (int k = 0; k < RES_N; ++k) {
                    const int o = tid + k * NTHREADS;
                    const int m = o / orows, t = o % orows;
                    if (o >= orows * MT || s_seq[m] < 0) continue;
                    atomicAdd(x_mid + (size_t)m * d + rank * orows + t, ytile[o] + resr[k]);
                }
            }
            load_f_params(l);  // before the barrier: independent of x_mid
            phase_end(a, 2 * l);
            target += (unsigned)G;
            if (!grid_sync(a.bar, target, a.err, &s_abort)) {
                ok = false;
                break;
            }
            // ======================================================= phase F
            phase_start(a, 2 * l + 1);
            if (fcl) issue_rows(x_mid);
            if (2 * l + 2 <= 2 * a.L - 1) zero_part(tbuf(2 * l + 2));
            if (l == a.L - 1) pdl_launch_dependents();
            if (fcl) {
                ok = consumer_all(wait_rows());  // x_mid(l), multicast into this CTA's x area
                if (!ok) break;
                float4 resv[RES_PER];  // residual cluster: x_mid + b2 of the columns this CTA reduces
#pragma unroll
                for (int k = 0; k < RES_PER; ++k) {
                    const int i = tid + k * NTHREADS;
                    resv[k] = b2v[k];
                    if (res_cl && i < MT * orows / 4) {
                        const int m = i / (orows / 4), c = rank * orows + (i % (orows / 4)) * 4;
                        const float4 xv = *reinterpret_cast<const float4*>(xs + (size_t)m * d + c);
                        resv[k].x += xv.x;
                        resv[k].y += xv.y;
                        resv[k].z += xv.z;
                        resv[k].w += xv.w;
                    }
                }
                RowRegs<MT> xr;
                if (fr > 0) load_resid(xr, xs);
                consumer_sync();  // every thread holds its rows before LN overwrites the x area
                if (fr > 0) {
                    ln_rows(xr, g2, be2);
                    phase_mark(a, 2 * l + 1, 0);
                    ok = consumer_all(wait_items(item, ffn.y));
                    phase_mark(a, 2 * l + 1, 1);
                    if (ok) {
                        const RingRows w{R.base, ring_slot(item, R.nst), R.nst, rps_shift, d * 2};
                        ring_rows_ksplit<MT>(w, fr, d, xb, xs, accs);
                    }
                    release_items(item, ffn.y);
                    item += ffn.y;
                    if (!ok) break;
                    phase_mark(a, 2 * l + 1, 2);
                    for (int k = 0; k < 2; ++k) {
                        const int o = tid + k * NTHREADS;
                        if (o >= MT * rpad) continue;
                        const int m = o / rpad, f = o % rpad;
                        const float v = f < fr ? gelu_erf(accs[f * MT + m] + b1v[k]) : 0.f;
                        const __nv_bfloat16 hi = __float2bfloat16_rn(v);
                        ub[m * (rpad + 8) + f] = hi;
                        ub[(MT + m) * (rpad + 8) + f] = __float2bfloat16_rn(v - __bfloat162float(hi));
                    }
                    consumer_sync();
                    ok = consumer_all(wait_items(item, ffn.y));
                    phase_mark(a, 2 * l + 1, 3);
                    if (ok) {
                        const RingRows w{R.base, ring_slot(item, R.nst), R.nst, rps_shift, d * 2};
                        ring_cols_trans_push<MT>(w, fr, rpad, d, ub, yrecv, &xf_bar, rank);
                    }
                    release_items(item, ffn.y);
                    item += ffn.y;
                    if (!ok) break;
                    phase_mark(a, 2 * l + 1, 4);
                }
                ok = consumer_all(mbar_wait_cluster(&xf_bar, par, a.err));
                if (!ok) break;
                phase_mark(a, 2 * l + 1, 5);
                // this CTA's columns: the cluster's partials + (residual cluster) x_mid + b2
#pragma unroll
                for (int k = 0; k < RES_PER; ++k) {
                    const int i = tid + k * NTHREADS;
                    if (i >= MT * orows / 4) continue;
                    const int m = i / (orows / 4), c4 = (i % (orows / 4)) * 4;
                    if (s_seq[m] < 0) continue;
                    float4 y = resv[k];
#pragma unroll
                    for (int r = 0; r < CL; ++r) {
                        if (a.ffn_range[cl * CL + r].y == 0) continue;
                        const float4 p = *reinterpret_cast<const float4*>(yrecv + ((size_t)r * MT + m) * orows + c4);
                        y.x += p.x;
                        y.y += p.y;
                        y.z += p.z;
                        y.w += p.w;
                    }
                    atomicAdd(reinterpret_cast<float4*>(x_out + (size_t)m * d + rank * orows + c4), y);
                }
                consumer_sync();  // every thread is done with yrecv before it is re-armed
                if (tid == 0) mbar_arrive_expect_tx(&xf_bar, xf_bytes);
                phase_mark(a, 2 * l + 1, 6);
            }
            if (l + 1 < a.L) load_a_params(l + 1);  // before the barrier: independent of x(l + 1)
            phase_end(a, 2 * l + 1);
            if (l + 1 < a.L) {
                target += (unsigned)G;
                if (!grid_sync(a.bar, target, a.err, &s_abort)) {
                    ok = false;
                    break;
                }
            }
        }
        if (!ok) s_abort = 1;
        if (tid == 0) s_consumed = item;
        trace_mark(a.trace, 7);
    }
    __syncthreads();  // producer and consumers are done
    if (tid == 0 && s_abort)  // copies issued but never consumed: wait for them (bounded) before leaving
        for (int i = s_consumed; i < s_issued; ++i) ring_wait_full(R, i, nullptr);
    __syncwarp();
    // no CTA leaves while a peer may still push into its shared memory
    cluster_arrive_release();
    cluster_wait();
    if (tid == 0) {  // the last CTA out resets the grid-barrier words for the next launch
        __threadfence();
        if (atomicAdd(a.bar + 1, 1u) == (unsigned)G - 1) {
            a.bar[0] = 0;
            a.bar[1] = 0;
            __threadfence();
        }
    }
}

// Self-test of the grid barrier's bound: the one CTA of the launch waits for
// two arrivals, only its own comes, the wait gives up after its poll limit,
// sets the error word and the CTA returns.  The counter is reset on the way out.
__device__ unsigned g_selftest_grid_ctr;

__global__ void __launch_bounds__(THREADS) selftest_grid_kernel(int* err) {
    __shared__ int s_abort;
    if (threadIdx.x == 0) s_abort = 0;
    __syncthreads();
    if (threadIdx.x >= NTHREADS) return;  // the producer warp takes no part in grid barriers
    grid_sync(&g_selftest_grid_ctr, 2u, err, &s_abort);
    if (threadIdx.x == 0) atomicExch(&g_selftest_grid_ctr, 0u);
}

}  // namespace

int step_ring_stages(int d, int mt) {
    // the most ring stages that fit the 227 KB a CTA may use beside its static shared memory
    const int limit = 227 * 1024 - 2048;
    int nst = SK_MAX_STAGES;
    while (nst > 4 && (int)SkLayout(d, mt, nst).total > limit) --nst;
    return nst;
}

cudaError_t step_kernel_configure(int d, int* max_clusters) {
    // co-residency with the largest shared-memory footprint (8 fed rows)
    const size_t smem = SkLayout(d, MAX_ROWS, step_ring_stages(d, MAX_ROWS)).total;
    auto kern = step_kernel<MAX_ROWS>;
    cudaError_t e = ensure_kernel_smem(reinterpret_cast<const void*>(kern), smem, true);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(CL);
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CL;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaOccupancyMaxActiveClusters(max_clusters, kern, &cfg);
}

template <int MT>
cudaError_t launch_step_t(const StepArgs& a, int grid, cudaStream_t s, bool pdl) {
    auto kern = step_kernel<MT>;
    const size_t smem = SkLayout(a.d, MT, a.ring_stages).total;
    cudaError_t e = ensure_kernel_smem(reinterpret_cast<const void*>(kern), smem, true);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, a);
}

cudaError_t launch_step_kernel(const StepArgs& a, int grid, cudaStream_t s, bool pdl) {
    if (a.rows < 1 || a.rows > MAX_ROWS || grid % CL || grid / CL < a.H || a.L < 2 ||
        a.ring_stages < 4 || a.ring_stages > SK_MAX_STAGES)
        return cudaErrorInvalidValue;
    if (a.rows <= 1) return launch_step_t<1>(a, grid, s, pdl);
    if (a.rows <= 2) return launch_step_t<2>(a, grid, s, pdl);
    if (a.rows <= 4) return launch_step_t<4>(a, grid, s, pdl);
    return launch_step_t<8>(a, grid, s, pdl);
}

cudaError_t launch_selftest_grid_barrier(int* err, cudaStream_t s) {
    selftest_grid_kernel<<<1, THREADS, 0, s>>>(err);
    return cudaGetLastError();
}

}  // namespace mtp
