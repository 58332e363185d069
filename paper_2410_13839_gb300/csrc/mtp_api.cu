// mtp_api.cu -- the C ABI of include/mtp.h over libmtp's kernels.
//
// Host runtime: weight upload, KV page allocator (host free list, device
// block table), slot state kept on the device, and the step orchestration:
//   decode step = for each chunk of <= 8 fed rows: embed, then per layer
//                 [LN1+QKV+KV append, attention, O-proj+residual,
//                  LN2+FFN1+GELU, FFN2+residual]; then the heads
//                 (LN_f + n x V logits) and one select kernel (log-softmax,
//                 top-k, Viterbi, acceptance, slot bookkeeping);
//   prefill      = the same layer stack over the prompt in chunks of 8 rows.
// Within a pass the kernels are chained with programmatic dependent launch;
// each (n_heads, top_k) decode step is captured once into a CUDA graph.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <map>
#include <mutex>
#include <tuple>
#include <string>
#include <utility>
#include <vector>

#include "common.cuh"
#include "kernels.cuh"
#include "mtp.h"

using namespace mtp;

namespace {

thread_local std::string g_err;

int fail(int code, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    g_err = buf;
    return code;
}

}  // namespace

cudaError_t mtp::ensure_kernel_smem(const void* kernel, size_t bytes, bool max_shared_carveout) {
    static std::mutex mu;
    static std::map<std::pair<const void*, int>, size_t> done;  // (kernel, device) -> configured bytes
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    size_t& have = done[{kernel, dev}];
    if (have >= bytes) return cudaSuccess;
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess && max_shared_carveout)
        e = cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 (int)cudaSharedmemCarveoutMaxShared);
    if (e == cudaSuccess) have = bytes;
    return e;
}

// error reporting for C-ABI functions defined in other translation units
int mtp::report_error(int code, const char* msg) {
    g_err = msg;
    return code;
}
void mtp::clear_error() { g_err.clear(); }

namespace {

#define CUDA_TRY(expr)                                                                                  \
    do {                                                                                                \
        cudaError_t e_ = (expr);                                                                        \
        if (e_ != cudaSuccess)                                                                          \
            return fail(MTP_ERR_CUDA, "%s: %s (%s:%d)", #expr, cudaGetErrorString(e_), __FILE__, __LINE__); \
    } while (0)

#define MTP_TRY(expr)              \
    do {                           \
        int r_ = (expr);           \
        if (r_ != MTP_OK) return r_; \
    } while (0)

struct Layer {
    const float *ln1_g, *ln1_b, *bqkv, *bo, *ln2_g, *ln2_b, *b1, *b2;
    const void *wqkv, *wo, *w1, *w2;
};

struct Prof {
    std::vector<std::pair<int, std::pair<cudaEvent_t, cudaEvent_t>>> ev;
};

bool is_device_ptr(const void* p) {
    if (!p) return false;
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

}  // namespace

struct mtp_ctx {
    mtp_config cfg{};
    cudaStream_t stream = nullptr;
    cudaStream_t cap_stream = nullptr;
    int device = 0, num_sms = 0, wbytes = 2;
    int mlp_clusters = 1;  // MLP clusters co-resident in one wave
    bool use_graphs = true, use_pdl = true, use_l2_prefetch = false;
    bool use_attn_tc = false;  // prefill passes: tensor-core attention (option; measured slower, see mtp.h)
    int use_heads_tc = 1;  // fused heads kernel: 0 never, 1 stand-alone heads calls, 2 also batched decode steps
    bool gemm_cluster = true;  // batched projections: one 128-row activation tile, K splits summed in clusters
    std::vector<void*> allocs;
    // weights
    void* d_weights = nullptr;
    const void *tok_phone = nullptr, *tok_codec = nullptr, *w_heads = nullptr;
    const float *lnf_g = nullptr, *lnf_b = nullptr, *b_heads = nullptr, *log_q = nullptr;
    std::vector<Layer> layers;
    // batched path (bf16 weights; more fed rows than one fused pass takes): tensor-core
    // projections over all rows of a step, row-wise glue kernels, split-KV attention
    bool use_batched = true, batched_ok = false;
    int bm_max = 0;  // rows of the batched buffers: max_batch * n_heads_max
    uint16_t* d_w2p = nullptr;  // W2 [layers][d][F] as stored in the blob (the fused kernels keep it transposed)
    float *d_bx = nullptr, *d_bqkv = nullptr, *d_bq = nullptr, *d_bh = nullptr;
    float* d_bws = nullptr;  // attention split partials
    int* d_bwc = nullptr;    // attention split counters
    int battn_ws_units = 1;  // (group, split) pairs the attention workspace holds
    int gemm_max_splits = 16;
    int lattice = 0;  // MTP_OPT_LATTICE
    int sampling = 0;          // MTP_OPT_SAMPLING
    uint32_t sample_seed = 0;  // MTP_OPT_SEED
    __nv_bfloat16 *d_ahi = nullptr, *d_alo = nullptr, *d_uhi = nullptr, *d_ulo = nullptr;
    struct LayerMaps {
        CUtensorMap wqkv, wo, w1, w2;
    };
    std::vector<LayerMaps> lmaps;
    CUtensorMap heads_map;  // the heads [n_heads_max * V][d] as GEMM weights (batched decode)
    CUtensorMap heads_map144;  // the same rows in boxes of 144 (the fused heads' last vocabulary slice)
    bool heads_tc_ok = false;  // the fused heads kernel serves this model (tensor maps, vocabulary size)
    CUtensorMap amap_hi[3], amap_lo[3], umap_hi[3], umap_lo[3];  // activation tiles of 32, 64, 128 rows
    float* d_pe = nullptr;
    // KV cache
    uint16_t* d_kv = nullptr;
    int n_pages = 0, pages_per_seq = 0;
    long long page_elems = 0;
    std::vector<int> free_pages;
    std::vector<std::vector<int>> slot_pages;
    std::vector<int> h_block_table;
    int* d_block_table = nullptr;
    // slot state
    int *d_len = nullptr, *d_npend = nullptr, *d_pending = nullptr, *d_remaining = nullptr, *d_done = nullptr,
        *d_active = nullptr, *d_gen_count = nullptr, *d_gen_tokens = nullptr, *d_prompt = nullptr;
    float* d_h_last = nullptr;
    // step buffers
    float *d_xb = nullptr, *d_logits = nullptr, *d_lse = nullptr, *d_cand_logp = nullptr;  // d_xb: 3 residual buffers
    int *d_row_seq = nullptr, *d_row_pos = nullptr, *d_row_last = nullptr, *d_cand_ids = nullptr, *d_path = nullptr,
        *d_out_tokens = nullptr, *d_out_accepted = nullptr;
    int* d_err = nullptr;
    int* d_kept = nullptr;  // VERIFY_GREEDY: drafts kept this step, per slot
    // admitted prompts (mtp_admit), run in the prefill lane of the batched steps
    int *d_prompt_left = nullptr, *d_prompt_nph = nullptr, *d_lane_take = nullptr;
    std::vector<int> h_prompt_left;  // host copy of prompt_left, advanced by the same rule as the device
    std::map<std::tuple<int, int, int>, cudaGraphExec_t> graphs;  // (n_heads, top_k, traced)
    std::map<std::tuple<int, int, int>, std::vector<int>> graph_kinds;
    int last_n = 0, last_k = 0;
    // persistent step kernel (bf16 weights, passes of <= 8 fed rows)
    bool use_persistent = false, sk_ok = false;  // measured slower than the block kernels at B = 1
    int sk_grid = 0, sk_unit_rows = 0, sk_res_cluster = 0;
    int sk_stages[4] = {0, 0, 0, 0};  // ring stages for passes of 1, 2, 4 and 8 rows
    long long sk_layer_stride = 0;
    float* d_skx = nullptr;         // residual rows [4][MAX_ROWS][d]
    unsigned* d_skbar = nullptr;    // grid-barrier words
    int2* d_skffn = nullptr;        // FFN units of each CTA
    // launch timeline (mtp_trace_step)
    unsigned long long* d_trace = nullptr;
    int trace_cap = 0;
    bool tracing = false;
    std::vector<int> trace_kinds;

    template <typename T>
    int alloc(T** p, size_t count) {
        void* q = nullptr;
        CUDA_TRY(cudaMalloc(&q, std::max<size_t>(count * sizeof(T), 16)));
        allocs.push_back(q);
        CUDA_TRY(cudaMemset(q, 0, std::max<size_t>(count * sizeof(T), 16)));
        *p = static_cast<T*>(q);
        return MTP_OK;
    }
};

namespace {

// ------------------------------------------------------------ launching ----

int record(Prof* prof, int kind, cudaStream_t s, bool start) {
    if (!prof) return MTP_OK;
    if (start) {
        cudaEvent_t a, b;
        CUDA_TRY(cudaEventCreate(&a));
        CUDA_TRY(cudaEventCreate(&b));
        prof->ev.push_back({kind, {a, b}});
        CUDA_TRY(cudaEventRecord(a, s));
    } else {
        CUDA_TRY(cudaEventRecord(prof->ev.back().second.second, s));
    }
    return MTP_OK;
}

#define LAUNCH(kind, expr)                                                                                  \
    do {                                                                                                   \
        MTP_TRY(record(prof, kind, s, true));                                                              \
        cudaError_t e_ = (expr);                                                                           \
        if (e_ != cudaSuccess)                                                                             \
            return fail(MTP_ERR_CUDA, "launch %s: %s (%s:%d)", #kind, cudaGetErrorString(e_), __FILE__, __LINE__); \
        MTP_TRY(record(prof, kind, s, false));                                                             \
    } while (0)

// CTAs and rows per CTA of a projection: one wave over the SMs while the
// weight slice fits the shared-memory budget, else more CTAs.
int gemv_grid(const mtp_ctx* c, int N, int K, int M, int* rpc) {
    int ctas = c->num_sms;
    for (;;) {
        *rpc = (N + ctas - 1) / ctas;
        if ((size_t)*rpc * K * c->wbytes <= 112 * 1024 || *rpc == 1) break;
        ctas *= 2;
    }
    return (N + *rpc - 1) / *rpc;
}

// Timeline record of the next launch (null unless a traced step is being enqueued).
unsigned long long* tslot(mtp_ctx* c, int kind) {
    if (!c->tracing || (int)c->trace_kinds.size() >= c->trace_cap) return nullptr;
    c->trace_kinds.push_back(kind);
    return c->d_trace + TRACE_WORDS * (c->trace_kinds.size() - 1);
}

GemvArgs gemv_base(mtp_ctx* c) {
    GemvArgs a;
    std::memset(&a, 0, sizeof(a));
    a.ln_eps = c->cfg.ln_eps;
    a.err = c->d_err;
    a.row_seq = c->d_row_seq;
    a.row_pos = c->d_row_pos;
    a.row_last = c->d_row_last;
    return a;
}

// Residual buffer of the rotation: in(l), mid(l) = in(l)+1, out(l) = in(l)+2 (mod 3),
// with out(l) = in(l + 1).  Layer 0 reads buffer 0 (written by the embedding).
float* xbuf(mtp_ctx* c, int i) { return c->d_xb + (size_t)(((i % 3) + 3) % 3) * MAX_ROWS * c->cfg.d_model; }
int x_in_index(int l) { return (3 - l % 3) % 3; }

// CTAs of the MLP kernel (clusters that are co-resident in one wave) and FFN rows per CTA.
int mlp_grid(const mtp_ctx* c, int* rpc) {
    const int ctas = std::max(1, c->mlp_clusters) * MLP_CLUSTER;
    *rpc = (c->cfg.d_ffn + ctas - 1) / ctas;
    const int used = (c->cfg.d_ffn + *rpc - 1) / *rpc;
    return (used + MLP_CLUSTER - 1) / MLP_CLUSTER * MLP_CLUSTER;
}

// The block stack over the M rows the embedding put in buffer 0 (G groups of rpg
// rows); returns the buffer holding the final hidden states.
int run_layers(mtp_ctx* c, int M, int G, int rpg, int plan, int seq_base, int val_seq, int val_old, int val_new,
               cudaStream_t s, bool pdl, Prof* prof, float** final_x) {
    (void)G;
    const mtp_config& cf = c->cfg;
    const int d = cf.d_model, H = cf.n_attn_heads, P = cf.page_size;
    const bool bf = cf.weight_dtype == MTP_BF16;
    int rpc;
    const int grid_b = mlp_grid(c, &rpc);
    for (int l = 0; l < cf.layers; ++l) {
        const Layer& L = c->layers[l];
        const int xi = x_in_index(l);
        LayerArgs a;
        std::memset(&a, 0, sizeof(a));
        a.M = M; a.d = d; a.d_ffn = cf.d_ffn; a.n_heads = H; a.rows_per_group = rpg;
        a.row_seq = c->d_row_seq; a.row_pos = c->d_row_pos; a.ln_eps = cf.ln_eps;
        a.kv_pool = reinterpret_cast<__nv_bfloat16*>(c->d_kv); a.page_elems = c->page_elems;
        a.layer_off = (long long)l * 2 * H * P * HEAD_DIM; a.page_size = P;
        a.block_table = c->d_block_table; a.bt_stride = c->pages_per_seq;
        a.plan = plan; a.seq_len = c->d_len; a.seq_new = c->d_npend; a.seq_base = seq_base;
        a.val_seq = val_seq; a.val_old = val_old; a.val_new = val_new;
        a.active = c->d_active; a.done = c->d_done; a.slots = cf.max_batch;
        a.err = c->d_err;
        const Layer* next = l + 1 < cf.layers && c->use_l2_prefetch ? &c->layers[l + 1] : nullptr;

        LayerArgs at = a;
        at.x_in = xbuf(c, xi); at.x_out = xbuf(c, xi + 1); at.x_zero = xbuf(c, xi + 2);
        at.ln_g = L.ln1_g; at.ln_b = L.ln1_b;
        at.wqkv = L.wqkv; at.bqkv = L.bqkv; at.wo = L.wo; at.bo = L.bo;
        at.next_w_a = next ? next->wqkv : nullptr; at.next_w_b = next ? next->wo : nullptr;
        at.trace = tslot(c, MTP_K_ATTN_BLOCK);
        LAUNCH(MTP_K_ATTN_BLOCK, launch_attn_block(at, bf, s, pdl));

        LayerArgs mb = a;
        mb.x_in = xbuf(c, xi + 1); mb.x_out = xbuf(c, xi + 2); mb.x_zero = xbuf(c, xi);
        mb.ln_g = L.ln2_g; mb.ln_b = L.ln2_b;
        mb.w1 = L.w1; mb.w2t = L.w2; mb.b1 = L.b1; mb.b2 = L.b2; mb.ffn_rows_per_cta = rpc;
        mb.next_w_a = next ? next->w1 : nullptr; mb.next_w_b = next ? next->w2 : nullptr;
        mb.trace = tslot(c, MTP_K_MLP);
        LAUNCH(MTP_K_MLP, launch_mlp(mb, bf, grid_b, s, pdl));
    }
    *final_x = xbuf(c, x_in_index(cf.layers - 1) + 2);
    return MTP_OK;
}

// K splits of a tensor-core GEMM: as many as keep one wave of CTAs (one per
// SM) with a whole number of 64-wide k-chunks each, up to c->gemm_max_splits
// (every split adds its partial tile to the output with fp32 atomics).
int gemm_splits(const mtp_ctx* c, int n_w, int k, int ntiles) {
    const int tiles = n_w / 128 * ntiles, chunks = k / 64;
    int s = 1;
    while (2 * s <= c->gemm_max_splits && chunks % (2 * s) == 0 && tiles * 2 * s <= c->num_sms) s *= 2;
    return s;
}

int tile_index(int nt) { return nt == 32 ? 0 : (nt == 64 ? 1 : 2); }

// The block stack over the M rows the embedding put in d_bx, as tensor-core
// projections plus row-wise kernels; the final hidden rows stay in d_bx.
// Attention groups: `groups` runs of rpg rows, each of one slot (decode:
// slot b's fed rows b*n.., plan PLAN_DEVICE; prefill: 8 consecutive prompt
// positions, plan PLAN_ROWS).  prefill_keys > 0: a prefill pass whose rows see
// at most that many keys; its attention runs on the tensor cores (tiles of 128
// rows) unless that option is off.
int run_layers_batched(mtp_ctx* c, int M, int rpg, int groups, int plan, cudaStream_t s, bool pdl, Prof* prof,
                       int prefill_keys = 0) {
    const mtp_config& cf = c->cfg;
    const int d = cf.d_model, F = cf.d_ffn, H = cf.n_attn_heads, P = cf.page_size;
    // activation tiles: a weight tile is streamed once per activation tile.  32-row
    // tiles keep enough CTAs streaming where K is short (q|k|v and W1 finish their
    // rows in the epilogue, one K split; W_o splits K); W2 (K = 4 d) takes whole
    // 128-row tiles and splits its long K instead
    // activation tiles: a weight tile is streamed once per activation tile, so more than 128 rows
    // take 128-row tiles (B = 128 decode, 512 rows: 1599 vs 2133 us per step with 32-row tiles);
    // up to 128 rows the projections without an accumulated output run one tile with K split over
    // a cluster (option, default), the others 32-row tiles (W_o: more CTAs) or 128 (W2, long K)
    auto tile_rows = [&](int k, int epilogue) {
        if (M > 128) return 128;
        return c->gemm_cluster && epilogue != TC_ACCUM ? tc_tile_rows(M) : std::min(k > 1024 ? 128 : 32, tc_tile_rows(M));
    };
    for (int l = 0; l < cf.layers; ++l) {
        const Layer& L = c->layers[l];
        const mtp_ctx::LayerMaps& W = c->lmaps[l];
        const long long layer_off = (long long)l * 2 * H * P * HEAD_DIM;
        auto pack = [&](int mode, const float* x, int k, const float* g, const float* bta, float* zero,
                        __nv_bfloat16* hi, __nv_bfloat16* lo) -> int {
            PackArgs pa;
            std::memset(&pa, 0, sizeof(pa));
            pa.mode = mode; pa.x = x; pa.ldx = k; pa.zero_after = zero; pa.gamma = g; pa.beta = bta;
            pa.eps = cf.ln_eps; pa.row_seq = c->d_row_seq; pa.hi = hi; pa.lo = lo; pa.k = k; pa.m = M;
            pa.trace = tslot(c, MTP_K_PACK);
            LAUNCH(MTP_K_PACK, launch_pack_rows(pa, s, pdl));
            return MTP_OK;
        };
        auto gemm = [&](const CUtensorMap& w, int n_w, int k, bool a_is_u, int epilogue, float* out, int ldo,
                        const float* bias, int w_rows_per_kchunk) -> int {
            const int nt = tile_rows(k, epilogue), ti = tile_index(nt), ntiles = (M + nt - 1) / nt;
            TcGemm g;
            std::memset(&g, 0, sizeof(g));
            g.w = w;
            g.a_hi = a_is_u ? c->umap_hi[ti] : c->amap_hi[ti];
            g.a_lo = a_is_u ? c->umap_lo[ti] : c->amap_lo[ti];
            g.n_w = n_w; g.nt = nt;
            int sc = 1;
            if (c->gemm_cluster && epilogue != TC_ACCUM) {  // K splits summed in a cluster, then the epilogue
                g.splits = std::min(gemm_splits(c, n_w, k, ntiles), TC_CLUSTER_SPLITS);
                sc = g.splits;
            } else {  // accumulated outputs: K splits added by atomics
                g.splits = epilogue == TC_ACCUM ? gemm_splits(c, n_w, k, ntiles) : 1;
            }
            TcGemmArgs& ga = g.args;
            ga.cluster_reduce = sc;
            ga.out = out; ga.ldo = ldo; ga.bias = bias; ga.m = M;
            ga.k_chunks = k / 64 / g.splits; ga.w_rows_per_kchunk = w_rows_per_kchunk;
            ga.epilogue = epilogue; ga.err = c->d_err;
            ga.row_seq = c->d_row_seq; ga.row_pos = c->d_row_pos;
            ga.kv_pool = reinterpret_cast<__nv_bfloat16*>(c->d_kv); ga.page_elems = c->page_elems;
            ga.layer_off = layer_off; ga.page_size = P; ga.n_heads = H;
            ga.block_table = c->d_block_table; ga.bt_stride = c->pages_per_seq;
            ga.pack_hi = c->d_uhi; ga.pack_lo = c->d_ulo;
            ga.trace = tslot(c, MTP_K_GEMM);
            LAUNCH(MTP_K_GEMM, launch_tc_gemm(g, s, pdl));
            return MTP_OK;
        };
        // LN1 -> q|k|v: queries out, keys and values appended to the cache
        MTP_TRY(pack(PACK_LN, c->d_bx, d, L.ln1_g, L.ln1_b, nullptr, c->d_ahi, c->d_alo));
        MTP_TRY(gemm(W.wqkv, 3 * d, d, false, TC_QKV, c->d_bq, d, L.bqkv, 0));
        // attention of every group's fed rows over its cached keys
        AttnArgs at;
        std::memset(&at, 0, sizeof(at));
        at.q = c->d_bq; at.ldq = d;
        at.kv_pool = reinterpret_cast<const __nv_bfloat16*>(c->d_kv); at.page_elems = c->page_elems;
        at.layer_off = layer_off;
        at.block_table = c->d_block_table; at.bt_stride = c->pages_per_seq;
        at.row_seq = c->d_row_seq; at.row_pos = c->d_row_pos;
        at.out_hi = c->d_ahi; at.out_lo = c->d_alo; at.ldb = d;  // straight into W_o's operand
        at.ws_part = c->d_bws; at.ws_count = c->d_bwc;
        at.rows_per_group = rpg; at.n_heads = H; at.page_size = P;
        // key splits.  Decode steps: about 2.5 waves of CTAs at four per SM, so the slots with the
        // longest contexts do not set the launch's length (B = 32 serving: 3 splits, 888 vs 972 us
        // per step with one; B = 128: one split, two measured 5.6 % slower).  Prefill passes: one
        // wave (their groups of 8 positions have similar key counts; the decode rule measured 13 %
        // slower at B = 32).
        {
            int want = attn_splits_for(groups, H, P, cf.max_ctx, c->num_sms);
            if (plan == PLAN_DEVICE) {
                const double waves = 2.5 * ATTN_CTAS_PER_SM * c->num_sms / std::max(1, groups * H);
                want = std::min({(int)std::lround(waves), (cf.max_ctx + P - 1) / P, ATTN_MAX_SPLITS});
            }
            at.n_splits = std::max(1, std::min(want, c->battn_ws_units / std::max(1, groups)));
        }
        at.plan = plan; at.seq_len = c->d_len; at.seq_new = c->d_npend; at.seq_base = 0;
        at.err = c->d_err; at.kv_swizzled = 1;
        if (prefill_keys > 0 && c->use_attn_tc && plan == PLAN_ROWS) {
            // tiles of 128 rows; splits as many as the batched attention workspace holds (S = 1 uses none)
            const int tiles = attn_tc_tiles(M);
            const size_t ws_floats = attn_workspace_floats(c->battn_ws_units, H, 1, MAX_ROWS);
            at.rows = M;
            at.n_splits = std::max(1, std::min(attn_tc_splits_for(tiles, H, prefill_keys, c->num_sms),
                                               (int)(ws_floats / attn_tc_workspace_floats(tiles, H, 1))));
            at.trace = tslot(c, MTP_K_ATTN_TC);
            LAUNCH(MTP_K_ATTN_TC, launch_attention_tc(at, s, pdl));
        } else {
            at.trace = tslot(c, MTP_K_ATTN);
            LAUNCH(MTP_K_ATTN, launch_attention(at, groups, s, pdl));
        }
        // x += attention W_o^T + b_o (the per-head W_o blocks are the k-chunks)
        MTP_TRY(gemm(W.wo, d, d, false, TC_ACCUM, c->d_bx, d, L.bo, d));
        // x += GELU(LN2(x) W1^T + b1) W2^T + b2 (W1's epilogue writes the GELU rows as bf16 hi + lo)
        MTP_TRY(pack(PACK_LN, c->d_bx, d, L.ln2_g, L.ln2_b, nullptr, c->d_ahi, c->d_alo));
        MTP_TRY(gemm(W.w1, F, d, false, TC_GELU_PACK, nullptr, F, L.b1, 0));
        MTP_TRY(gemm(W.w2, d, F, true, TC_ACCUM, c->d_bx, d, L.b2, 0));
    }
    return MTP_OK;
}

// The persistent step kernel: ring stages, grid (clusters resident at once),
// and the FFN units of each CTA (one ring stage of W1 rows plus the same rows of
// W2^T each): spread evenly over every CTA, the remainder to the CTAs without
// attention work first.  Leaves sk_ok false where the path does not apply.
int setup_step_kernel(mtp_ctx* c) {
    const mtp_config& cf = c->cfg;
    const int d = cf.d_model, F = cf.d_ffn, H = cf.n_attn_heads;
    if (c->wbytes != 2 || (d != 256 && d != 512 && d != 1024) || cf.layers < 2 || c->layers.size() < 2)
        return MTP_OK;
    const long long stride = (const char*)c->layers[1].wqkv - (const char*)c->layers[0].wqkv;
    auto same_stride = [&](const void* p0, const void* p1) { return (const char*)p1 - (const char*)p0 == stride; };
    const Layer &L0 = c->layers[0], &L1 = c->layers[1];
    if (!same_stride(L0.ln1_g, L1.ln1_g) || !same_stride(L0.wo, L1.wo) || !same_stride(L0.w1, L1.w1) ||
        !same_stride(L0.w2, L1.w2) || !same_stride(L0.b2, L1.b2) || !same_stride(L0.bqkv, L1.bqkv))
        return MTP_OK;
    int clusters = 0;
    if (step_kernel_configure(d, &clusters) != cudaSuccess) {
        cudaGetLastError();
        return MTP_OK;
    }
    const int nst = step_ring_stages(d, MAX_ROWS);  // the fewest (8 rows): bounds the FFN units per CTA
    clusters = std::min(clusters, c->num_sms / SK_CLUSTER);
    const int rps = SK_STAGE_BYTES / (2 * d);
    const int units = F / rps;
    const int G = clusters * SK_CLUSTER;
    const int max_units = std::min(64 / rps, nst - 2);
    if (clusters < H || F % rps || units > G * max_units) return MTP_OK;
    // every CTA takes FFN units (more CTAs, shorter chains in the MLP phase); the attention
    // CTAs, busy in the other phase, take the remainder's smaller share
    std::vector<int> count(G, units / G);
    int extra = units % G;
    for (int i = SK_CLUSTER * H; i < G && extra > 0; ++i, --extra) ++count[i];
    for (int i = 0; i < SK_CLUSTER * H && extra > 0; ++i, --extra) ++count[i];
    for (int i = 0; i < G; ++i)
        if (count[i] > max_units) return MTP_OK;
    std::vector<int2> ranges(G);
    for (int i = 0, first = 0; i < G; ++i) {
        ranges[i] = make_int2(first, count[i]);
        if (first == 0 && count[i] > 0) c->sk_res_cluster = i / SK_CLUSTER;
        first += count[i];
    }
    MTP_TRY(c->alloc(&c->d_skx, (size_t)4 * MAX_ROWS * d));
    MTP_TRY(c->alloc(&c->d_skbar, 2));
    MTP_TRY(c->alloc(&c->d_skffn, (size_t)G));
    CUDA_TRY(cudaMemcpy(c->d_skffn, ranges.data(), G * sizeof(int2), cudaMemcpyHostToDevice));
    c->sk_grid = G;
    for (int i = 0; i < 4; ++i) c->sk_stages[i] = step_ring_stages(d, 1 << i);
    c->sk_unit_rows = rps;
    c->sk_layer_stride = stride;
    c->sk_ok = true;
    return MTP_OK;
}

// One pass of <= MAX_ROWS fed rows (slots seq_base .., rpg rows each) through
// the persistent kernel; returns the buffer holding the pass's final rows.
int launch_step_pass(mtp_ctx* c, int rows, int rpg, int seq_base, cudaStream_t s, bool pdl, Prof* prof,
                     float** final_x) {
    const mtp_config& cf = c->cfg;
    const Layer& L = c->layers[0];
    StepArgs a;
    std::memset(&a, 0, sizeof(a));
    a.L = cf.layers; a.d = cf.d_model; a.F = cf.d_ffn; a.H = cf.n_attn_heads;
    a.rows = rows; a.rpg = rpg; a.seq_base = seq_base; a.slots = cf.max_batch;
    a.n_max = cf.n_heads_max; a.page_size = cf.page_size; a.codec_vocab = cf.codec_vocab; a.max_pos = cf.max_ctx;
    a.ln_eps = cf.ln_eps;
    a.ln1_g = L.ln1_g; a.ln1_b = L.ln1_b; a.bqkv = L.bqkv; a.bo = L.bo;
    a.ln2_g = L.ln2_g; a.ln2_b = L.ln2_b; a.b1 = L.b1; a.b2 = L.b2;
    a.wqkv = static_cast<const __nv_bfloat16*>(L.wqkv);
    a.wo = static_cast<const __nv_bfloat16*>(L.wo);
    a.w1 = static_cast<const __nv_bfloat16*>(L.w1);
    a.w2t = static_cast<const __nv_bfloat16*>(L.w2);
    a.layer_stride = c->sk_layer_stride;
    a.tok_codec = static_cast<const __nv_bfloat16*>(c->tok_codec);
    a.pe = c->d_pe;
    a.active = c->d_active; a.done = c->d_done; a.n_pending = c->d_npend; a.pending = c->d_pending;
    a.seq_len = c->d_len;
    a.kv_pool = reinterpret_cast<__nv_bfloat16*>(c->d_kv); a.page_elems = c->page_elems;
    a.block_table = c->d_block_table; a.bt_stride = c->pages_per_seq;
    a.ffn_range = c->d_skffn; a.ffn_unit_rows = c->sk_unit_rows; a.res_cluster = c->sk_res_cluster;
    a.ring_stages = c->sk_stages[rows <= 1 ? 0 : rows <= 2 ? 1 : rows <= 4 ? 2 : 3];
    a.xbuf = c->d_skx; a.bar = c->d_skbar;
    a.row_seq = c->d_row_seq; a.row_pos = c->d_row_pos; a.row_last = c->d_row_last;
    a.err = c->d_err;
    a.trace = nullptr;
    if (c->tracing && (int)c->trace_kinds.size() + 1 + 2 * cf.layers + 2 * c->sk_grid <= c->trace_cap) {
        a.trace = tslot(c, MTP_K_STEP);  // then one record per phase, then per CTA and phase of the middle layer
        for (int l = 0; l < cf.layers; ++l) {
            tslot(c, MTP_K_STEP_ATTN);
            tslot(c, MTP_K_STEP_MLP);
        }
        for (int i = 0; i < 2 * c->sk_grid; ++i) tslot(c, MTP_K_STEP_CTA);
    }
    LAUNCH(MTP_K_STEP, launch_step_kernel(a, c->sk_grid, s, pdl));
    *final_x = c->d_skx + (size_t)step_final_buffer(cf.layers) * MAX_ROWS * cf.d_model;
    return MTP_OK;
}

// Buffers and tensor maps of the batched path (bf16 weights only).
int setup_batched(mtp_ctx* c) {
    const mtp_config& cf = c->cfg;
    const int d = cf.d_model, F = cf.d_ffn, H = cf.n_attn_heads, P = cf.page_size;
    // every slot's fed rows plus a prefill lane of up to PREFILL_ROWS prompt rows
    c->bm_max = cf.max_batch * cf.n_heads_max + PREFILL_ROWS;
    if (c->wbytes != 2 || !c->d_w2p) return MTP_OK;
    const size_t M = (size_t)c->bm_max;
    MTP_TRY(c->alloc(&c->d_bx, M * d));
    MTP_TRY(c->alloc(&c->d_bqkv, M * 3 * d));
    MTP_TRY(c->alloc(&c->d_bq, M * d));
    MTP_TRY(c->alloc(&c->d_bh, M * F));
    uint16_t *ahi, *alo, *uhi, *ulo;
    MTP_TRY(c->alloc(&ahi, M * d));
    MTP_TRY(c->alloc(&alo, M * d));
    MTP_TRY(c->alloc(&uhi, M * F));
    MTP_TRY(c->alloc(&ulo, M * F));
    c->d_ahi = reinterpret_cast<__nv_bfloat16*>(ahi);
    c->d_alo = reinterpret_cast<__nv_bfloat16*>(alo);
    c->d_uhi = reinterpret_cast<__nv_bfloat16*>(uhi);
    c->d_ulo = reinterpret_cast<__nv_bfloat16*>(ulo);
    {  // attention workspace for the decode groups (slots, plus the lane's groups of as few as one row)
        // and the prefill groups (8-row runs)
        const int gd = cf.max_batch + PREFILL_ROWS, gp = (c->bm_max + 7) / 8;
        c->battn_ws_units = std::max(gd * attn_splits_for(gd, H, P, cf.max_ctx, c->num_sms),
                                     gp * attn_splits_for(gp, H, P, cf.max_ctx, c->num_sms));
        MTP_TRY(c->alloc(&c->d_bws, attn_workspace_floats(c->battn_ws_units, H, 1, MAX_ROWS)));
        MTP_TRY(c->alloc(&c->d_bwc, (size_t)std::max(gd, gp) * H));
    }
    c->lmaps.resize(cf.layers);
    int bad = 0;
    for (int l = 0; l < cf.layers; ++l) {
        const Layer& L = c->layers[l];
        mtp_ctx::LayerMaps& W = c->lmaps[l];
        bad |= tc_encode_2d(&W.wqkv, L.wqkv, (uint64_t)d, (uint64_t)3 * d, 128, true);
        bad |= tc_encode_2d(&W.wo, L.wo, (uint64_t)HEAD_DIM, (uint64_t)H * d, 128, true);
        bad |= tc_encode_2d(&W.w1, L.w1, (uint64_t)d, (uint64_t)F, 128, true);
        bad |= tc_encode_2d(&W.w2, c->d_w2p + (size_t)l * d * F, (uint64_t)F, (uint64_t)d, 128, false);
    }
    const int nts[3] = {32, 64, 128};
    for (int t = 0; t < 3; ++t) {
        bad |= tc_encode_2d(&c->amap_hi[t], c->d_ahi, (uint64_t)d, M, (uint32_t)nts[t], false);
        bad |= tc_encode_2d(&c->amap_lo[t], c->d_alo, (uint64_t)d, M, (uint32_t)nts[t], false);
        bad |= tc_encode_2d(&c->umap_hi[t], c->d_uhi, (uint64_t)F, M, (uint32_t)nts[t], false);
        bad |= tc_encode_2d(&c->umap_lo[t], c->d_ulo, (uint64_t)F, M, (uint32_t)nts[t], false);
    }
    bad |= tc_encode_2d(&c->heads_map, c->w_heads, (uint64_t)d, (uint64_t)cf.n_heads_max * cf.codec_vocab, 128,
                        false);
    c->heads_tc_ok = tc_encode_2d(&c->heads_map144, c->w_heads, (uint64_t)d,
                                  (uint64_t)cf.n_heads_max * cf.codec_vocab, (uint32_t)heads_tc_box_rows_wide(),
                                  false) == 0 &&
                     heads_tc_supported(cf.codec_vocab, 1);
    c->batched_ok = bad == 0;  // without tensor maps the fused path serves every batch
    return MTP_OK;
}

EmbedArgs embed_base(mtp_ctx* c) {
    EmbedArgs e;
    std::memset(&e, 0, sizeof(e));
    e.tok_phone = c->tok_phone; e.tok_codec = c->tok_codec;
    e.w_bf16 = c->cfg.weight_dtype == MTP_BF16;
    e.phone_vocab = c->cfg.phone_vocab; e.codec_vocab = c->cfg.codec_vocab;
    e.pe = c->d_pe; e.d = c->cfg.d_model; e.max_pos = c->cfg.max_ctx;
    e.x = xbuf(c, 0); e.zero_buf = xbuf(c, 1); e.row_seq = c->d_row_seq; e.row_pos = c->d_row_pos; e.row_last = c->d_row_last;
    e.n_max = c->cfg.n_heads_max; e.slots = c->cfg.max_batch;
    e.active = c->d_active; e.done = c->d_done; e.n_pending = c->d_npend; e.pending = c->d_pending;
    e.seq_len = c->d_len; e.prompt = c->d_prompt; e.prompt_stride = c->cfg.max_ctx;
    e.err = c->d_err;
    return e;
}

// Heads on the hidden states of slots [b0, b0 + m): rows of A, or, with
// `gather`, the slot's last row fed this step in the single pass `gather`.
// The heads over B hidden rows x [B][d] (B <= the batched buffers' rows) on the
// tensor cores: LN_f rows as bf16 hi + lo (the same kernel zeroes the logits),
// then one split-K GEMM over the first n heads' n V rows, added into
// logits [B][n V].
int launch_heads_batched(mtp_ctx* c, const float* x, int B, int n, float* logits, cudaStream_t s, bool pdl,
                         Prof* prof) {
    const mtp_config& cf = c->cfg;
    const int d = cf.d_model, V = cf.codec_vocab;
    PackArgs pa;
    std::memset(&pa, 0, sizeof(pa));
    pa.mode = PACK_LN; pa.x = x; pa.ldx = d; pa.gamma = c->lnf_g; pa.beta = c->lnf_b;
    pa.eps = cf.ln_eps; pa.row_seq = nullptr; pa.hi = c->d_ahi; pa.lo = c->d_alo; pa.k = d; pa.m = B;
    pa.zero_buf = logits; pa.zero_n = (long long)B * n * V;
    pa.trace = tslot(c, MTP_K_PACK);
    LAUNCH(MTP_K_PACK, launch_pack_rows(pa, s, pdl));
    const int nt = tc_tile_rows(B), ntiles = (B + nt - 1) / nt;
    const int n_w = (n * V + 127) / 128 * 128, tiles = n_w / 128, chunks = d / 64;
    int splits = 1;
    while (2 * splits <= c->gemm_max_splits && chunks % (2 * splits) == 0 && tiles * ntiles * 2 * splits <= c->num_sms)
        splits *= 2;
    TcGemm g;
    std::memset(&g, 0, sizeof(g));
    g.w = c->heads_map;
    g.a_hi = c->amap_hi[tile_index(nt)];
    g.a_lo = c->amap_lo[tile_index(nt)];
    g.n_w = n_w; g.nt = nt; g.splits = splits;
    TcGemmArgs& ga = g.args;
    ga.out = logits; ga.ldo = n * V; ga.bias = c->b_heads; ga.m = B;
    ga.k_chunks = chunks / splits; ga.epilogue = TC_ACCUM; ga.n_valid = n * V; ga.err = c->d_err;
    ga.trace = tslot(c, MTP_K_HEADS);
    LAUNCH(MTP_K_HEADS, launch_tc_gemm(g, s, pdl));
    return MTP_OK;
}

bool heads_fused_ok(const mtp_ctx* c, int k, bool decode_step) {
    return c->use_heads_tc >= (decode_step ? 2 : 1) && c->batched_ok && c->heads_tc_ok &&
           heads_tc_supported(c->cfg.codec_vocab, k);
}

// The heads fused with their log-softmax and top-k over B hidden rows x [B][d]
// (B <= the batched buffers' rows): LN_f rows as bf16 hi + lo, then one kernel
// that writes the candidates (ids, logp [B][n][k]), lse [B][n] and, when
// `logits` is not null, the logits [B][n V].
int launch_heads_fused(mtp_ctx* c, const float* x, int B, int n, int k, int32_t* ids, float* logp, float* lse,
                       float* logits, cudaStream_t s, bool pdl, Prof* prof) {
    const mtp_config& cf = c->cfg;
    const int d = cf.d_model, V = cf.codec_vocab;
    PackArgs pa;
    std::memset(&pa, 0, sizeof(pa));
    pa.mode = PACK_LN; pa.x = x; pa.ldx = d; pa.gamma = c->lnf_g; pa.beta = c->lnf_b;
    pa.eps = cf.ln_eps; pa.row_seq = nullptr; pa.hi = c->d_ahi; pa.lo = c->d_alo; pa.k = d; pa.m = B;
    pa.trace = tslot(c, MTP_K_PACK);
    LAUNCH(MTP_K_PACK, launch_pack_rows(pa, s, pdl));
    HeadsTc g;
    std::memset(&g, 0, sizeof(g));
    g.w128 = c->heads_map; g.w144 = c->heads_map144;
    const int ar = tc_tile_rows(B);  // 32, 64 or 128 activation rows per stage
    g.a_hi = c->amap_hi[tile_index(ar)]; g.a_lo = c->amap_lo[tile_index(ar)];
    HeadsTcArgs& ha = g.args;
    ha.bias = c->b_heads; ha.m = B; ha.n = n; ha.V = V; ha.k = k; ha.k_chunks = d / 64; ha.a_rows = ar;
    ha.out_ids = ids; ha.out_logp = logp; ha.out_lse = lse; ha.out_logits = logits; ha.ldl = n * V;
    ha.err = c->d_err;
    ha.trace = tslot(c, MTP_K_HEADS);
    LAUNCH(MTP_K_HEADS, launch_heads_tc(g, s, pdl));
    return MTP_OK;
}

int launch_heads(mtp_ctx* c, const float* A, int m, int n, float* logits, const float* gather, int b0,
                 cudaStream_t s, bool pdl, Prof* prof) {
    const int d = c->cfg.d_model, V = c->cfg.codec_vocab;
    GemvArgs h = gemv_base(c);
    h.A = A; h.lda = d; h.ln_g = c->lnf_g; h.ln_b = c->lnf_b;
    h.W = c->w_heads; h.bias = c->b_heads; h.N = n * V; h.K = d; h.M = m;
    int rpc;
    const int grid = gemv_grid(c, h.N, h.K, m, &rpc);
    h.rows_per_cta = rpc;
    h.row_seq = nullptr;
    h.out = logits; h.ldo = n * V;
    if (gather) {
        h.gather_x = gather; h.gather_npend = c->d_npend; h.gather_n = n; h.gather_base = b0;
    }
    h.trace = tslot(c, MTP_K_HEADS);
    LAUNCH(MTP_K_HEADS, launch_gemv(h, EPI_LOGITS, true, c->cfg.weight_dtype == MTP_BF16, grid, s, pdl));
    return MTP_OK;
}

SelectArgs select_base(mtp_ctx* c, int n, int k) {
    SelectArgs a;
    std::memset(&a, 0, sizeof(a));
    a.logits = c->d_logits; a.lse = c->d_lse; a.cand_ids = c->d_cand_ids; a.cand_logp = c->d_cand_logp;
    a.path = c->d_path; a.log_q = c->log_q;
    a.n = n; a.k = k; a.V = c->cfg.codec_vocab; a.eos_id = c->cfg.eos_id; a.n_max = c->cfg.n_heads_max;
    a.active = c->d_active; a.done = c->d_done; a.n_pending = c->d_npend; a.pending = c->d_pending;
    a.seq_len = c->d_len; a.remaining = c->d_remaining; a.gen_count = c->d_gen_count;
    a.gen_tokens = c->d_gen_tokens; a.gen_stride = c->cfg.max_ctx;
    a.out_tokens = c->d_out_tokens; a.out_accepted = c->d_out_accepted;
    a.err = c->d_err;
    a.policy = c->cfg.accept_policy; a.kept = c->d_kept; a.lattice = c->lattice;
    a.sampling = c->sampling; a.seed = c->sample_seed;
    a.prompt_left = c->d_prompt_left; a.lane_take = c->d_lane_take; a.lane = 0;
    return a;
}

// VERIFY_GREEDY: head 1 at every fed row of one pass (x: the pass's final rows,
// rows = slots * n, written to d_logits row by row), then the kept drafts and
// the last kept row's hidden state of each slot.
int enqueue_verify(mtp_ctx* c, const float* x, int slots, int n, int b0, cudaStream_t s, bool pdl, Prof* prof) {
    const int d = c->cfg.d_model, V = c->cfg.codec_vocab, rows = slots * n;
    for (int r0 = 0; r0 < rows; r0 += MAX_ROWS) {
        const int m = std::min(MAX_ROWS, rows - r0);
        MTP_TRY(launch_heads(c, x + (size_t)r0 * d, m, 1, c->d_logits + (size_t)r0 * V, nullptr, 0, s, pdl, prof));
    }
    VerifyArgs va;
    std::memset(&va, 0, sizeof(va));
    va.logits1 = c->d_logits; va.x = x; va.h_last = c->d_h_last; va.kept = c->d_kept;
    va.active = c->d_active; va.done = c->d_done; va.n_pending = c->d_npend; va.pending = c->d_pending;
    va.n = n; va.V = V; va.d = d; va.n_max = c->cfg.n_heads_max; va.seq_base = b0;
    va.trace = tslot(c, MTP_K_SELECT);
    LAUNCH(MTP_K_SELECT, launch_verify(va, slots, s, pdl));
    return MTP_OK;
}

// ---- the prefill lane (prompts admitted with mtp_admit) ----

// Prompt rows the lane of a batched step takes: up to PREFILL_ROWS, whole groups of n.
int lane_rows(int n) { return PREFILL_ROWS / n * n; }

bool lane_pending(const mtp_ctx* c) {
    for (int v : c->h_prompt_left)
        if (v > 0) return true;
    return false;
}

// The host's copy of the lane rule of lane_plan_kernel (slot order, padded demands).
void lane_mirror(mtp_ctx* c, int capacity, int rpg) {
    int start = 0;
    for (int& left : c->h_prompt_left) {
        if (left <= 0) continue;
        const int demand = (left + rpg - 1) / rpg * rpg;
        if (start < capacity) left -= std::min(left, capacity - start);
        start += demand;
    }
}

int enqueue_lane_plan(mtp_ctx* c, int row0, int capacity, int rpg, cudaStream_t s, bool pdl, Prof* prof) {
    LanePlanArgs lp;
    std::memset(&lp, 0, sizeof(lp));
    lp.slots = c->cfg.max_batch; lp.rpg = rpg; lp.capacity = capacity; lp.row0 = row0;
    lp.prompt_left = c->d_prompt_left; lp.seq_len = c->d_len; lp.active = c->d_active; lp.done = c->d_done;
    lp.row_seq = c->d_row_seq; lp.row_pos = c->d_row_pos; lp.row_last = c->d_row_last; lp.lane_take = c->d_lane_take;
    LAUNCH(MTP_K_EMBED, launch_lane_plan(lp, s, pdl));
    EmbedArgs e = embed_base(c);
    e.mode = 2; e.rows = capacity; e.row0 = row0; e.prompt_nph = c->d_prompt_nph;
    e.x = c->d_bx + (size_t)row0 * c->cfg.d_model; e.zero_buf = nullptr;
    e.trace = tslot(c, MTP_K_EMBED);
    LAUNCH(MTP_K_EMBED, launch_embed(e, s, pdl));
    return MTP_OK;
}

// chain: the step follows another step in the same stream or graph; its first
// kernel then starts under programmatic launch (it waits for the previous
// step's selection before it lets the next kernels start).
// lane: the pass also runs up to lane_rows(n) prompt rows of admitted slots
// (batched path; the caller checked that it is available).
int enqueue_step(mtp_ctx* c, int n, int k, cudaStream_t s, bool pdl, Prof* prof, bool chain = false,
                 bool lane = false) {
    const int B = c->cfg.max_batch, d = c->cfg.d_model, V = c->cfg.codec_vocab;
    const int spc = std::max(1, MAX_ROWS / n);
    const bool verify = c->cfg.accept_policy == MTP_VERIFY_GREEDY;
    // one pass feeds every slot: the heads read its rows directly (VERIFY_GREEDY: the kept row, via h_last)
    const bool single = B <= spc && !verify;
    float* final_x = nullptr;
    const int P = lane ? lane_rows(n) : 0;
    if ((B > spc || lane) && c->use_batched && c->batched_ok && B * n + P <= c->bm_max) {  // every slot's rows in one pass
        const int Md = B * n, M = Md + P;
        EmbedArgs e = embed_base(c);
        e.mode = 0; e.rows = Md; e.seq_base = 0; e.n_heads = n; e.x = c->d_bx; e.zero_buf = nullptr;
        e.trace = tslot(c, MTP_K_EMBED);
        LAUNCH(MTP_K_EMBED, launch_embed(e, s, chain && pdl));
        if (lane) MTP_TRY(enqueue_lane_plan(c, Md, P, n, s, pdl, prof));
        // with a lane the groups are read from the rows' plan (slots of n rows, then the lane's groups)
        MTP_TRY(run_layers_batched(c, M, n, M / n, lane ? PLAN_ROWS : PLAN_DEVICE, s, pdl, prof));
        if (verify) {
            MTP_TRY(enqueue_verify(c, c->d_bx, B, n, 0, s, pdl, prof));
        } else {
            unsigned long long* tr = tslot(c, MTP_K_SAVE);
            LAUNCH(MTP_K_SAVE, launch_save_last(c->d_bx, c->d_row_seq, c->d_row_last, c->d_h_last, d, M, tr, s, pdl));
        }
        const bool fused = heads_fused_ok(c, k, true);
        if (fused)  // candidates, lse and the logits (kept for mtp_debug_logits and the union lattice)
            MTP_TRY(launch_heads_fused(c, c->d_h_last, B, n, k, c->d_cand_ids, c->d_cand_logp, c->d_lse, c->d_logits,
                                       s, pdl, prof));
        else
            MTP_TRY(launch_heads_batched(c, c->d_h_last, B, n, c->d_logits, s, pdl, prof));
        SelectArgs sa = select_base(c, n, k);
        sa.pre_topk = fused ? 1 : 0;
        sa.lane = lane ? 1 : 0;
        sa.trace = tslot(c, MTP_K_SELECT);
        LAUNCH(MTP_K_SELECT, launch_select(sa, B, true, s, pdl));
        return MTP_OK;
    }
    for (int b0 = 0; b0 < B; b0 += spc) {
        const int G = std::min(spc, B - b0), M = G * n;
        if (c->use_persistent && c->sk_ok) {  // the pass's embedding and blocks in one kernel
            // it reads nothing from earlier kernels before its dependency wait: always under programmatic launch
            MTP_TRY(launch_step_pass(c, M, n, b0, s, pdl, prof, &final_x));
        } else {
            EmbedArgs e = embed_base(c);
            e.mode = 0; e.rows = M; e.seq_base = b0; e.n_heads = n;
            e.trace = tslot(c, MTP_K_EMBED);
            // full dependency on the previous pass; the step's first pass may chain to the previous step
            LAUNCH(MTP_K_EMBED, launch_embed(e, s, b0 == 0 && chain && pdl));
            MTP_TRY(run_layers(c, M, G, n, PLAN_DEVICE, b0, 0, 0, 0, s, pdl, prof, &final_x));
        }
        if (verify) {
            MTP_TRY(enqueue_verify(c, final_x, G, n, b0, s, pdl, prof));
        } else if (!single) {
            unsigned long long* tr = tslot(c, MTP_K_SAVE);
            LAUNCH(MTP_K_SAVE,
                   launch_save_last(final_x, c->d_row_seq, c->d_row_last, c->d_h_last, d, MAX_ROWS, tr, s, pdl));
        }
    }
    for (int b0 = 0; b0 < B; b0 += MAX_ROWS) {
        const int m = std::min(MAX_ROWS, B - b0);
        MTP_TRY(launch_heads(c, c->d_h_last + (size_t)b0 * d, m, n, c->d_logits + (size_t)b0 * n * V,
                             single ? final_x : nullptr, b0, s, pdl, prof));
    }
    SelectArgs sa = select_base(c, n, k);
    sa.trace = tslot(c, MTP_K_SELECT);
    LAUNCH(MTP_K_SELECT, launch_select(sa, B, true, s, pdl));
    return MTP_OK;
}

int run_step(mtp_ctx* c, int n, int k, bool lane = false) {
    c->last_n = n;
    c->last_k = k;
    if (!c->use_graphs) {
        c->trace_kinds.clear();
        return enqueue_step(c, n, k, c->stream, c->use_pdl, nullptr, false, lane);
    }
    const auto key = std::make_tuple(n, k, (c->tracing ? 1 : 0) | (lane ? 4 : 0));
    auto it = c->graphs.find(key);
    if (it == c->graphs.end()) {
        cudaGraph_t graph = nullptr;
        cudaGraphExec_t exec = nullptr;
        c->trace_kinds.clear();
        CUDA_TRY(cudaStreamBeginCapture(c->cap_stream, cudaStreamCaptureModeRelaxed));
        const int r = enqueue_step(c, n, k, c->cap_stream, c->use_pdl, nullptr, false, lane);
        const cudaError_t ec = cudaStreamEndCapture(c->cap_stream, &graph);
        if (r != MTP_OK) {
            if (graph) cudaGraphDestroy(graph);
            return r;
        }
        CUDA_TRY(ec);
        const cudaError_t ei = cudaGraphInstantiate(&exec, graph, 0);
        cudaGraphDestroy(graph);
        CUDA_TRY(ei);
        it = c->graphs.emplace(key, exec).first;
        c->graph_kinds[key] = c->trace_kinds;
    }
    c->trace_kinds = c->graph_kinds[key];
    CUDA_TRY(cudaGraphLaunch(it->second, c->stream));
    return MTP_OK;
}

// `count` decode steps: graphs of STEPS_PER_GRAPH chained steps, then single steps.
constexpr int STEPS_PER_GRAPH = 8;
int run_steps(mtp_ctx* c, int n, int k, int count) {
    if (!c->use_graphs || c->tracing) {
        for (int i = 0; i < count; ++i) MTP_TRY(run_step(c, n, k));
        return MTP_OK;
    }
    int done = 0;
    if (count >= STEPS_PER_GRAPH) {
        const auto key = std::make_tuple(n, k, 2);  // 2: the chained multi-step graph
        auto it = c->graphs.find(key);
        if (it == c->graphs.end()) {
            cudaGraph_t graph = nullptr;
            cudaGraphExec_t exec = nullptr;
            c->trace_kinds.clear();
            CUDA_TRY(cudaStreamBeginCapture(c->cap_stream, cudaStreamCaptureModeRelaxed));
            int r = MTP_OK;
            for (int i = 0; i < STEPS_PER_GRAPH && r == MTP_OK; ++i)
                r = enqueue_step(c, n, k, c->cap_stream, c->use_pdl, nullptr, i > 0);
            const cudaError_t ec = cudaStreamEndCapture(c->cap_stream, &graph);
            if (r != MTP_OK) {
                if (graph) cudaGraphDestroy(graph);
                return r;
            }
            CUDA_TRY(ec);
            const cudaError_t ei = cudaGraphInstantiate(&exec, graph, 0);
            cudaGraphDestroy(graph);
            CUDA_TRY(ei);
            it = c->graphs.emplace(key, exec).first;
            c->graph_kinds[key] = c->trace_kinds;
        }
        c->last_n = n;
        c->last_k = k;
        for (; done + STEPS_PER_GRAPH <= count; done += STEPS_PER_GRAPH) CUDA_TRY(cudaGraphLaunch(it->second, c->stream));
    }
    for (; done < count; ++done) MTP_TRY(run_step(c, n, k));
    return MTP_OK;
}

int check_device_error(mtp_ctx* c) {
    int err = 0;
    CUDA_TRY(cudaMemcpyAsync(&err, c->d_err, sizeof(int), cudaMemcpyDeviceToHost, c->stream));
    CUDA_TRY(cudaStreamSynchronize(c->stream));
    if (err) return fail(MTP_ERR_DEVICE, "device error word 0x%x (1 = bounded wait ran out, 2 = index check)", err);
    return MTP_OK;
}

int copy_out(void* dst, const void* src, size_t bytes, cudaStream_t s) {
    if (!dst || bytes == 0) return MTP_OK;
    CUDA_TRY(cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDefault, s));
    return MTP_OK;
}

int slot_set(mtp_ctx* c, int slot, int len, int pend, int rem, int done, int active, int gen, int prompt_left = -1,
             int prompt_nph = -1) {
    SlotSet ss;
    ss.slot = slot;
    ss.seq_len = c->d_len; ss.n_pending = c->d_npend; ss.remaining = c->d_remaining;
    ss.done = c->d_done; ss.active = c->d_active; ss.gen_count = c->d_gen_count;
    ss.prompt_left = c->d_prompt_left; ss.prompt_nph = c->d_prompt_nph;
    ss.set_len = len; ss.set_pending = pend; ss.set_remaining = rem;
    ss.set_done = done; ss.set_active = active; ss.set_gen = gen;
    ss.set_prompt_left = prompt_left; ss.set_prompt_nph = prompt_nph;
    CUDA_TRY(launch_slot_set(ss, c->stream));
    return MTP_OK;
}

int read_slot_ints(mtp_ctx* c, const int* dptr, std::vector<int>& out) {
    out.resize(c->cfg.max_batch);
    CUDA_TRY(cudaMemcpyAsync(out.data(), dptr, out.size() * sizeof(int), cudaMemcpyDeviceToHost, c->stream));
    CUDA_TRY(cudaStreamSynchronize(c->stream));
    return MTP_OK;
}

int validate_config(const mtp_config& c) {
    if (c.layers < 1 || c.layers > 256) return fail(MTP_ERR_INVALID, "layers %d out of range", c.layers);
    if (c.d_model < 256 || c.d_model % 256 || c.d_model > 1024)
        return fail(MTP_ERR_INVALID, "d_model %d: need a multiple of 256 up to 1024", c.d_model);
    if (c.n_attn_heads * HEAD_DIM != c.d_model)
        return fail(MTP_ERR_INVALID, "d_model / n_attn_heads must be %d", HEAD_DIM);
    if (c.d_ffn < 256 || c.d_ffn % 256 || c.d_ffn > 4096)
        return fail(MTP_ERR_INVALID, "d_ffn %d: need a multiple of 256 up to 4096", c.d_ffn);
    if (c.phone_vocab < 1) return fail(MTP_ERR_INVALID, "phone_vocab %d", c.phone_vocab);
    if (c.codec_vocab < 2 || c.codec_vocab > MAX_VOCAB)
        return fail(MTP_ERR_INVALID, "codec_vocab %d: need 2..%d", c.codec_vocab, MAX_VOCAB);
    if (c.eos_id < 0 || c.eos_id >= c.codec_vocab) return fail(MTP_ERR_INVALID, "eos_id %d", c.eos_id);
    if (c.n_heads_max < 1 || c.n_heads_max > MAX_NHEADS)
        return fail(MTP_ERR_INVALID, "n_heads_max %d: need 1..%d", c.n_heads_max, MAX_NHEADS);
    if (c.top_k_max < 1 || c.top_k_max > MAX_TOPK || c.top_k_max > c.codec_vocab)
        return fail(MTP_ERR_INVALID, "top_k_max %d: need 1..%d", c.top_k_max, MAX_TOPK);
    if (c.max_batch < 1 || c.max_batch > 1024) return fail(MTP_ERR_INVALID, "max_batch %d", c.max_batch);
    if (c.max_ctx < 2 || c.max_ctx > (1 << 20)) return fail(MTP_ERR_INVALID, "max_ctx %d", c.max_ctx);
    if (c.page_size != 16 && c.page_size != 32 && c.page_size != 64 && c.page_size != 128)
        return fail(MTP_ERR_INVALID, "page_size %d: need 16, 32, 64 or 128", c.page_size);
    if (c.n_pages < 0) return fail(MTP_ERR_INVALID, "n_pages %d", c.n_pages);
    if (c.weight_dtype != MTP_F32 && c.weight_dtype != MTP_BF16)
        return fail(MTP_ERR_INVALID, "weight_dtype %d", c.weight_dtype);
    if (c.accept_policy != MTP_ACCEPT_ALL && c.accept_policy != MTP_VERIFY_GREEDY)
        return fail(MTP_ERR_INVALID, "accept_policy %d", c.accept_policy);
    if (!(c.ln_eps > 0.f)) return fail(MTP_ERR_INVALID, "ln_eps must be > 0");
    return MTP_OK;
}

struct TensorSpec {
    size_t numel;
    bool matrix;
};

std::vector<TensorSpec> blob_specs(const mtp_config& c) {
    const size_t d = c.d_model, F = c.d_ffn, V = c.codec_vocab;
    std::vector<TensorSpec> t;
    t.push_back({(size_t)c.phone_vocab * d, true});
    t.push_back({V * d, true});
    for (int l = 0; l < c.layers; ++l) {
        t.push_back({d, false}); t.push_back({d, false});
        t.push_back({3 * d * d, true}); t.push_back({3 * d, false});
        t.push_back({d * d, true}); t.push_back({d, false});
        t.push_back({d, false}); t.push_back({d, false});
        t.push_back({F * d, true}); t.push_back({F, false});
        t.push_back({d * F, true}); t.push_back({d, false});
    }
    t.push_back({d, false}); t.push_back({d, false});
    t.push_back({(size_t)c.n_heads_max * V * d, true});
    t.push_back({(size_t)c.n_heads_max * V, false});
    t.push_back({V * V, false});
    return t;
}

// Device layouts of a block's matrices (element size es bytes):
//   j = 2  wqkv [3d][d]  -> head-major [H][q 64 | k 64 | v 64][d]
//   j = 3  bqkv [3d]     -> head-major [H][192]
//   j = 4  wo   [d][d]   -> [H][d][64]: head h's input columns of every output row
//   j = 10 w2   [d][F]   -> transposed [F][d]
void relayout(const mtp_config& cf, int j, int es, const unsigned char* src, unsigned char* dst) {
    const size_t d = cf.d_model, F = cf.d_ffn, H = cf.n_attn_heads;
    if (j == 2 || j == 3) {
        const size_t row = (j == 2 ? d : 1) * es;
        for (size_t h = 0; h < H; ++h)
            for (size_t r = 0; r < 3 * HEAD_DIM; ++r) {
                const size_t sec = r / HEAD_DIM, within = r % HEAD_DIM;
                std::memcpy(dst + (h * 3 * HEAD_DIM + r) * row, src + (sec * d + h * HEAD_DIM + within) * row, row);
            }
    } else if (j == 4) {
        for (size_t h = 0; h < H; ++h)
            for (size_t f = 0; f < d; ++f)
                std::memcpy(dst + ((h * d + f) * HEAD_DIM) * es, src + (f * d + h * HEAD_DIM) * es, HEAD_DIM * es);
    } else if (j == 10) {
        for (size_t c = 0; c < d; ++c)
            for (size_t f = 0; f < F; ++f) std::memcpy(dst + (f * d + c) * es, src + (c * F + f) * es, es);
    } else {
        std::memcpy(dst, src, F * d * es);
    }
}

// bf16 matrices feed ldmatrix from shared memory: 16-byte chunk c of row g is
// stored at chunk c ^ (g & 7) of that row, so the eight rows one ldmatrix
// phase reads fall in eight different bank groups.  Rows hold >= 8 chunks.
void swizzle_rows(unsigned char* w, size_t rows, size_t row_bytes) {
    const size_t chunks = row_bytes / 16;
    std::vector<unsigned char> row(row_bytes);
    for (size_t g = 0; g < rows; ++g) {
        unsigned char* r = w + g * row_bytes;
        std::memcpy(row.data(), r, row_bytes);
        for (size_t c = 0; c < chunks; ++c) std::memcpy(r + (c ^ (g & 7)) * 16, row.data() + c * 16, 16);
    }
}

int upload_weights(mtp_ctx* c, const void* blob, size_t bytes) {
    const mtp_config& cf = c->cfg;
    const unsigned char* b = static_cast<const unsigned char*>(blob);
    if (!blob || bytes < 24) return fail(MTP_ERR_WEIGHTS, "weight blob missing or shorter than its header");
    if (std::memcmp(b, "MTPWGT01", 8) != 0) return fail(MTP_ERR_WEIGHTS, "bad weight blob magic");
    uint32_t version, n_t;
    std::memcpy(&version, b + 8, 4);
    std::memcpy(&n_t, b + 12, 4);
    const std::vector<TensorSpec> specs = blob_specs(cf);
    if (version != 1) return fail(MTP_ERR_WEIGHTS, "weight blob version %u (expected 1)", version);
    if (n_t != specs.size()) return fail(MTP_ERR_WEIGHTS, "blob has %u tensors, config needs %zu", n_t, specs.size());
    if (bytes < 24 + 16 * (size_t)n_t) return fail(MTP_ERR_WEIGHTS, "blob shorter than its tensor table");
    std::vector<size_t> dev_off(n_t);
    size_t total = 0;
    for (uint32_t i = 0; i < n_t; ++i) {
        uint64_t off, nb;
        std::memcpy(&off, b + 24 + 16 * i, 8);
        std::memcpy(&nb, b + 24 + 16 * i + 8, 8);
        const size_t want = specs[i].numel * (specs[i].matrix ? c->wbytes : 4);
        if (nb != want) return fail(MTP_ERR_WEIGHTS, "tensor %u has %llu bytes, config needs %zu", i,
                                    (unsigned long long)nb, want);
        if (off % 256 || off + nb > bytes) return fail(MTP_ERR_WEIGHTS, "tensor %u offset %llu invalid", i,
                                                        (unsigned long long)off);
        dev_off[i] = total;
        total += align256(nb);
    }
    unsigned char* dw = nullptr;
    MTP_TRY(c->alloc(&dw, total));
    c->d_weights = dw;
    std::vector<unsigned char> tmp;
    for (uint32_t i = 0; i < n_t; ++i) {
        uint64_t off, nb;
        std::memcpy(&off, b + 24 + 16 * i, 8);
        std::memcpy(&nb, b + 24 + 16 * i + 8, 8);
        const unsigned char* src = b + off;
        const int j = i >= 2 && i < 2 + 12u * cf.layers ? (int)((i - 2) % 12) : -1;
        if (j == 2 || j == 3 || j == 4 || j == 10 || (j == 8 && c->wbytes == 2)) {  // fused-kernel layouts
            tmp.resize(nb);
            relayout(cf, j, j == 3 ? 4 : c->wbytes, src, tmp.data());
            if (c->wbytes == 2 && j != 3) {
                const size_t row_elems = j == 4 ? HEAD_DIM : cf.d_model;
                swizzle_rows(tmp.data(), nb / (row_elems * 2), row_elems * 2);
            }
            src = tmp.data();
        }
        if (j == 10 && c->wbytes == 2) {  // W2 [d][F] as given, for the batched path's tensor-core GEMM
            if (!c->d_w2p) MTP_TRY(c->alloc(&c->d_w2p, (size_t)cf.layers * cf.d_model * cf.d_ffn));
            const int l = (int)((i - 2) / 12);
            CUDA_TRY(cudaMemcpy(c->d_w2p + (size_t)l * cf.d_model * cf.d_ffn, b + off, nb, cudaMemcpyHostToDevice));
        }
        CUDA_TRY(cudaMemcpy(dw + dev_off[i], src, nb, cudaMemcpyHostToDevice));
    }
    size_t i = 0;
    auto nxt = [&]() { return static_cast<const void*>(dw + dev_off[i++]); };
    c->tok_phone = nxt();
    c->tok_codec = nxt();
    c->layers.resize(cf.layers);
    for (int l = 0; l < cf.layers; ++l) {
        Layer& L = c->layers[l];
        L.ln1_g = (const float*)nxt(); L.ln1_b = (const float*)nxt();
        L.wqkv = nxt(); L.bqkv = (const float*)nxt();
        L.wo = nxt(); L.bo = (const float*)nxt();
        L.ln2_g = (const float*)nxt(); L.ln2_b = (const float*)nxt();
        L.w1 = nxt(); L.b1 = (const float*)nxt();
        L.w2 = nxt(); L.b2 = (const float*)nxt();
    }
    c->lnf_g = (const float*)nxt();
    c->lnf_b = (const float*)nxt();
    c->w_heads = nxt();
    c->b_heads = (const float*)nxt();
    c->log_q = (const float*)nxt();
    return MTP_OK;
}

void release_slot_pages(mtp_ctx* c, int slot) {
    for (int p : c->slot_pages[slot]) c->free_pages.push_back(p);
    c->slot_pages[slot].clear();
    std::fill(c->h_block_table.begin() + (size_t)slot * c->pages_per_seq,
              c->h_block_table.begin() + (size_t)(slot + 1) * c->pages_per_seq, -1);
}

int check_ctx(mtp_ctx* c) {
    if (!c) return fail(MTP_ERR_INVALID, "null context");
    return MTP_OK;
}

int check_slot(mtp_ctx* c, int slot) {
    MTP_TRY(check_ctx(c));
    if (slot < 0 || slot >= c->cfg.max_batch) return fail(MTP_ERR_INVALID, "slot %d out of range", slot);
    return MTP_OK;
}

int check_nk(mtp_ctx* c, int n, int k) {
    if (n < 1 || n > c->cfg.n_heads_max) return fail(MTP_ERR_INVALID, "n_heads %d: need 1..%d", n, c->cfg.n_heads_max);
    if (k < 1 || k > c->cfg.top_k_max) return fail(MTP_ERR_INVALID, "top_k %d: need 1..%d", k, c->cfg.top_k_max);
    return MTP_OK;
}

void destroy(mtp_ctx* c) {
    if (!c) return;
    for (auto& g : c->graphs) cudaGraphExecDestroy(g.second);
    for (void* p : c->allocs) cudaFree(p);
    if (c->cap_stream) cudaStreamDestroy(c->cap_stream);
    delete c;
}

}  // namespace

int mtp::attention_standalone_plan(const mtp_attention_args* a, bool check_pointers, AttnStandalonePlan* p) {
    if (!a || a->rows < 1 || a->rows_per_group < 1 || a->rows_per_group > MAX_ROWS || a->n_heads < 1 ||
        (a->page_size != 16 && a->page_size != 32 && a->page_size != 64 && a->page_size != 128) || a->layers < 1 ||
        a->layer < 0 || a->layer >= a->layers || a->bt_stride < 1 || a->max_keys < 1)
        return fail(MTP_ERR_INVALID, "attention: invalid sizes");
    if (check_pointers && (!a->q || !a->kv_pool || !a->block_table || !a->row_seq || !a->row_pos || !a->out))
        return fail(MTP_ERR_INVALID, "attention: null pointer");
    int dev = 0, sms = 0;
    CUDA_TRY(cudaGetDevice(&dev));
    CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    p->groups = (a->rows + a->rows_per_group - 1) / a->rows_per_group;
    p->splits = attn_splits_for(p->groups, a->n_heads, a->page_size, a->max_keys, sms);
    p->part_bytes = align256(attn_workspace_floats(p->groups, a->n_heads, p->splits, a->rows_per_group) * sizeof(float));
    p->count_bytes = align256((size_t)p->groups * a->n_heads * sizeof(int));
    p->need = p->part_bytes + p->count_bytes;
    return MTP_OK;
}

int mtp::attention_standalone_launch(const mtp_attention_args* a, const AttnStandalonePlan& p, void* workspace,
                                     cudaStream_t stream) {
    AttnArgs at;
    std::memset(&at, 0, sizeof(at));
    const int d = a->n_heads * HEAD_DIM;
    at.q = a->q; at.ldq = d;
    at.kv_pool = reinterpret_cast<const __nv_bfloat16*>(a->kv_pool);
    at.page_elems = (long long)a->layers * 2 * a->n_heads * a->page_size * HEAD_DIM;
    at.layer_off = (long long)a->layer * 2 * a->n_heads * a->page_size * HEAD_DIM;
    at.block_table = a->block_table; at.bt_stride = a->bt_stride;
    at.row_seq = a->row_seq; at.row_pos = a->row_pos;
    at.out = a->out; at.ldo = d;
    at.ws_part = static_cast<float*>(workspace);
    at.ws_count = reinterpret_cast<int*>(static_cast<char*>(workspace) + p.part_bytes);
    at.rows_per_group = a->rows_per_group; at.n_heads = a->n_heads; at.page_size = a->page_size;
    at.n_splits = p.splits; at.plan = PLAN_ROWS;
    at.err = nullptr;
    CUDA_TRY(launch_attention(at, p.groups, stream, false));
    return MTP_OK;
}

// ================================================================ C ABI ====

extern "C" {

MTP_API const char* mtp_last_error(void) { return g_err.c_str(); }

MTP_API int mtp_create(const mtp_config* config, const void* weights_blob, size_t blob_bytes, void* cuda_stream,
                       mtp_ctx** out) {
    g_err.clear();
    if (!config || !out) return fail(MTP_ERR_INVALID, "null config or output handle");
    *out = nullptr;
    MTP_TRY(validate_config(*config));
    mtp_ctx* c = new mtp_ctx();
    c->cfg = *config;
    c->stream = static_cast<cudaStream_t>(cuda_stream);
    c->wbytes = config->weight_dtype == MTP_BF16 ? 2 : 4;
    auto bail = [&](int r) {
        destroy(c);
        return r;
    };
    int r;
    if (cudaGetDevice(&c->device) != cudaSuccess ||
        cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device) != cudaSuccess) {
        cudaGetLastError();
        return bail(fail(MTP_ERR_CUDA, "no usable CUDA device"));
    }
    if (cudaStreamCreateWithFlags(&c->cap_stream, cudaStreamNonBlocking) != cudaSuccess)
        return bail(fail(MTP_ERR_CUDA, "cudaStreamCreateWithFlags failed"));
    const mtp_config& cf = c->cfg;
    if ((r = upload_weights(c, weights_blob, blob_bytes)) != MTP_OK) return bail(r);

    const int d = cf.d_model, H = cf.n_attn_heads, P = cf.page_size, B = cf.max_batch;
    const int V = cf.codec_vocab, nm = cf.n_heads_max;
    c->pages_per_seq = (cf.max_ctx + P - 1) / P;
    c->n_pages = cf.n_pages > 0 ? cf.n_pages : B * c->pages_per_seq;
    c->page_elems = (long long)cf.layers * 2 * H * P * HEAD_DIM;
    // the fused block kernels' shared memory; MLP clusters that fit one wave
    {
        int clusters = 0;
        if (mlp_max_clusters(d, c->num_sms, c->wbytes, cf.d_ffn, &clusters) != cudaSuccess || clusters < 1) {
            cudaGetLastError();
            clusters = std::max(1, c->num_sms / MLP_CLUSTER / 2);
        }
        c->mlp_clusters = std::min(clusters, std::max(1, c->num_sms / MLP_CLUSTER));
        int rpc;
        mlp_grid(c, &rpc);
        const size_t sa = attn_block_smem_bytes(d, c->wbytes, P), sb = mlp_smem_bytes(d, rpc, c->wbytes);
        int hrpc;
        gemv_grid(c, nm * V, d, MAX_ROWS, &hrpc);
        const size_t sh = gemv_smem_bytes(hrpc, d, c->wbytes, MAX_ROWS);
        if (sa > 200 * 1024 || sb > 200 * 1024 || sh > 200 * 1024)
            return bail(fail(MTP_ERR_INVALID, "model too wide for the shared-memory plan (%zu, %zu, %zu bytes)", sa,
                             sb, sh));
    }
    const int lb = std::max(B, MAX_ROWS);
    const int row_cap = (B * nm + PREFILL_ROWS + 7) / 8 * 8;  // rows of one pass (slots' rows + the prefill lane)
    if ((r = c->alloc(&c->d_pe, (size_t)cf.max_ctx * d)) ||
        (r = c->alloc(&c->d_kv, (size_t)c->n_pages * c->page_elems)) ||
        (r = c->alloc(&c->d_block_table, (size_t)B * c->pages_per_seq)) ||
        (r = c->alloc(&c->d_len, B)) || (r = c->alloc(&c->d_npend, B)) ||
        (r = c->alloc(&c->d_pending, (size_t)B * nm)) || (r = c->alloc(&c->d_remaining, B)) ||
        (r = c->alloc(&c->d_done, B)) || (r = c->alloc(&c->d_active, B)) || (r = c->alloc(&c->d_gen_count, B)) ||
        (r = c->alloc(&c->d_gen_tokens, (size_t)B * cf.max_ctx)) ||
        (r = c->alloc(&c->d_prompt, (size_t)B * cf.max_ctx)) || (r = c->alloc(&c->d_h_last, (size_t)lb * d)) ||
        (r = c->alloc(&c->d_xb, (size_t)3 * MAX_ROWS * d)) ||
        (r = c->alloc(&c->d_logits, (size_t)lb * nm * V)) || (r = c->alloc(&c->d_lse, (size_t)lb * nm)) ||
        (r = c->alloc(&c->d_cand_logp, (size_t)lb * nm * MAX_TOPK)) ||
        (r = c->alloc(&c->d_cand_ids, (size_t)lb * nm * MAX_TOPK)) || (r = c->alloc(&c->d_path, (size_t)lb * nm)) ||
        (r = c->alloc(&c->d_out_tokens, (size_t)B * nm)) || (r = c->alloc(&c->d_out_accepted, B)) ||
        (r = c->alloc(&c->d_row_seq, row_cap)) || (r = c->alloc(&c->d_row_pos, row_cap)) ||
        (r = c->alloc(&c->d_row_last, row_cap)) || (r = c->alloc(&c->d_err, 1)) || (r = c->alloc(&c->d_kept, B)) ||
        (r = c->alloc(&c->d_prompt_left, B)) || (r = c->alloc(&c->d_prompt_nph, B)) ||
        (r = c->alloc(&c->d_lane_take, B)) ||
        (r = setup_batched(c)) || (r = setup_step_kernel(c)))
        return bail(r);
    c->h_block_table.assign((size_t)B * c->pages_per_seq, -1);
    c->h_prompt_left.assign(B, 0);
    if (cudaMemcpy(c->d_block_table, c->h_block_table.data(), c->h_block_table.size() * sizeof(int),
                   cudaMemcpyHostToDevice) != cudaSuccess)
        return bail(fail(MTP_ERR_CUDA, "block table upload failed"));
    c->slot_pages.assign(B, {});
    for (int p = c->n_pages - 1; p >= 0; --p) c->free_pages.push_back(p);
    if (launch_pe_table(c->d_pe, cf.max_ctx, d, c->stream) != cudaSuccess ||
        cudaStreamSynchronize(c->stream) != cudaSuccess)
        return bail(fail(MTP_ERR_CUDA, "position table: %s", cudaGetErrorString(cudaGetLastError())));
    *out = c;
    return MTP_OK;
}

MTP_API void mtp_destroy(mtp_ctx* ctx) {
    if (!ctx) return;
    cudaStreamSynchronize(ctx->stream);
    destroy(ctx);
}

MTP_API int mtp_set_option(mtp_ctx* c, int option, int value) {
    g_err.clear();
    MTP_TRY(check_ctx(c));
    bool changed = false;
    if (option == MTP_OPT_GRAPHS) {
        c->use_graphs = value != 0;
    } else if (option == MTP_OPT_PDL) {
        changed = c->use_pdl != (value != 0);
        c->use_pdl = value != 0;
    } else if (option == MTP_OPT_L2_PREFETCH) {
        changed = c->use_l2_prefetch != (value != 0);
        c->use_l2_prefetch = value != 0;
    } else if (option == MTP_OPT_GEMM_SPLITS) {
        if (value < 1 || value > 64 || (value & (value - 1)))
            return fail(MTP_ERR_INVALID, "GEMM splits %d: need a power of two in 1..64", value);
        changed = c->gemm_max_splits != value;
        c->gemm_max_splits = value;
    } else if (option == MTP_OPT_LATTICE) {
        if (value != 0 && value != 1) return fail(MTP_ERR_INVALID, "lattice %d: need 0 or 1", value);
        changed = c->lattice != value;
        c->lattice = value;
    } else if (option == MTP_OPT_SAMPLING) {
        if (value != 0 && value != 1) return fail(MTP_ERR_INVALID, "sampling %d: need 0 or 1", value);
        changed = c->sampling != value;
        c->sampling = value;
    } else if (option == MTP_OPT_SEED) {
        changed = c->sample_seed != (uint32_t)value;
        c->sample_seed = (uint32_t)value;
    } else if (option == MTP_OPT_PERSISTENT) {
        changed = c->use_persistent != (value != 0);
        c->use_persistent = value != 0;
    } else if (option == MTP_OPT_PREFILL_TC) {
        c->use_attn_tc = value != 0;  // prefill passes are not captured
    } else if (option == MTP_OPT_GEMM_CLUSTER) {
        changed = c->gemm_cluster != (value != 0);
        c->gemm_cluster = value != 0;
    } else if (option == MTP_OPT_HEADS_FUSED) {
        if (value < 0 || value > 2) return fail(MTP_ERR_INVALID, "heads option %d: 0, 1 or 2", value);
        changed = c->use_heads_tc != value;
        c->use_heads_tc = value;
    } else if (option == MTP_OPT_BATCHED) {
        changed = c->use_batched != (value != 0);
        c->use_batched = value != 0;
    } else if (option == MTP_OPT_MLP_CLUSTERS) {
        if (value < 1 || value > std::max(1, 2 * c->num_sms / MLP_CLUSTER))
            return fail(MTP_ERR_INVALID, "MLP clusters %d out of range", value);
        int rpc;
        const int keep = c->mlp_clusters;
        c->mlp_clusters = value;
        mlp_grid(c, &rpc);
        if (mlp_smem_bytes(c->cfg.d_model, rpc, c->wbytes) > 200 * 1024) {
            c->mlp_clusters = keep;
            return fail(MTP_ERR_INVALID, "%d MLP clusters need too much shared memory", value);
        }
        changed = keep != value;
    } else {
        return fail(MTP_ERR_INVALID, "unknown option %d", option);
    }
    if (changed) {  // captured steps bake these in
        for (auto& g : c->graphs) cudaGraphExecDestroy(g.second);
        c->graphs.clear();
        c->graph_kinds.clear();
    }
    return MTP_OK;
}

MTP_API int mtp_get_option(mtp_ctx* c, int option, int32_t* value) {
    g_err.clear();
    MTP_TRY(check_ctx(c));
    if (!value) return fail(MTP_ERR_INVALID, "null output");
    switch (option) {
        case MTP_OPT_GRAPHS: *value = c->use_graphs; break;
        case MTP_OPT_PDL: *value = c->use_pdl; break;
        case MTP_OPT_L2_PREFETCH: *value = c->use_l2_prefetch; break;
        case MTP_OPT_MLP_CLUSTERS: *value = c->mlp_clusters; break;
        case MTP_OPT_BATCHED: *value = c->use_batched && c->batched_ok; break;
        case MTP_OPT_GEMM_SPLITS: *value = c->gemm_max_splits; break;
        case MTP_OPT_LATTICE: *value = c->lattice; break;
        case MTP_OPT_SAMPLING: *value = c->sampling; break;
        case MTP_OPT_SEED: *value = (int32_t)c->sample_seed; break;
        case MTP_OPT_PERSISTENT: *value = c->use_persistent && c->sk_ok; break;
        case MTP_OPT_PREFILL_TC: *value = c->use_attn_tc; break;
        case MTP_OPT_HEADS_FUSED: *value = c->heads_tc_ok && c->batched_ok ? c->use_heads_tc : 0; break;
        case MTP_OPT_GEMM_CLUSTER: *value = c->gemm_cluster; break;
        default: return fail(MTP_ERR_INVALID, "unknown option %d", option);
    }
    return MTP_OK;
}

// Validation, page reservation and the prompt's copy to the device, shared by
// mtp_prefill and mtp_admit; *T_out = prompt length.
static int take_prompt(mtp_ctx* c, int slot, const int32_t* phonemes, int n_ph, const int32_t* acoustic, int n_ac,
                int max_new_tokens, long long* T_out) {
    MTP_TRY(check_slot(c, slot));
    const mtp_config& cf = c->cfg;
    if (n_ph < 0 || n_ac < 0 || n_ph + n_ac < 1) return fail(MTP_ERR_INVALID, "empty prompt");
    if ((n_ph && !phonemes) || (n_ac && !acoustic)) return fail(MTP_ERR_INVALID, "null prompt pointer");
    if (max_new_tokens < 1) return fail(MTP_ERR_INVALID, "max_new_tokens %d", max_new_tokens);
    const long long T = (long long)n_ph + n_ac;
    const long long need = T + max_new_tokens + cf.n_heads_max;
    if (need > cf.max_ctx)
        return fail(MTP_ERR_INVALID, "prompt %lld + max_new %d + n_heads_max %d exceeds max_ctx %d", T,
                    max_new_tokens, cf.n_heads_max, cf.max_ctx);
    // host-side id checks (device prompts are checked by the embedding kernel)
    const bool ph_dev = is_device_ptr(phonemes), ac_dev = is_device_ptr(acoustic);
    if (!ph_dev)
        for (int i = 0; i < n_ph; ++i)
            if (phonemes[i] < 0 || phonemes[i] >= cf.phone_vocab)
                return fail(MTP_ERR_INVALID, "phoneme id %d at %d out of range", phonemes[i], i);
    if (!ac_dev)
        for (int i = 0; i < n_ac; ++i)
            if (acoustic[i] < 0 || acoustic[i] >= cf.codec_vocab)
                return fail(MTP_ERR_INVALID, "acoustic id %d at %d out of range", acoustic[i], i);
    release_slot_pages(c, slot);
    const int P = cf.page_size;
    const int n_pages = (int)((need + P - 1) / P);
    if ((int)c->free_pages.size() < n_pages)
        return fail(MTP_ERR_NO_PAGES, "slot %d needs %d pages, %zu free", slot, n_pages, c->free_pages.size());
    for (int i = 0; i < n_pages; ++i) {
        const int p = c->free_pages.back();
        c->free_pages.pop_back();
        c->slot_pages[slot].push_back(p);
        c->h_block_table[(size_t)slot * c->pages_per_seq + i] = p;
    }
    cudaStream_t s = c->stream;
    CUDA_TRY(cudaMemcpyAsync(c->d_block_table + (size_t)slot * c->pages_per_seq,
                             c->h_block_table.data() + (size_t)slot * c->pages_per_seq,
                             c->pages_per_seq * sizeof(int), cudaMemcpyHostToDevice, s));
    int* prompt = c->d_prompt + (size_t)slot * cf.max_ctx;
    if (n_ph) CUDA_TRY(cudaMemcpyAsync(prompt, phonemes, n_ph * sizeof(int), cudaMemcpyDefault, s));
    if (n_ac) CUDA_TRY(cudaMemcpyAsync(prompt + n_ph, acoustic, n_ac * sizeof(int), cudaMemcpyDefault, s));
    *T_out = T;
    return MTP_OK;
}

MTP_API int mtp_prefill(mtp_ctx* c, int slot, const int32_t* phonemes, int n_ph, const int32_t* acoustic, int n_ac,
                        int max_new_tokens) {
    g_err.clear();
    long long T = 0;
    MTP_TRY(take_prompt(c, slot, phonemes, n_ph, acoustic, n_ac, max_new_tokens, &T));
    const mtp_config& cf = c->cfg;
    cudaStream_t s = c->stream;
    c->h_prompt_left[slot] = 0;
    MTP_TRY(slot_set(c, slot, 0, 0, max_new_tokens, 0, 1, 0, 0, n_ph));
    Prof* prof = nullptr;
    float* final_x = nullptr;
    if (c->use_batched && c->batched_ok) {  // chunks of PREFILL_ROWS positions through the batched path
        for (int p0 = 0; p0 < T; p0 += PREFILL_ROWS) {
            const int m = (int)std::min<long long>(PREFILL_ROWS, T - p0);
            const int rows = (m + 7) / 8 * 8;
            EmbedArgs e = embed_base(c);
            e.mode = 1; e.rows = m; e.slot = slot; e.p0 = p0; e.n_ph = n_ph; e.total = (int)T;
            e.x = c->d_bx; e.zero_buf = nullptr;
            LAUNCH(MTP_K_EMBED, launch_embed(e, s, false));
            MTP_TRY(run_layers_batched(c, rows, 8, rows / 8, PLAN_ROWS, s, c->use_pdl, prof, p0 + m));
            LAUNCH(MTP_K_SAVE, launch_save_last(c->d_bx, c->d_row_seq, c->d_row_last, c->d_h_last, cf.d_model, rows,
                                                nullptr, s, c->use_pdl));
        }
        MTP_TRY(slot_set(c, slot, (int)T, -1, -1, -1, -1, -1));
        return MTP_OK;
    }
    for (int p0 = 0; p0 < T; p0 += MAX_ROWS) {
        const int m = (int)std::min<long long>(MAX_ROWS, T - p0);
        EmbedArgs e = embed_base(c);
        e.mode = 1; e.rows = m; e.slot = slot; e.p0 = p0; e.n_ph = n_ph; e.total = (int)T;
        LAUNCH(MTP_K_EMBED, launch_embed(e, s, false));
        MTP_TRY(run_layers(c, m, 1, m, PLAN_VALUE, 0, slot, p0, m, s, c->use_pdl, prof, &final_x));
    }
    LAUNCH(MTP_K_SAVE, launch_save_last(final_x, c->d_row_seq, c->d_row_last, c->d_h_last, cf.d_model, MAX_ROWS, nullptr, s,
                                        c->use_pdl));
    MTP_TRY(slot_set(c, slot, (int)T, -1, -1, -1, -1, -1));
    // pageable host prompts: copies above are complete when the call returns
    return MTP_OK;
}

MTP_API int mtp_release(mtp_ctx* c, int slot) {
    g_err.clear();
    MTP_TRY(check_slot(c, slot));
    release_slot_pages(c, slot);
    CUDA_TRY(cudaMemcpyAsync(c->d_block_table + (size_t)slot * c->pages_per_seq,
                             c->h_block_table.data() + (size_t)slot * c->pages_per_seq,
                             c->pages_per_seq * sizeof(int), cudaMemcpyHostToDevice, c->stream));
    MTP_TRY(slot_set(c, slot, 0, 0, 0, 0, 0, 0, 0));
    c->h_prompt_left[slot] = 0;
    CUDA_TRY(cudaStreamSynchronize(c->stream));
    return MTP_OK;
}

// The prefill lane can serve admitted prompts: batched path, ACCEPT_ALL.
static bool lane_usable(const mtp_ctx* c) {
    return c->use_batched && c->batched_ok && c->cfg.accept_policy == MTP_ACCEPT_ALL;
}

MTP_API int mtp_admit(mtp_ctx* c, int slot, const int32_t* phonemes, int n_ph, const int32_t* acoustic, int n_ac,
                      int max_new_tokens) {
    g_err.clear();
    MTP_TRY(check_ctx(c));
    if (!lane_usable(c)) return mtp_prefill(c, slot, phonemes, n_ph, acoustic, n_ac, max_new_tokens);
    long long T = 0;
    MTP_TRY(take_prompt(c, slot, phonemes, n_ph, acoustic, n_ac, max_new_tokens, &T));
    MTP_TRY(slot_set(c, slot, 0, 0, max_new_tokens, 0, 1, 0, (int)T, n_ph));
    c->h_prompt_left[slot] = (int)T;
    return MTP_OK;
}

MTP_API int mtp_prefill_pending(mtp_ctx* c) {
    g_err.clear();
    MTP_TRY(check_ctx(c));
    if (!lane_pending(c)) return 0;
    if (!lane_usable(c)) return fail(MTP_ERR_INVALID, "admitted prompts need the batched path");
    const mtp_config& cf = c->cfg;
    cudaStream_t s = c->stream;
    const int P = c->bm_max / 8 * 8;  // prompt rows per pass, in attention groups of 8 positions
    int passes = 0;
    while (lane_pending(c)) {
        MTP_TRY(enqueue_lane_plan(c, 0, P, 8, s, c->use_pdl, nullptr));
        MTP_TRY(run_layers_batched(c, P, 8, P / 8, PLAN_ROWS, s, c->use_pdl, nullptr, cf.max_ctx));
        Prof* prof = nullptr;
        LAUNCH(MTP_K_SAVE, launch_save_last(c->d_bx, c->d_row_seq, c->d_row_last, c->d_h_last, cf.d_model, P, nullptr, s,
                                            c->use_pdl));
        lane_mirror(c, P, 8);
        ++passes;
    }
    MTP_TRY(check_device_error(c));
    return passes;
}

MTP_API int mtp_decode_step(mtp_ctx* c, int n, int k, int32_t* out_tokens, int32_t* out_accepted,
                            int32_t* out_done) {
    g_err.clear();
    MTP_TRY(check_ctx(c));
    MTP_TRY(check_nk(c, n, k));
    const bool lane = lane_pending(c);
    if (lane && !lane_usable(c)) return fail(MTP_ERR_INVALID, "admitted prompts need the batched path");
    MTP_TRY(run_step(c, n, k, lane));
    if (lane) lane_mirror(c, lane_rows(n), n);
    const int B = c->cfg.max_batch, nm = c->cfg.n_heads_max;
    if (out_tokens)
        CUDA_TRY(cudaMemcpy2DAsync(out_tokens, n * sizeof(int), c->d_out_tokens, nm * sizeof(int), n * sizeof(int), B,
                                   cudaMemcpyDefault, c->stream));
    MTP_TRY(copy_out(out_accepted, c->d_out_accepted, B * sizeof(int), c->stream));
    MTP_TRY(copy_out(out_done, c->d_done, B * sizeof(int), c->stream));
    const bool host_io = (out_tokens && !is_device_ptr(out_tokens)) || (out_accepted && !is_device_ptr(out_accepted)) ||
                         (out_done && !is_device_ptr(out_done));
    if (host_io) MTP_TRY(check_device_error(c));
    return MTP_OK;
}

MTP_API int mtp_generate(mtp_ctx* c, int n, int k, int32_t* out_tokens, int out_stride, int32_t* out_lens) {
    g_err.clear();
    MTP_TRY(check_ctx(c));
    MTP_TRY(check_nk(c, n, k));
    if (out_tokens && out_stride < 1) return fail(MTP_ERR_INVALID, "out_stride %d", out_stride);
    // Rounds of steps without host synchronisation: a step emits at most n tokens,
    // so ceil(remaining / n) more steps are needed at least; ACCEPT_ALL (n tokens per
    // step until EOS or the budget) finishes in one round, VERIFY_GREEDY (1..n) in a few.
    std::vector<int> rem, done, active;
    int steps = 0;
    // admitted prompts first: steps with a prefill lane (the other slots decode meanwhile)
    if (lane_pending(c) && !lane_usable(c)) return fail(MTP_ERR_INVALID, "admitted prompts need the batched path");
    for (; lane_pending(c); ++steps) {
        MTP_TRY(run_step(c, n, k, true));
        lane_mirror(c, lane_rows(n), n);
    }
    for (;;) {
        MTP_TRY(read_slot_ints(c, c->d_remaining, rem));
        MTP_TRY(read_slot_ints(c, c->d_done, done));
        MTP_TRY(read_slot_ints(c, c->d_active, active));
        int round = 0;
        for (int b = 0; b < c->cfg.max_batch; ++b)
            if (active[b] && !done[b]) round = std::max(round, (rem[b] + n - 1) / n);
        if (round == 0) break;
        MTP_TRY(run_steps(c, n, k, round));
        steps += round;
        MTP_TRY(check_device_error(c));
    }
    const int B = c->cfg.max_batch, gs = c->cfg.max_ctx;
    if (out_tokens) {
        const int w = std::min(out_stride, gs);
        CUDA_TRY(cudaMemcpy2DAsync(out_tokens, out_stride * sizeof(int), c->d_gen_tokens, gs * sizeof(int),
                                   w * sizeof(int), B, cudaMemcpyDefault, c->stream));
    }
    MTP_TRY(copy_out(out_lens, c->d_gen_count, B * sizeof(int), c->stream));
    CUDA_TRY(cudaStreamSynchronize(c->stream));
    return steps;
}

MTP_API int mtp_rollback(mtp_ctx* c, int slot, int n_tokens) {
    g_err.clear();
    MTP_TRY(check_slot(c, slot));
    std::vector<int> len;
    MTP_TRY(read_slot_ints(c, c->d_len, len));
    if (n_tokens < 0 || n_tokens > len[slot])
        return fail(MTP_ERR_INVALID, "cannot roll back %d of %d cached tokens", n_tokens, len[slot]);
    MTP_TRY(slot_set(c, slot, len[slot] - n_tokens, -1, -1, -1, -1, -1));
    CUDA_TRY(cudaStreamSynchronize(c->stream));
    return MTP_OK;
}

MTP_API int mtp_set_teacher_tokens(mtp_ctx* c, int slot, const int32_t* tokens, int n) {
    g_err.clear();
    MTP_TRY(check_slot(c, slot));
    if (!tokens || n < 1 || n > c->cfg.n_heads_max)
        return fail(MTP_ERR_INVALID, "teacher tokens: need 1..%d host ids", c->cfg.n_heads_max);
    for (int i = 0; i < n; ++i)
        if (tokens[i] < 0 || tokens[i] >= c->cfg.codec_vocab)
            return fail(MTP_ERR_INVALID, "teacher token %d out of range", tokens[i]);
    CUDA_TRY(cudaMemcpyAsync(c->d_pending + (size_t)slot * c->cfg.n_heads_max, tokens, n * sizeof(int),
                             cudaMemcpyHostToDevice, c->stream));
    MTP_TRY(slot_set(c, slot, -1, n, -1, -1, -1, -1));
    CUDA_TRY(cudaStreamSynchronize(c->stream));
    return MTP_OK;
}

MTP_API int mtp_seq_state(mtp_ctx* c, int slot, int32_t* out6) {
    g_err.clear();
    MTP_TRY(check_slot(c, slot));
    if (!out6) return fail(MTP_ERR_INVALID, "null output");
    const int* src[6] = {c->d_len, c->d_npend, c->d_remaining, c->d_done, c->d_active, c->d_gen_count};
    for (int i = 0; i < 6; ++i)
        CUDA_TRY(cudaMemcpyAsync(out6 + i, src[i] + slot, sizeof(int), cudaMemcpyDeviceToHost, c->stream));
    CUDA_TRY(cudaStreamSynchronize(c->stream));
    return MTP_OK;
}

MTP_API int mtp_debug_logits(mtp_ctx* c, float* out_logits, float* out_lse) {
    g_err.clear();
    MTP_TRY(check_ctx(c));
    if (c->last_n == 0) return fail(MTP_ERR_INVALID, "no decode step has run");
    const size_t B = c->cfg.max_batch, n = c->last_n, V = c->cfg.codec_vocab;
    MTP_TRY(copy_out(out_logits, c->d_logits, B * n * V * sizeof(float), c->stream));
    MTP_TRY(copy_out(out_lse, c->d_lse, B * n * sizeof(float), c->stream));
    CUDA_TRY(cudaStreamSynchronize(c->stream));
    return MTP_OK;
}

MTP_API int mtp_debug_lattice(mtp_ctx* c, int32_t* out_ids, float* out_logp, int32_t* out_path) {
    g_err.clear();
    MTP_TRY(check_ctx(c));
    if (c->last_n == 0) return fail(MTP_ERR_INVALID, "no decode step has run");
    const size_t B = c->cfg.max_batch, n = c->last_n, k = c->last_k;
    MTP_TRY(copy_out(out_ids, c->d_cand_ids, B * n * k * sizeof(int), c->stream));
    MTP_TRY(copy_out(out_logp, c->d_cand_logp, B * n * k * sizeof(float), c->stream));
    MTP_TRY(copy_out(out_path, c->d_path, B * n * sizeof(int), c->stream));
    CUDA_TRY(cudaStreamSynchronize(c->stream));
    return MTP_OK;
}

MTP_API int mtp_profile_step(mtp_ctx* c, int n, int k, float* out_ms, int32_t* out_launches) {
    g_err.clear();
    MTP_TRY(check_ctx(c));
    MTP_TRY(check_nk(c, n, k));
    Prof prof;
    c->last_n = n;
    c->last_k = k;
    const int r = enqueue_step(c, n, k, c->stream, false, &prof);
    cudaError_t e = cudaStreamSynchronize(c->stream);
    for (int i = 0; i < MTP_K_COUNT; ++i) {
        if (out_ms) out_ms[i] = 0.f;
        if (out_launches) out_launches[i] = 0;
    }
    for (auto& ev : prof.ev) {
        float ms = 0.f;
        if (r == MTP_OK && e == cudaSuccess) e = cudaEventElapsedTime(&ms, ev.second.first, ev.second.second);
        if (out_ms) out_ms[ev.first] += ms;
        if (out_launches) out_launches[ev.first] += 1;
        cudaEventDestroy(ev.second.first);
        cudaEventDestroy(ev.second.second);
    }
    if (r != MTP_OK) return r;
    CUDA_TRY(e);
    return check_device_error(c);
}

MTP_API int mtp_trace_step(mtp_ctx* c, int n, int k, int64_t* out, int cap) {
    g_err.clear();
    MTP_TRY(check_ctx(c));
    MTP_TRY(check_nk(c, n, k));
    if (!out || cap < 1) return fail(MTP_ERR_INVALID, "trace: null output or capacity < 1");
    if (!c->d_trace) {
        c->trace_cap = 4096;
        MTP_TRY(c->alloc(&c->d_trace, (size_t)TRACE_WORDS * c->trace_cap));
    }
    CUDA_TRY(launch_trace_reset(c->d_trace, c->trace_cap, c->stream));
    c->tracing = true;
    const int r = run_step(c, n, k);
    c->tracing = false;
    MTP_TRY(r);
    std::vector<unsigned long long> h(TRACE_WORDS * (size_t)c->trace_cap);
    CUDA_TRY(cudaMemcpyAsync(h.data(), c->d_trace, h.size() * sizeof(unsigned long long), cudaMemcpyDeviceToHost,
                             c->stream));
    MTP_TRY(check_device_error(c));
    const int count = std::min<int>((int)c->trace_kinds.size(), cap);
    for (int i = 0; i < count; ++i) {
        out[(TRACE_WORDS + 1) * i] = c->trace_kinds[i];
        for (int j = 0; j < TRACE_WORDS; ++j) out[(TRACE_WORDS + 1) * i + 1 + j] = (int64_t)h[(size_t)TRACE_WORDS * i + j];
    }
    return count;
}

MTP_API int mtp_step_bytes(mtp_ctx* c, int n, uint64_t* out_bytes) {
    g_err.clear();
    MTP_TRY(check_ctx(c));
    if (n < 1 || n > c->cfg.n_heads_max || !out_bytes) return fail(MTP_ERR_INVALID, "bad arguments");
    const mtp_config& cf = c->cfg;
    const uint64_t d = cf.d_model, F = cf.d_ffn, V = cf.codec_vocab, wb = c->wbytes;
    uint64_t bytes = (uint64_t)cf.layers * ((3 * d * d + d * d + 2 * d * F) * wb + (3 * d + d + F + d + 4 * d) * 4);
    bytes += (uint64_t)n * V * d * wb + (uint64_t)n * V * 4 + 2 * d * 4;
    std::vector<int> len, npend, active, done;
    MTP_TRY(read_slot_ints(c, c->d_len, len));
    MTP_TRY(read_slot_ints(c, c->d_npend, npend));
    MTP_TRY(read_slot_ints(c, c->d_active, active));
    MTP_TRY(read_slot_ints(c, c->d_done, done));
    for (int b = 0; b < cf.max_batch; ++b) {
        if (!active[b] || done[b] || npend[b] == 0) continue;
        // keys and values (bf16) read over the visible context, and written for the fed rows
        bytes += (uint64_t)cf.layers * (uint64_t)(len[b] + npend[b]) * d * 2 * 2;
        bytes += (uint64_t)cf.layers * (uint64_t)npend[b] * d * 2 * 2;
    }
    *out_bytes = bytes;
    return MTP_OK;
}

MTP_API int mtp_viterbi(int batch, int n, int k, int vocab, int eos_id, const int32_t* cand_ids,
                        const float* cand_logp, const float* log_q, const int32_t* remaining, int32_t* out_path,
                        float* out_score, int32_t* out_accepted, int32_t* out_rollback, void* cuda_stream) {
    g_err.clear();
    if (batch < 0 || n < 1 || n > MAX_NHEADS || k < 1 || k > MAX_TOPK || vocab < 1 || k > vocab)
        return fail(MTP_ERR_INVALID, "viterbi: batch %d, n %d (1..%d), k %d (1..%d), vocab %d", batch, n,
                    MAX_NHEADS, k, MAX_TOPK, vocab);
    if (batch > 0 && (!cand_ids || !cand_logp || !log_q || !out_path || !out_accepted))
        return fail(MTP_ERR_INVALID, "viterbi: null pointer");
    ViterbiArgs a;
    a.batch = batch; a.n = n; a.k = k; a.vocab = vocab; a.eos_id = eos_id;
    a.cand_ids = cand_ids; a.cand_logp = cand_logp; a.log_q = log_q; a.remaining = remaining;
    a.path = out_path; a.score = out_score; a.accepted = out_accepted; a.rollback = out_rollback;
    CUDA_TRY(launch_viterbi(a, static_cast<cudaStream_t>(cuda_stream)));
    return MTP_OK;
}

namespace {
// A barrier with one expected arrival that never comes: the bounded wait runs out.
__global__ void selftest_wait_kernel(int* err) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) mbar_wait(&bar, 0, err);
}
}  // namespace

MTP_API int mtp_selftest_bounded_wait(int32_t* err_word, void* cuda_stream) {
    g_err.clear();
    if (!err_word) return fail(MTP_ERR_INVALID, "selftest: null error word");
    selftest_wait_kernel<<<1, 32, 0, static_cast<cudaStream_t>(cuda_stream)>>>(err_word);
    CUDA_TRY(cudaGetLastError());
    return MTP_OK;
}

MTP_API int mtp_selftest_grid_barrier(int32_t* err_word, void* cuda_stream) {
    g_err.clear();
    if (!err_word) return fail(MTP_ERR_INVALID, "selftest: null error word");
    CUDA_TRY(launch_selftest_grid_barrier(err_word, static_cast<cudaStream_t>(cuda_stream)));
    return MTP_OK;
}

MTP_API int mtp_heads_topk(mtp_ctx* c, int batch, const void* hidden, int hidden_dtype, int n, int k,
                           int32_t* out_ids, float* out_logp, float* out_logits, float* out_lse) {
    g_err.clear();
    MTP_TRY(check_ctx(c));
    MTP_TRY(check_nk(c, n, k));
    if (batch < 0 || (batch > 0 && (!hidden || !out_ids || !out_logp)))
        return fail(MTP_ERR_INVALID, "heads_topk: bad batch or null pointer");
    if (hidden_dtype != MTP_F32 && hidden_dtype != MTP_BF16) return fail(MTP_ERR_INVALID, "hidden dtype");
    const int d = c->cfg.d_model, V = c->cfg.codec_vocab;
    cudaStream_t s = c->stream;
    Prof* prof = nullptr;
    // more rows than one fused pass: tensor-core heads over chunks of the batched buffers' rows
    // (of the context's logits rows when the caller passes no logits / lse buffers)
    const int lrows = std::max(c->cfg.max_batch, MAX_ROWS);
    const int tc_rows = out_logits && out_lse ? c->bm_max : std::min(c->bm_max, lrows);
    // the fused heads need no logits buffer: chunks of every batched row
    const bool fused = c->use_batched && c->batched_ok && batch > MAX_ROWS && heads_fused_ok(c, k, false);
    const bool tc = !fused && c->use_batched && c->batched_ok && batch > MAX_ROWS && tc_rows > MAX_ROWS;
    const int chunk = fused ? c->bm_max : (tc ? tc_rows : MAX_ROWS);
    for (int b0 = 0; b0 < batch; b0 += chunk) {
        const int m = std::min(chunk, batch - b0);
        if (fused) {
            const size_t es = hidden_dtype == MTP_BF16 ? 2 : 4;
            CUDA_TRY(launch_convert_rows(static_cast<const char*>(hidden) + (size_t)b0 * d * es,
                                         hidden_dtype == MTP_BF16, c->d_bx, m, d, s));
            MTP_TRY(launch_heads_fused(c, c->d_bx, m, n, k, out_ids + (size_t)b0 * n * k,
                                       out_logp + (size_t)b0 * n * k, out_lse ? out_lse + (size_t)b0 * n : nullptr,
                                       out_logits ? out_logits + (size_t)b0 * n * V : nullptr, s, false, prof));
            continue;
        }
        if (tc) {
            const size_t es = hidden_dtype == MTP_BF16 ? 2 : 4;
            CUDA_TRY(launch_convert_rows(static_cast<const char*>(hidden) + (size_t)b0 * d * es,
                                         hidden_dtype == MTP_BF16, c->d_bx, m, d, s));
            float* logits = out_logits ? out_logits + (size_t)b0 * n * V : c->d_logits;
            MTP_TRY(launch_heads_batched(c, c->d_bx, m, n, logits, s, false, prof));
            SelectArgs sa = select_base(c, n, k);
            sa.logits = logits;
            sa.lse = out_lse ? out_lse + (size_t)b0 * n : c->d_lse;
            sa.cand_ids = out_ids + (size_t)b0 * n * k;
            sa.cand_logp = out_logp + (size_t)b0 * n * k;
            CUDA_TRY(launch_select(sa, m, false, s, false));
            continue;
        }
        const size_t es = hidden_dtype == MTP_BF16 ? 2 : 4;
        CUDA_TRY(launch_convert_rows(static_cast<const char*>(hidden) + (size_t)b0 * d * es,
                                     hidden_dtype == MTP_BF16, xbuf(c, 0), m, d, s));
        float* logits = out_logits ? out_logits + (size_t)b0 * n * V : c->d_logits;
        MTP_TRY(launch_heads(c, xbuf(c, 0), m, n, logits, nullptr, 0, s, false, prof));
        SelectArgs sa = select_base(c, n, k);
        sa.logits = logits;
        sa.lse = out_lse ? out_lse + (size_t)b0 * n : c->d_lse;
        sa.cand_ids = out_ids + (size_t)b0 * n * k;
        sa.cand_logp = out_logp + (size_t)b0 * n * k;
        CUDA_TRY(launch_select(sa, m, false, s, false));
    }
    return MTP_OK;
}

MTP_API size_t mtp_attention_workspace_bytes(const mtp_attention_args* a) {
    AttnStandalonePlan p;
    const std::string keep = g_err;  // a size query leaves the last error alone
    const int r = attention_standalone_plan(a, false, &p);
    g_err = keep;
    return r == MTP_OK ? p.need : 0;
}

MTP_API int mtp_attention(const mtp_attention_args* a, void* workspace, size_t workspace_bytes, void* cuda_stream) {
    g_err.clear();
    AttnStandalonePlan p;
    MTP_TRY(attention_standalone_plan(a, true, &p));
    if (!workspace) return fail(MTP_ERR_INVALID, "attention: null workspace");
    if (workspace_bytes < p.need)
        return fail(MTP_ERR_INVALID, "attention: workspace %zu bytes, need %zu", workspace_bytes, p.need);
    return attention_standalone_launch(a, p, workspace, static_cast<cudaStream_t>(cuda_stream));
}

}  // extern "C"

namespace {
// Tiles, splits and workspace of mtp_attention_tc (sizes as mtp_attention; rows_per_group unused).
int attention_tc_plan(const mtp_attention_args* a, bool check_pointers, AttnStandalonePlan* p) {
    if (!a || a->rows < 1 || a->n_heads < 1 ||
        (a->page_size != 16 && a->page_size != 32 && a->page_size != 64 && a->page_size != 128) || a->layers < 1 ||
        a->layer < 0 || a->layer >= a->layers || a->bt_stride < 1 || a->max_keys < 1)
        return fail(MTP_ERR_INVALID, "attention_tc: invalid sizes");
    if (check_pointers && (!a->q || !a->kv_pool || !a->block_table || !a->row_seq || !a->row_pos || !a->out))
        return fail(MTP_ERR_INVALID, "attention_tc: null pointer");
    if (check_pointers && (reinterpret_cast<uintptr_t>(a->q) & 15))
        return fail(MTP_ERR_INVALID, "attention_tc: q must be 16-byte aligned");
    int dev = 0, sms = 0;
    CUDA_TRY(cudaGetDevice(&dev));
    CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    p->groups = attn_tc_tiles(a->rows);
    p->splits = attn_tc_splits_for(p->groups, a->n_heads, a->max_keys, sms);
    p->part_bytes = align256(attn_tc_workspace_floats(p->groups, a->n_heads, p->splits) * sizeof(float));
    p->count_bytes = align256((size_t)p->groups * a->n_heads * sizeof(int));
    p->need = p->part_bytes + p->count_bytes;
    return MTP_OK;
}
}  // namespace

extern "C" {

MTP_API size_t mtp_attention_tc_workspace_bytes(const mtp_attention_args* a) {
    AttnStandalonePlan p;
    const std::string keep = g_err;  // a size query leaves the last error alone
    const int r = attention_tc_plan(a, false, &p);
    g_err = keep;
    return r == MTP_OK ? p.need : 0;
}

MTP_API int mtp_attention_tc(const mtp_attention_args* a, void* workspace, size_t workspace_bytes,
                             void* cuda_stream) {
    g_err.clear();
    AttnStandalonePlan p;
    MTP_TRY(attention_tc_plan(a, true, &p));
    if (!workspace) return fail(MTP_ERR_INVALID, "attention_tc: null workspace");
    if (workspace_bytes < p.need)
        return fail(MTP_ERR_INVALID, "attention_tc: workspace %zu bytes, need %zu", workspace_bytes, p.need);
    AttnArgs at;
    std::memset(&at, 0, sizeof(at));
    const int d = a->n_heads * HEAD_DIM;
    at.q = a->q; at.ldq = d;
    at.kv_pool = reinterpret_cast<const __nv_bfloat16*>(a->kv_pool);
    at.page_elems = (long long)a->layers * 2 * a->n_heads * a->page_size * HEAD_DIM;
    at.layer_off = (long long)a->layer * 2 * a->n_heads * a->page_size * HEAD_DIM;
    at.block_table = a->block_table; at.bt_stride = a->bt_stride;
    at.row_seq = a->row_seq; at.row_pos = a->row_pos;
    at.out = a->out; at.ldo = d;
    at.ws_part = static_cast<float*>(workspace);
    at.ws_count = reinterpret_cast<int*>(static_cast<char*>(workspace) + p.part_bytes);
    at.rows = a->rows; at.n_heads = a->n_heads; at.page_size = a->page_size;
    at.n_splits = p.splits; at.plan = PLAN_ROWS; at.kv_swizzled = 1;
    at.err = nullptr;
    CUDA_TRY(launch_attention_tc(at, static_cast<cudaStream_t>(cuda_stream), false));
    return MTP_OK;
}

}  // extern "C"
