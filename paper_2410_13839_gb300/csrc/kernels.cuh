// kernels.cuh -- argument blocks and host launchers of libmtp's kernels.
//
// Each launcher enqueues one kernel on `stream`.  With `pdl` set the launch
// carries the programmatic-stream-serialisation attribute: the kernel may
// start while its predecessor is still running, prefetches what does not
// depend on it (weights, old keys/values), then waits (griddepcontrol.wait).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

struct mtp_attention_args;  // include/mtp.h

namespace mtp {

constexpr int HEAD_DIM = 64;     // attention head width (fixed by the kernels)
constexpr int MAX_ROWS = 8;      // rows per weight-streaming pass (B * n_heads per chunk)
constexpr int PREFILL_ROWS = 128; // prompt positions per batched-path prefill chunk
constexpr int MAX_TOPK = 32;     // one warp lane per candidate
constexpr int MAX_NHEADS = 8;    // prediction heads
constexpr int MAX_VOCAB = 1056;  // 33 logits per lane in the top-k warp

// ---------------------------------------------------------------- GEMV ----
// y[m, f] = epilogue( sum_k A'[m, k] W[f, k] + bias[f] ),  A' = LN(A) if ln_g.
enum Epilogue : int {
    EPI_QKV = 0,     // f < d: q[m, f];  d <= f < 3d: key/value into the KV page pool
    EPI_RESID = 1,   // out[m, f] += y   (residual stream); optional h_last copy
    EPI_GELU = 2,    // out[m, f] = GELU(y)
    EPI_LOGITS = 3,  // out[m, f] = y
};

struct GemvArgs {
    const float* A; int lda;             // input rows [M][K] fp32
    const float* ln_g; const float* ln_b; float ln_eps;  // LayerNorm prologue (ln_g null: none)
    const void* W;                       // [N][K] row-major, bf16 or fp32
    const float* bias;                   // [N]
    int N, K, M;                         // M <= rows of the instantiation
    int rows_per_cta;
    const int* row_seq;                  // [M] slot of each row, < 0 inactive (null: all active)
    const int* row_pos;                  // [M] position of each row (EPI_QKV)
    const int* row_last;                 // [M] 1 if the row is its slot's last fed row
    float* out; int ldo;                 // q / residual / hidden / logits
    float* h_last; int ld_h;             // EPI_RESID: copy of the final row per slot (may be null)
    // EPI_QKV key/value placement
    uint16_t* kv_pool; long long page_elems; long long layer_off; int n_heads, page_size, d_model;
    const int* block_table; int bt_stride;
    // optional row gather: row m is gather_x row (m * gather_n + npend - 1) when
    // npend = gather_npend[gather_base + m] > 0, else A row m
    const float* gather_x; const int* gather_npend; int gather_n, gather_base;
    int* err;
    unsigned long long* trace;           // timeline record of this launch (may be null)
};

size_t gemv_smem_bytes(int rows_per_cta, int K, int wbytes, int M);
cudaError_t launch_gemv(const GemvArgs& a, int epi, bool ln, bool w_bf16, int grid, cudaStream_t s, bool pdl);

// ----------------------------------------------------------- attention ----
enum AttnPlan : int {
    PLAN_ROWS = 0,    // slot and key count read from row_seq/row_pos after the wait
    PLAN_DEVICE = 1,  // slot = seq_base + group; old length and new count from device state
    PLAN_VALUE = 2,   // one group: slot, old length and new count passed by value
};

struct AttnArgs {
    const float* q; int ldq;                   // [rows][H*64]
    const __nv_bfloat16* kv_pool; long long page_elems; long long layer_off;
    const int* block_table; int bt_stride;
    const int* row_seq; const int* row_pos;
    float* out; int ldo;                       // fp32 output rows, or null
    __nv_bfloat16* out_hi; __nv_bfloat16* out_lo; int ldb;  // or null: output rows as bf16 hi + lo (the
                                               // W_o GEMM's operand; rows of no sequence written as zeros)
    float* ws_part; int* ws_count;             // split partials and per-(group, head) counters
    int rows_per_group, n_heads, page_size, n_splits;
    int plan;
    const int* seq_len; const int* seq_new; int seq_base;   // PLAN_DEVICE
    int val_seq, val_old, val_new;                           // PLAN_VALUE
    int* err;
    unsigned long long* trace;
    int kv_swizzled;                                         // pages store chunk c of key row t at c ^ (t & 7)
    int rows;                                                // attention_tc: rows of the pass (tiles of 128)
};

constexpr int ATTN_CTAS_PER_SM = 4;  // attn_kernel: 128 threads x at most 128 registers, ~51 KB of shared memory
constexpr int ATTN_MAX_SPLITS = 32;  // key splits one launch merges
size_t attn_workspace_floats(int groups, int n_heads, int n_splits, int rows_per_group);
size_t attn_smem_bytes(int page_size);
int attn_splits_for(int groups, int n_heads, int page_size, int max_keys, int num_sms);
cudaError_t launch_attention(const AttnArgs& a, int groups, cudaStream_t s, bool pdl);
// Tensor-core (tcgen05) causal attention of prompt rows: tiles of 128 rows of
// any slots, 128-key items, swizzled pages only; grid (n_splits, heads, tiles).
size_t attn_tc_workspace_floats(int tiles, int n_heads, int n_splits);
int attn_tc_tiles(int rows);
int attn_tc_splits_for(int tiles, int n_heads, int max_keys, int num_sms);
cudaError_t launch_attention_tc(const AttnArgs& a, cudaStream_t s, bool pdl);

// ------------------------------------------------------- fused block ----
// One transformer block over <= MAX_ROWS fed rows: attn_block (LN1, q|k|v,
// key/value append, attention, W_o) and mlp (LN2, W1, GELU, W2), each
// accumulating into a zeroed residual buffer.
constexpr int MLP_CLUSTER = 4;   // CTAs per cluster of the MLP kernel (4: 36 clusters fit one CTA per SM)

struct LayerArgs {
    const float* x_in;        // [M][d] input rows of the kernel
    float* x_out;             // [MAX_ROWS][d] accumulation target (zero on entry)
    float* x_zero;            // [MAX_ROWS][d] buffer the next kernel accumulates into
    int M, d, d_ffn, n_heads, rows_per_group;
    const int* row_seq; const int* row_pos;
    const float* ln_g; const float* ln_b; float ln_eps;
    // attention half (weights head-major: q|k|v rows of head h, W_o columns of head h)
    const void* wqkv;         // [H][3*64][d]
    const float* bqkv;        // [H][3*64]
    const void* wo;           // [H][d][64]
    const float* bo;          // [d]
    __nv_bfloat16* kv_pool; long long page_elems; long long layer_off; int page_size;
    const int* block_table; int bt_stride;
    int plan; const int* seq_len; const int* seq_new; int seq_base; int val_seq, val_old, val_new;
    const int* active; const int* done; int slots;          // PLAN_DEVICE row rule (as the embedding)
    // next layer's weights of the same kernel, prefetched into L2 (null: none)
    const void* next_w_a; const void* next_w_b;
    // MLP half
    const void* w1;           // [d_ffn][d]
    const void* w2t;          // [d_ffn][d]  (W2 transposed)
    const float* b1; const float* b2;
    int ffn_rows_per_cta;
    int* err;
    unsigned long long* trace;
};

size_t attn_block_smem_bytes(int d, int wbytes, int page_size);
size_t mlp_smem_bytes(int d, int rows_per_cta, int wbytes);
cudaError_t launch_attn_block(const LayerArgs& a, bool w_bf16, cudaStream_t s, bool pdl);
cudaError_t launch_mlp(const LayerArgs& a, bool w_bf16, int grid, cudaStream_t s, bool pdl);
// clusters of the MLP kernel that can be resident at once (rows per CTA chosen for that count)
cudaError_t mlp_max_clusters(int d, int num_sms, int wbytes, int d_ffn, int* clusters);

// ------------------------------------------------ persistent step ----
// The embedding and every block of one decode pass (<= MAX_ROWS fed rows,
// bf16 weights) as one persistent kernel of clusters of SK_CLUSTER CTAs, one
// CTA per SM, each fed by a ring of SK_STAGE_BYTES shared-memory stages
// (step_kernel.cu).
constexpr int SK_CLUSTER = 4;
constexpr int SK_STAGE_BYTES = 16384;
constexpr int SK_MAX_STAGES = 12;

struct StepArgs {
    int L, d, F, H;                  // layers, model width, FFN width, attention heads (d = 64 H)
    int rows, rpg, seq_base, slots;  // fed rows, rows per slot (n), first slot, slots in the context
    int n_max, page_size, codec_vocab, max_pos;
    float ln_eps;
    // layer 0's tensors in their device layouts; layer l's is at + l * layer_stride bytes
    const float *ln1_g, *ln1_b, *bqkv, *bo, *ln2_g, *ln2_b, *b1, *b2;
    const __nv_bfloat16* wqkv;       // [H][q|k|v 64 rows][d]
    const __nv_bfloat16* wo;         // [H][d][64]
    const __nv_bfloat16* w1;         // [F][d]
    const __nv_bfloat16* w2t;        // [F][d] (W2 transposed)
    long long layer_stride;
    const __nv_bfloat16* tok_codec;  // [codec_vocab][d]
    const float* pe;                 // [max_pos][d]
    // slot state, read after the dependency wait
    const int *active, *done, *n_pending, *pending, *seq_len;
    __nv_bfloat16* kv_pool; long long page_elems;
    const int* block_table; int bt_stride;
    // work split and ring
    const int2* ffn_range;           // [grid]: first FFN unit and unit count of each CTA
    int res_cluster;                 // the cluster (one with FFN units) that adds x_mid + b2
    int ffn_unit_rows;               // FFN rows per unit = weight rows per stage (SK_STAGE_BYTES / (2 d))
    int ring_stages;
    // buffers: residual rows [4][MAX_ROWS][d] (buffer 3 must be zero at entry), grid-barrier words [2]
    float* xbuf; unsigned* bar;
    int *row_seq, *row_pos, *row_last;  // [MAX_ROWS] plan of the pass (for the kernels after it)
    int* err;
    unsigned long long* trace;
};
// The residual buffer that holds the pass's final rows.
inline int step_final_buffer(int layers) { return (2 * layers - 2) % 3; }
// Ring stages that fit beside the kernel's other shared memory for mt (1, 2, 4 or 8) fed rows.
int step_ring_stages(int d, int mt);
// Clusters of SK_CLUSTER CTAs that can be resident at once (the 8-row footprint).
cudaError_t step_kernel_configure(int d, int* max_clusters);
cudaError_t launch_step_kernel(const StepArgs& a, int grid, cudaStream_t s, bool pdl);
// one CTA at a grid barrier that never completes: the bounded wait sets err and returns
cudaError_t launch_selftest_grid_barrier(int* err, cudaStream_t s);

// --------------------------------------------------------------- embed ----
struct EmbedArgs {
    int mode;                  // 0 = decode rows from slot state, 1 = prefill chunk, 2 = prefill lane rows
                               // (slot and position already in row_seq / row_pos at row0 + r, token from prompt)
    const void* tok_phone; const void* tok_codec; int w_bf16;
    int phone_vocab, codec_vocab;
    const float* pe; int d; int max_pos;   // positional table [max_pos][d]
    float* x;                  // [MAX_ROWS][d]
    int* row_seq; int* row_pos; int* row_last;
    int rows;                  // rows in this pass (<= MAX_ROWS); the rest are inactive
    // decode
    int seq_base, n_heads, n_max, slots;
    const int* active; const int* done; const int* n_pending; const int* pending; const int* seq_len;
    // prefill
    int slot, p0, n_ph, total, prompt_stride; const int* prompt;
    // prefill lane (mode 2): rows row0.. of the plan arrays; phoneme count of each slot's prompt
    int row0; const int* prompt_nph;
    float* zero_buf;           // [MAX_ROWS][d] zeroed (first residual accumulation target)
    int* err;
    unsigned long long* trace;
};
cudaError_t launch_embed(const EmbedArgs& a, cudaStream_t s, bool pdl);

// The prefill lane of a pass: up to `capacity` rows (a multiple of rpg) from
// row0 on, given to the slots with prompt tokens left in slot order, each
// slot's share padded to a multiple of rpg (attention groups hold one slot).
// Slot b gets take_b = min(left_b, capacity - start_b) rows, start_b = the
// padded demands of the slots before it; row i of its share is prompt
// position len_b + i, the share's last row is marked when it ends the
// prompt.  The kernel writes the rows' plan (row_seq/row_pos/row_last, -1
// for unused rows) and lane_take, and advances prompt_left and seq_len.
struct LanePlanArgs {
    int slots, rpg, capacity, row0;
    int* prompt_left; int* seq_len; const int* active; const int* done;
    int* row_seq; int* row_pos; int* row_last; int* lane_take;
};
cudaError_t launch_lane_plan(const LanePlanArgs& a, cudaStream_t s, bool pdl);
cudaError_t launch_pe_table(float* pe, int max_ctx, int d, cudaStream_t s);

// -------------------------------------------------------------- select ----
struct SelectArgs {
    const float* logits;      // [B][n][V]
    float* lse;               // [B][n]
    int32_t* cand_ids; float* cand_logp;   // [B][n][k]
    int32_t* path;            // [B][n]
    const float* log_q;       // [V][V]
    int n, k, V, eos_id, n_max, seq_base;
    // slot state (decode); null for the stand-alone heads call
    int* active; int* done; int* n_pending; int* pending; int* seq_len; int* remaining;
    int* gen_count; int* gen_tokens; int gen_stride;
    int* out_tokens; int* out_accepted;   // [B][n_max], [B]
    int* err;
    unsigned long long* trace;
    int policy;               // mtp_accept
    const int* kept;          // [B] VERIFY_GREEDY: drafts kept this step (verify_kernel)
    int lattice;              // 0: per-head top-k states (reading A); 1: union of all heads' top-k (reading B)
    int sampling;             // 0: the lattice's best path (Viterbi); 1: a path drawn from its posterior
    unsigned long long seed;  // path draws: counter-based uniforms of (seed, slot, tokens generated, position)
    const int* prompt_left;   // slots with prompt tokens left select nothing (null: no admitted prompts)
    const int* lane_take;     // with `lane`: slots whose prompt rows ran in this step's lane select nothing
    int lane;
    int pre_topk;             // 1: cand_ids / cand_logp / lse already hold the step's top-k (fused heads)
};
cudaError_t launch_select(const SelectArgs& a, int batch, bool do_accept, cudaStream_t s, bool pdl);

// VERIFY_GREEDY, per slot of one pass: head 1's top-1 at every fed row
// (logits1 [rows][V], row = slot-in-pass * n + j), the drafts kept (pending
// token j + 1 equal to the top-1 at row j), and the hidden row of the last
// kept position copied to h_last.
struct VerifyArgs {
    const float* logits1;     // head 1 logits of the pass's fed rows
    const float* x;           // the pass's final hidden rows [rows][d]
    float* h_last;            // [slots][d]
    int* kept;                // [slots]
    const int* active; const int* done; const int* n_pending; const int* pending;
    int n, V, d, n_max, seq_base;
    unsigned long long* trace;
};
cudaError_t launch_verify(const VerifyArgs& a, int slots, cudaStream_t s, bool pdl);

struct ViterbiArgs {
    int batch, n, k, vocab, eos_id;
    const int32_t* cand_ids; const float* cand_logp; const float* log_q; const int32_t* remaining;
    int32_t* path; float* score; int32_t* accepted; int32_t* rollback;
};
cudaError_t launch_viterbi(const ViterbiArgs& a, cudaStream_t s);

// --------------------------------------------------------------- misc ----
cudaError_t launch_convert_rows(const void* src, int src_bf16, float* dst, int rows, int d, cudaStream_t s);

// set fields of one slot's device state (a field is left alone when its value is < 0)
struct SlotSet {
    int slot;
    int* seq_len; int* n_pending; int* remaining; int* done; int* active; int* gen_count;
    int* prompt_left; int* prompt_nph;
    int set_len, set_pending, set_remaining, set_done, set_active, set_gen;
    int set_prompt_left, set_prompt_nph;
};
cudaError_t launch_slot_set(const SlotSet& set, cudaStream_t s);
cudaError_t launch_trace_reset(unsigned long long* trace, int records, cudaStream_t s);
// copy each slot's last fed row (row_last) of x [MAX_ROWS][d] into h_last [slot][d]
cudaError_t launch_save_last(const float* x, const int* row_seq, const int* row_last, float* h_last, int d, int rows,
                             unsigned long long* trace, cudaStream_t s, bool pdl);

// ------------------------------------------------------- batched path ----
enum PackMode : int { PACK_LN = 0, PACK_COPY = 1, PACK_GELU = 2 };
struct PackArgs {
    int mode;                     // PackMode
    const float* x; int ldx;      // input rows [m][ldx], k columns used
    float* zero_after;            // PACK_GELU: rows zeroed after reading (may be x), or null
    const float* gamma; const float* beta; float eps;   // PACK_LN
    const int* row_seq;           // rows with row_seq < 0 are packed as zeros (null: every row is packed,
                                  // and zero_buf [zero_n] is zeroed first)
    __nv_bfloat16* hi; __nv_bfloat16* lo;  // [m][k] bf16 parts: hi + lo = the fp32 row
    int k, m;                     // k <= 4096
    float* zero_buf; long long zero_n;  // or null: zeroed (an accumulation target of the next kernel)
    unsigned long long* trace;
};
cudaError_t launch_pack_rows(const PackArgs& a, cudaStream_t s, bool pdl);

// ------------------------------------------------ tensor-core GEMM ----
// out[n][f] (+)= sum_k (a_hi[n][k] + a_lo[n][k]) w[f][k] with tcgen05 (tc_gemm.cu).
enum TcEpilogue : int {
    TC_STORE = 0,     // out[n][f] = acc + bias (one K split only)
    TC_ACCUM = 1,     // out[n][f] += acc (+ bias from K split 0), fp32 atomics
    TC_QKV = 2,       // q|k|v rows (head-major features): q -> q_out, k and v -> the paged cache (one K split)
    TC_GELU_PACK = 3  // GELU(acc + bias) as bf16 hi + lo rows -> pack_hi / pack_lo (one K split)
};
struct TcGemmArgs {
    float* out; int ldo;          // [m][ldo] fp32, column f = weight row (TC_STORE, TC_ACCUM; TC_QKV: queries)
    const float* bias;            // [n_w] added once (by K split 0), or null
    int m;                        // activation rows
    int k_chunks;                 // 64-wide k-chunks per CTA (K / 64 / splits)
    int w_rows_per_kchunk;        // 0: weight k-chunk kc at columns 64 kc; else at rows kc * this (W_o per head)
    int epilogue;                 // TcEpilogue
    const int* row_seq; const int* row_pos;   // TC_QKV, TC_GELU_PACK: rows of no sequence are skipped / zero
    // TC_QKV: the paged cache (chunk c of key row t stored at c ^ (t & 7))
    __nv_bfloat16* kv_pool; long long page_elems; long long layer_off; int page_size, n_heads;
    const int* block_table; int bt_stride;
    __nv_bfloat16* pack_hi; __nv_bfloat16* pack_lo;  // TC_GELU_PACK: [m][n_w]
    int n_valid;                  // TC_ACCUM: 0, or only features < n_valid are added (element atomics, any ldo)
    int cluster_reduce;           // 0/1: none; c in 2..8: each c consecutive K splits of a tile are one cluster
                                  // that sums its partials in DSMEM, each CTA finishing 1/c of the rows
                                  // (any epilogue; more splits than c only for TC_ACCUM, added by atomics)
    int* err;
    unsigned long long* trace;
};
struct TcGemm {
    CUtensorMap w, a_hi, a_lo;    // boxes: 64 x 128 weight rows, 64 x nt activation rows
    TcGemmArgs args;
    int n_w, splits, nt;          // weight rows (multiple of 128), K splits, activation rows per tile
};
// 2-D bf16 tensor map [rows][inner] with a 64 x box_rows box; pre_swizzled: the
// tensor already stores chunk c of row r at c ^ (r & 7) (copied verbatim).
int tc_encode_2d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows, uint32_t box_rows,
                 bool pre_swizzled);
int tc_tile_rows(int m);          // activation rows per tile for m rows: 32, 64 or 128
cudaError_t launch_tc_gemm(const TcGemm& g, cudaStream_t s, bool pdl);
constexpr int TC_CLUSTER_SPLITS = 4;  // K splits one cluster sums in the batched path (clusters of 8 at one CTA per
                                      // SM: only 15 fit this GPU at once)

// ------------------------------------ fused heads + log-softmax + top-k ----
// The n heads over m rows of LN_f(h) given as bf16 hi + lo (heads_tc.cu): per
// (row, head) the lse and the top-k of logp = logit - lse by (logp desc, id
// asc); logits to memory only on request.
struct HeadsTcArgs {
    const float* bias;            // [n_max * V]
    int m, n, V, k;               // rows, heads, vocabulary, candidates
    int k_chunks;                 // d / 64
    int a_rows;                   // rows of the activation box: 32 or 64 (m <= that), else 128
    int32_t* out_ids; float* out_logp;   // [m][n][k]
    float* out_lse;               // [m][n] or null
    float* out_logits; int ldl;   // [m][ldl], head i at column i * V, or null
    float z;                      // set by launch_heads_tc: candidates are logp >= mean + z sd of the row (pruning)
    int* err;
    unsigned long long* trace;
};
struct HeadsTc {
    CUtensorMap w128, w144;       // head weight rows [n_max * V][d]: boxes of 64 x 128 and 64 x 144 rows
    CUtensorMap a_hi, a_lo;       // LN_f rows: boxes of 64 x a_rows rows
    HeadsTcArgs args;
};
bool heads_tc_supported(int V, int k);
int heads_tc_box_rows_wide();
cudaError_t launch_heads_tc(const HeadsTc& g, cudaStream_t s, bool pdl);

// Raise `kernel`'s dynamic shared-memory limit to at least `bytes` on the
// current device (and, with max_shared_carveout, prefer the whole unified L1
// as shared memory).  The attribute is per device: the call is made once per
// (kernel, device, size) and is safe from several threads.
cudaError_t ensure_kernel_smem(const void* kernel, size_t bytes, bool max_shared_carveout = false);

// The stand-alone attention operator (mtp_attention*): its arguments checked
// and its workspace laid out once, for every entry point that runs it.  The
// workspace holds the split partials (part_bytes, a multiple of 256) and then
// the per-(group, head) merge counters (count_bytes), which must be zero when
// a launch starts and are left zero by it.
struct AttnStandalonePlan {
    int groups, splits;
    size_t part_bytes, count_bytes, need;
};
// MTP_OK or MTP_ERR_INVALID / MTP_ERR_CUDA (message set); with check_pointers
// the device pointers must be non-null too.
int attention_standalone_plan(const struct ::mtp_attention_args* a, bool check_pointers, AttnStandalonePlan* p);
// Enqueue the kernel on `stream` with `workspace` laid out as `p` describes.
int attention_standalone_launch(const struct ::mtp_attention_args* a, const AttnStandalonePlan& p, void* workspace,
                                cudaStream_t stream);

// C-ABI error reporting shared by the translation units (message for mtp_last_error)
int report_error(int code, const char* msg);
void clear_error();

}  // namespace mtp
