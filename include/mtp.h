/*
 * mtp.h -- C ABI of the GB300 (sm_103a) multi-token-prediction decode path.
 *
 * The operation: accelerated inference of an autoregressive codec-token
 * language model (Sec. III-A, Eq. 1) extended with n multi-token-prediction
 * heads (Sec. III-B) and Viterbi-based selection of the token sequence to
 * accept from the heads' top-k candidates (Sec. III-C).  Every step of the
 * path runs in this library's CUDA kernels; the caller supplies memory
 * (host or device pointers, as each call states) and a CUDA stream.
 *
 * Conventions for every call:
 *   - return value: MTP_OK (0) or a negative mtp_status; mtp_last_error()
 *     then gives a message (per thread, valid until the next call);
 *   - pointers marked "host or device" are classified with
 *     cudaPointerGetAttributes; device pointers must be on the context's GPU;
 *   - the caller owns every buffer it passes; the library owns only the
 *     device state inside an mtp_ctx and frees it in mtp_destroy;
 *   - calls on one context are not thread-safe; calls on different contexts are;
 *   - work is ordered on the stream given to mtp_create (or, for the
 *     stand-alone operators, the stream passed in); calls that return data
 *     to host memory synchronise that stream first.
 */
#ifndef MTP_H
#define MTP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define MTP_API __attribute__((visibility("default")))
#define MTP_ABI_VERSION 1

typedef enum mtp_status {
    MTP_OK = 0,
    MTP_ERR_INVALID = -1,   /* bad argument, size or handle                          */
    MTP_ERR_NO_PAGES = -2,  /* KV page pool cannot hold the requested sequence        */
    MTP_ERR_CUDA = -3,      /* a CUDA runtime call failed (message has the CUDA text) */
    MTP_ERR_WEIGHTS = -4,   /* weight blob malformed or inconsistent with the config  */
    MTP_ERR_DEVICE = -5     /* a kernel set the device error word (bounded wait ran
                               out or an index failed its check); the context must be
                               destroyed */
} mtp_status;

typedef enum mtp_dtype { MTP_F32 = 0, MTP_BF16 = 1 } mtp_dtype;

/* Acceptance of the selected path (Sec. III-C).
 *   MTP_ACCEPT_ALL      the paper's rule: the whole Viterbi path is accepted each
 *                       step, cut after the first EOS and at the remaining budget.
 *   MTP_VERIFY_GREEDY   speculative decoding with the heads as drafter (the
 *                       "speculative decoding" framing of Sec. I-II): a step feeds
 *                       the confirmed token and the drafts of the previous step,
 *                       keeps the drafts while each equals head 1's argmax at the
 *                       row before it, rolls back the cache rows of the rest, and
 *                       emits the kept drafts plus head 1's argmax at the last kept
 *                       row.  The next drafts are the Viterbi path with position 1
 *                       forced to that argmax.  The output equals greedy AR decoding. */
typedef enum mtp_accept { MTP_ACCEPT_ALL = 0, MTP_VERIFY_GREEDY = 1 } mtp_accept;

/* Model and capacity.  The model is a decoder-only transformer over one
 * concatenated sequence [phonemes ; acoustic prompt ; generated codes]
 * (Sec. III-A) with sinusoidal absolute positions, pre-LN blocks (exact-erf
 * GELU MLP, biased linears), a final LayerNorm and n_heads_max linear heads
 * d_model -> codec_vocab; head i (1-based) predicts the token i positions
 * ahead (Sec. III-B). */
typedef struct mtp_config {
    int32_t layers;        /* transformer blocks                                   */
    int32_t d_model;       /* multiple of 256, at most 1024                         */
    int32_t n_attn_heads;  /* d_model / n_attn_heads must be 64                    */
    int32_t d_ffn;         /* multiple of 256                                      */
    int32_t phone_vocab;   /* phoneme table rows                                   */
    int32_t codec_vocab;   /* codec ids + EOS (1025 in the paper's setting), <= 1056 */
    int32_t eos_id;        /* EOS id inside [0, codec_vocab)                        */
    int32_t n_heads_max;   /* heads stored in the blob, 1..8                        */
    int32_t top_k_max;     /* largest top_k a call may ask for, 1..32               */
    int32_t max_batch;     /* sequence slots, 1..1024                               */
    int32_t max_ctx;       /* longest prompt + generation + n_heads_max per slot    */
    int32_t page_size;     /* KV tokens per page: 16, 32, 64 or 128                 */
    int32_t n_pages;       /* pages in the pool; 0 = max_batch * ceil(max_ctx/page) */
    int32_t weight_dtype;  /* mtp_dtype of matrices and embedding tables            */
    int32_t accept_policy; /* mtp_accept                                            */
    float ln_eps;          /* LayerNorm epsilon                                     */
} mtp_config;

/*
 * Weight blob (host memory, read during mtp_create only):
 *   bytes 0..7   magic "MTPWGT01"
 *   u32          version (1)
 *   u32          n_tensors = 5 + 12 * layers + 2
 *   u64          reserved (0)
 *   n_tensors x { u64 offset_from_blob_start; u64 nbytes; }
 *   tensor data; every offset a multiple of 256.
 * Tensors in this order (row-major; "W" = weight_dtype, "f" = fp32):
 *   tok_phone [phone_vocab, d] W      tok_codec [codec_vocab, d] W
 *   per layer: ln1_g [d] f, ln1_b [d] f, wqkv [3d, d] W (rows q | k | v, head h
 *              at rows h*64..h*64+63 of each part), bqkv [3d] f, wo [d, d] W,
 *              bo [d] f, ln2_g [d] f, ln2_b [d] f, w1 [d_ffn, d] W,
 *              b1 [d_ffn] f, w2 [d, d_ffn] W, b2 [d] f
 *   lnf_g [d] f, lnf_b [d] f, w_heads [n_heads_max, codec_vocab, d] W,
 *   b_heads [n_heads_max, codec_vocab] f,
 *   log_q [codec_vocab, codec_vocab] f  -- log of the token transition matrix
 *              Q of Sec. III-C, log_q[i][j] = log Q(i -> j).
 * A linear layer computes y = x W^T + b.
 */

typedef struct mtp_ctx mtp_ctx;

/* Create a context on the current CUDA device for the model of Sec. III-A
 * (the AR decoder theta_AR of Eq. 1) with the n MTP heads of Sec. III-B and
 * the transition matrix Q of Sec. III-C: validates config and blob, copies
 * the weights to the device (the caller keeps the blob), allocates the KV
 * page pool and all step buffers.  `cuda_stream` is a cudaStream_t
 * (NULL = legacy default stream) used by every later call on the context.
 * Errors: MTP_ERR_INVALID (config), MTP_ERR_WEIGHTS (blob), MTP_ERR_CUDA. */
MTP_API int mtp_create(const mtp_config* config, const void* weights_blob, size_t blob_bytes,
                       void* cuda_stream, mtp_ctx** out);

/* Free every device resource of the context made by mtp_create (the model of
 * Sec. III-A/B/C and its KV cache); NULL is ignored.  Synchronises the
 * context's stream first. */
MTP_API void mtp_destroy(mtp_ctx* ctx);

/* Message of the last failed call on this thread ("" if none). */
MTP_API const char* mtp_last_error(void);

/* Admit a sequence into slot `seq_slot` and run the prompt through the model
 * (Sec. III-A: [phonemes ; acoustic prompt] as one sequence).  Reserves
 * ceil((n_ph + n_ac + max_new_tokens + n_heads_max) / page_size) pages for
 * the slot (released by mtp_release or the next prefill of the slot), fills
 * their keys/values and keeps the last position's hidden state, from which
 * the next mtp_decode_step selects the first tokens.  `phonemes` and
 * `acoustic` are int32 ids, host or device; n_ph + n_ac >= 1.
 * Errors: MTP_ERR_INVALID (slot, ids out of range, length > max_ctx),
 * MTP_ERR_NO_PAGES, MTP_ERR_CUDA. */
MTP_API int mtp_prefill(mtp_ctx* ctx, int seq_slot, const int32_t* phonemes, int n_ph,
                        const int32_t* acoustic, int n_ac, int max_new_tokens);

/* Admit a sequence into slot `seq_slot` without running its prompt: the same
 * checks, page reservation and prompt copy as mtp_prefill, then the prompt
 * [phonemes ; acoustic prompt] (Sec. III-A) is prefilled by the following
 * decode steps, inside their batched pass beside the other slots' fed rows:
 * each step's prefill lane takes up to 128 prompt positions (a multiple of
 * n_heads) from the admitted slots in slot order, and a slot selects its
 * first tokens in the step after its last prompt row ran.  mtp_generate runs
 * such steps first; mtp_prefill_pending runs all admitted prompts at once.
 * Needs the batched path (bf16 weights) and MTP_ACCEPT_ALL; otherwise the
 * call is mtp_prefill.  Errors: as mtp_prefill. */
MTP_API int mtp_admit(mtp_ctx* ctx, int seq_slot, const int32_t* phonemes, int n_ph, const int32_t* acoustic,
                      int n_ac, int max_new_tokens);

/* Run every admitted prompt now (Sec. III-A prefill, many sequences per
 * pass): passes of up to all the batched rows, filled with the admitted
 * slots' remaining prompt positions in slot order, in attention groups of 8
 * positions of one slot.  Returns the number of passes (0: none pending).
 * Errors: MTP_ERR_INVALID (no batched path), MTP_ERR_CUDA, MTP_ERR_DEVICE. */
MTP_API int mtp_prefill_pending(mtp_ctx* ctx);

/* Return the slot's pages to the pool and mark it inactive. */
MTP_API int mtp_release(mtp_ctx* ctx, int seq_slot);  /* Errors: MTP_ERR_INVALID (slot), MTP_ERR_CUDA. */

/* One decode step for every active, unfinished slot (Fig. 1 caption,
 * Sec. III-B/C): feed the tokens accepted by the previous step (appending
 * their keys/values), apply the first `n_heads` heads to the last fed
 * position, take each head's `top_k` candidates (log-softmax descending,
 * lower id first on ties), select a path with Viterbi over that n x k
 * lattice and accept it under the context's policy.
 * Outputs (each may be NULL; host or device):
 *   out_tokens   int32 [max_batch][n_heads]: accepted tokens, -1 after them
 *   out_accepted int32 [max_batch]: tokens accepted this step (0 if idle)
 *   out_done     int32 [max_batch]: 1 once the slot has finished
 * Errors: MTP_ERR_INVALID (n_heads, top_k), MTP_ERR_CUDA, MTP_ERR_DEVICE. */
MTP_API int mtp_decode_step(mtp_ctx* ctx, int n_heads, int top_k, int32_t* out_tokens,
                            int32_t* out_accepted, int32_t* out_done);

/* Run decode steps until every active slot has finished, with no host
 * synchronisation between steps (ACCEPT_ALL: one round of ceil(budget / n)
 * steps; VERIFY_GREEDY, which emits 1..n tokens a step: rounds of
 * ceil(remaining / n) steps with one state read between rounds).  out_tokens (host or device, may be NULL)
 * receives each slot's generated tokens in row b at stride `out_stride`
 * (>= the slot's max_new_tokens); out_lens (may be NULL) their counts.
 * Steps run as CUDA graphs of eight chained steps where possible.
 * Returns the number of steps run (>= 0) or an error: MTP_ERR_INVALID
 * (n_heads, top_k, out_stride), MTP_ERR_CUDA, MTP_ERR_DEVICE. */
MTP_API int mtp_generate(mtp_ctx* ctx, int n_heads, int top_k, int32_t* out_tokens,
                         int out_stride, int32_t* out_lens);

/* Remove the last `n_tokens` cached positions of a slot: the rejected
 * tokens of a step, whose keys/values were appended when they were fed but
 * which the selection did not accept (the speculative-decoding framing of
 * Sec. I-II and the acceptance of Sec. III-C; MTP_VERIFY_GREEDY rolls back
 * on the device in the same way).  The pages stay reserved for the slot and
 * are reused by later appends.
 * Errors: MTP_ERR_INVALID (slot, n_tokens < 0 or > the cached length), MTP_ERR_CUDA. */
MTP_API int mtp_rollback(mtp_ctx* ctx, int seq_slot, int n_tokens);

/* Replace the tokens the next step feeds for a slot: the codec tokens that
 * extend the concatenated sequence of Sec. III-A (teacher forcing, for parity
 * tests; under MTP_VERIFY_GREEDY tokens[0] is the confirmed token and the
 * rest the drafts).  `tokens` (host, int32) of length 1..n_heads_max.
 * Errors: MTP_ERR_INVALID (slot, n, ids out of range), MTP_ERR_CUDA. */
MTP_API int mtp_set_teacher_tokens(mtp_ctx* ctx, int seq_slot, const int32_t* tokens, int n);

/* Slot state (host int32[6]): cached length, tokens pending to be fed,
 * remaining budget, done flag, active flag, tokens generated so far.
 * Errors: MTP_ERR_INVALID (slot, null), MTP_ERR_CUDA. */
MTP_API int mtp_seq_state(mtp_ctx* ctx, int seq_slot, int32_t* out6);

/* Logits and log-sum-exp of the last decode step (host or device):
 * out_logits float [max_batch][n_heads][codec_vocab] and out_lse float
 * [max_batch][n_heads] (either may be NULL), for the n_heads of that step.
 * The kernels rank candidates by logp = logits - lse rounded to fp32.
 * Errors: MTP_ERR_INVALID (no step run yet), MTP_ERR_CUDA. */
MTP_API int mtp_debug_logits(mtp_ctx* ctx, float* out_logits, float* out_lse);

/* Candidate lattice and selected path of the last decode step (host or
 * device, may be NULL): out_ids int32 and out_logp float [max_batch][n][k],
 * out_path int32 [max_batch][n].  Errors: MTP_ERR_INVALID (no step run yet), MTP_ERR_CUDA. */
MTP_API int mtp_debug_lattice(mtp_ctx* ctx, int32_t* out_ids, float* out_logp, int32_t* out_path);

/* Options:
 *   MTP_OPT_GRAPHS       1 = capture each (n_heads, top_k) step into a CUDA graph (default)
 *   MTP_OPT_PDL          1 = programmatic dependent launch between kernels (default)
 *   MTP_OPT_L2_PREFETCH  1 = each block kernel prefetches the next layer's weights into L2; 0 = no
 *                        prefetch (default: measured no faster, and it doubles the DRAM reads)
 *   MTP_OPT_MLP_CLUSTERS thread-block clusters of the MLP kernel (>= 1; default: as many as
 *                        the GPU holds at once)
 *   MTP_OPT_BATCHED      1 = decode steps whose fed rows (max_batch * n_heads) exceed one fused
 *                        pass (8 rows) run the batched path: tensor-core projections over all
 *                        rows at once (bf16 weights only; default); 0 = fused passes of 8 rows
 *   MTP_OPT_GEMM_SPLITS  most K splits of a batched-path projection (power of two 1..64; each
 *                        split adds its partial tile with fp32 atomics; default 16)
 *   MTP_OPT_LATTICE      states of the Viterbi search (Sec. III-C): 0 = each position's own head
 *                        top-k (default); 1 = the union of all heads' top-k at every position,
 *                        each scored by that position's head (the paper's reduced m x m matrix)
 *   MTP_OPT_SAMPLING     0 = select the lattice's best path (Viterbi, default); 1 = draw one path
 *                        from the lattice's posterior P(path) ~ prod_t Q(c_{t-1}, c_t) S_t(c_t)
 *                        (the top-k sampling that keeps diversity, Fig. 2 caption), by forward
 *                        filtering and backward sampling in fp32.  Under MTP_VERIFY_GREEDY only
 *                        the drafts are drawn; the output stays greedy.
 *   MTP_OPT_PERSISTENT   1 = a pass of <= 8 fed rows with bf16 weights runs its embedding and all
 *                        blocks as one persistent kernel (one CTA per SM in clusters of 4, weights
 *                        and cached keys streamed into shared-memory rings ahead of use, bounded grid
 *                        barriers between the attention and MLP phases), where the model and GPU
 *                        allow it; 0 = two block kernels per layer (default: faster on GB300 at B = 1)
 *   MTP_OPT_PREFILL_TC   1 = prefill passes (mtp_prefill, mtp_prefill_pending) run their attention
 *                        on the tensor cores (tcgen05: tiles of 128 prompt rows, 128-key items, S and
 *                        P V accumulated in TMEM); 0 = the split-key kernel of the decode steps, in
 *                        groups of 8 rows (default: on GB300 the serving prompts prefill faster so,
 *                        42 vs 58 ms at B = 32, 125 vs 144 ms at B = 128)
 *   MTP_OPT_GEMM_CLUSTER 1 = the batched path's projections at up to 128 fed rows run as one
 *                        activation tile per weight tile, their K split over the CTAs of a cluster
 *                        (up to 8) that sum the partial tiles in distributed shared memory, each
 *                        CTA finishing its share of the rows (q|k|v append, GELU pack, residual
 *                        add); more splits than a cluster holds add by atomics (default); 0 =
 *                        tiles of 32 rows, K split only where the output is accumulated
 *   MTP_OPT_HEADS_FUSED  heads, log-softmax and top-k of more than 8 hidden rows as one tensor-core
 *                        kernel (LN_f rows as bf16 hi + lo; per (tile of 128 rows, head) a cluster of
 *                        8 CTAs over vocabulary slices, lse merged in the cluster before the top-k):
 *                        0 = never (heads GEMM into memory, then the selection kernel's top-k);
 *                        1 = in mtp_heads_topk (default: 65.8 vs 94.6 us for 256 rows, n = 8, top-16);
 *                        2 = also in batched decode steps (measured 1.2 % slower per step at B = 32)
 *   MTP_OPT_SEED         seed of the path draws (any 32-bit value, zero-extended; default 0).
 *                        Position t of a draw of slot b that has generated g tokens uses the
 *                        uniform (SplitMix64(x) >> 40) / 2^24, x = ((seed * P + b) * P + g) * P + t
 *                        mod 2^64, P = 0x100000001B3, so runs are reproducible.  Changing either
 *                        option recaptures the step graphs. */
typedef enum mtp_option {
    MTP_OPT_GRAPHS = 0, MTP_OPT_PDL = 1, MTP_OPT_L2_PREFETCH = 2, MTP_OPT_MLP_CLUSTERS = 3, MTP_OPT_BATCHED = 4,
    MTP_OPT_GEMM_SPLITS = 5, MTP_OPT_LATTICE = 6, MTP_OPT_SAMPLING = 7, MTP_OPT_SEED = 8,
    MTP_OPT_PERSISTENT = 9, MTP_OPT_PREFILL_TC = 10, MTP_OPT_HEADS_FUSED = 11, MTP_OPT_GEMM_CLUSTER = 12
} mtp_option;
MTP_API int mtp_set_option(mtp_ctx* ctx, int option, int value);
MTP_API int mtp_get_option(mtp_ctx* ctx, int option, int32_t* value);

/* Kernel classes reported by mtp_profile_step. */
/*   EMBED       token embedding + position of the fed rows
 *   ATTN_BLOCK  LN1, q|k|v projection, key/value append, attention, W_o
 *   MLP         LN2, W1, GELU, W2
 *   HEADS       LN_f and the n heads' logits
 *   SELECT      log-softmax, top-k, Viterbi, acceptance
 *   SAVE        copy of each slot's last hidden state (multi-pass steps, prefill)
 * and of the batched path (all slots' rows in one pass, bf16 weights):
 *   PACK        LN / copy / GELU of the rows into bf16 hi + lo GEMM operands
 *   GEMM        a tensor-core projection (q|k|v, W_o, W1 or W2)
 *   QKV         query rows out, keys and values appended to the cache
 *   ATTN        split-KV attention of the fed rows over the cache
 * and of the persistent path (bf16 weights, <= 8 fed rows per pass):
 *   STEP        one persistent kernel: the fed rows' embedding and every block
 *   STEP_ATTN   (trace only) one attention phase of a layer inside STEP
 *   STEP_MLP    (trace only) one MLP phase of a layer inside STEP
 *   STEP_CTA    (trace only) one CTA's attention or MLP phase of the middle layer */
typedef enum mtp_kernel_kind {
    MTP_K_EMBED = 0, MTP_K_ATTN_BLOCK = 1, MTP_K_MLP = 2, MTP_K_HEADS = 3, MTP_K_SELECT = 4,
    MTP_K_SAVE = 5, MTP_K_PACK = 6, MTP_K_GEMM = 7, MTP_K_QKV = 8, MTP_K_ATTN = 9, MTP_K_STEP = 10,
    MTP_K_STEP_ATTN = 11, MTP_K_STEP_MLP = 12,
    MTP_K_STEP_CTA = 13, MTP_K_ATTN_TC = 14, MTP_K_COUNT = 15
} mtp_kernel_kind;

/* Run one decode step with each kernel launched alone (no graph, no PDL)
 * and bracketed by CUDA events on the context's stream.  out_ms[kind]
 * receives the summed device time (ms) and out_launches[kind] the launch
 * count, for kinds 0..MTP_K_COUNT-1 (host arrays).  The step's effect on
 * the slots is the same as mtp_decode_step. */
MTP_API int mtp_profile_step(mtp_ctx* ctx, int n_heads, int top_k, float* out_ms,
                             int32_t* out_launches);

/* Run one decode step (graph and PDL as the options say) with a timeline
 * record per kernel launch: out int64 [cap][MTP_TRACE_COLS] rows of
 * {mtp_kernel_kind, earliest CTA start, latest CTA past its dependency wait,
 * latest CTA end, then 8 phase marks (latest CTA past each, 0 if unused)},
 * times in ns of the GPU's global timer.  A STEP launch is followed by one
 * row per phase of each layer (STEP_ATTN, STEP_MLP): earliest CTA start of the
 * phase, latest CTA start, latest CTA end, marks; then two rows per CTA
 * (STEP_CTA, attention then MLP phase of the middle layer): that CTA's start,
 * its index, its end and marks.  Returns the number of launches
 * recorded (<= cap).  The step's effect on the slots is that of
 * mtp_decode_step. */
#define MTP_TRACE_COLS 12
MTP_API int mtp_trace_step(mtp_ctx* ctx, int n_heads, int top_k, int64_t* out, int cap);

/* Algorithmic bytes of one decode step: weights read (all blocks and the
 * first n_heads heads) plus keys/values read and written for every active
 * slot, from the current slot state (host uint64 out). */
MTP_API int mtp_step_bytes(mtp_ctx* ctx, int n_heads, uint64_t* out_bytes);

/* Self-test of the bounded waits (failure detection without a GPU fault): one
 * block waits on a shared-memory barrier that nothing completes.  The wait
 * gives up after its poll limit (the same bounded wait every kernel's barrier
 * waits use; well under a few seconds), ORs MTP_DEVICE_ERR_WAIT (1) into
 * *err_word and the kernel returns, leaving the CUDA context usable.
 *   err_word  int32, device memory
 * Errors: MTP_ERR_INVALID (null), MTP_ERR_CUDA. */
#define MTP_DEVICE_ERR_WAIT 1
MTP_API int mtp_selftest_bounded_wait(int32_t* err_word, void* cuda_stream);

/* Self-test of the persistent step kernel's grid barrier bound: one CTA
 * arrives at a grid barrier that expects two arrivals.  Its poll loop gives up
 * after its limit (about a second), ORs MTP_DEVICE_ERR_WAIT into *err_word,
 * and the kernel returns; the barrier's counter is left at zero.
 *   err_word  int32, device memory
 * Errors: MTP_ERR_INVALID (null), MTP_ERR_CUDA. */
MTP_API int mtp_selftest_grid_barrier(int32_t* err_word, void* cuda_stream);

/* ---- stand-alone operators (device pointers, caller's stream) ---------- */

/* Viterbi selection over candidate lattices (Sec. III-C, reading A: the
 * states at position t are head t's top-k candidates).  In the log domain,
 * delta_1(j) = s_1(j) and
 *   delta_t(j) = max_i [ delta_{t-1}(i) + log_q(c_{t-1,i}, c_{t,j}) ] + s_t(j),
 * each add one fp32 add in that order, the lowest i taking ties; the path
 * ends in the lowest j maximising delta_n.  Then ACCEPT_ALL: accepted =
 * min(n, first EOS index + 1, remaining[b]) and rollback = 0.
 *   cand_ids  int32 [batch][n][k], ids in [0, vocab)
 *   cand_logp float [batch][n][k]
 *   log_q     float [vocab][vocab]
 *   remaining int32 [batch] or NULL (no budget)
 * Outputs int32 out_path [batch][n], float out_score [batch] (may be NULL),
 * int32 out_accepted [batch], int32 out_rollback [batch] (may be NULL).
 * Limits: 1 <= n <= 8, 1 <= k <= 32.  Errors: MTP_ERR_INVALID, MTP_ERR_CUDA. */
MTP_API int mtp_viterbi(int batch, int n, int k, int vocab, int eos_id,
                        const int32_t* cand_ids, const float* cand_logp, const float* log_q,
                        const int32_t* remaining, int32_t* out_path, float* out_score,
                        int32_t* out_accepted, int32_t* out_rollback, void* cuda_stream);

/* The context's heads on `batch` hidden states (Sec. III-B): z = LN_f(h),
 * logits_i = z W_i^T + b_i for i < n_heads, logp = logits - lse, top-k.
 *   hidden     [batch][d_model], dtype hidden_dtype (mtp_dtype), device
 *   out_ids    int32 [batch][n_heads][top_k]; out_logp float, same shape
 *   out_logits float [batch][n_heads][codec_vocab] or NULL
 *   out_lse    float [batch][n_heads] or NULL
 * More than 8 rows with bf16 weights run on the tensor cores (LN_f rows packed
 * as bf16 hi + lo, one GEMM over the n_heads * codec_vocab weight rows, head
 * weights streamed once per chunk of rows); otherwise passes of 8 rows.
 * Uses the context's stream.  Errors: MTP_ERR_INVALID, MTP_ERR_CUDA. */
MTP_API int mtp_heads_topk(mtp_ctx* ctx, int batch, const void* hidden, int hidden_dtype,
                           int n_heads, int top_k, int32_t* out_ids, float* out_logp,
                           float* out_logits, float* out_lse);

/* Causal attention of `rows` query rows over a paged bf16 KV pool (the
 * attention of one block, Sec. III-A), split over the key axis with a
 * log-sum-exp merge.  Pool layout: bf16 [n_pages][layers][2][n_heads][page_size][64],
 * index 0 of the "2" axis keys, 1 values.  Rows are grouped: group g is rows
 * g*rows_per_group ..; all active rows of a group belong to one slot.
 *   q          float [rows][n_heads*64] (unscaled)
 *   row_seq    int32 [rows]: slot of the row, < 0 = inactive row (skipped)
 *   row_pos    int32 [rows]: position; the row sees keys 0..row_pos
 *   block_table int32 [slots][bt_stride]: page of each page_size span
 *   out        float [rows][n_heads*64]
 *   workspace  device scratch of mtp_attention_workspace_bytes(...) bytes;
 *              its counters must be zero on the first call and are left zero.
 *   max_keys   upper bound of (row_pos + 1) over all rows; sets the split count
 * Keys/values for positions 0..max row_pos of each group must be present.
 * Errors: MTP_ERR_INVALID, MTP_ERR_CUDA. */
typedef struct mtp_attention_args {
    int32_t rows, rows_per_group, n_heads, page_size, layers, layer, bt_stride, max_keys;
    const float* q;
    const uint16_t* kv_pool;
    const int32_t* block_table;
    const int32_t* row_seq;
    const int32_t* row_pos;
    float* out;
} mtp_attention_args;
MTP_API size_t mtp_attention_workspace_bytes(const mtp_attention_args* args);
MTP_API int mtp_attention(const mtp_attention_args* args, void* workspace, size_t workspace_bytes,
                          void* cuda_stream);

/* The same attention on the tensor cores (tcgen05), as prefill passes run it
 * (Sec. III-A: every prompt position attends to itself and the positions before
 * it).  Rows form tiles of 128 (rows_per_group is not used); the rows of a tile
 * may belong to any slots, each row sees keys 0..row_pos of its own slot.  Per
 * tile, head and 128 cached keys: S = Q K^T and O = P V on the tensor cores
 * with fp32 accumulators in TMEM (Q and P as bf16 hi + lo pairs), the online
 * softmax in registers; key ranges split across CTAs are merged with a
 * log-sum-exp.  The pool must hold each key and value row in the context's
 * cache layout: 16-byte chunk c of row t of a page at chunk position
 * c ^ (t mod 8).  Other arguments and layouts as mtp_attention; row_seq < 0 rows
 * are left untouched.  workspace: mtp_attention_tc_workspace_bytes(args) bytes,
 * counters zero on the first call and left zero.
 * Errors: MTP_ERR_INVALID (sizes, null pointers, workspace too small, q not
 * 16-byte aligned), MTP_ERR_CUDA. */
MTP_API size_t mtp_attention_tc_workspace_bytes(const mtp_attention_args* args);
MTP_API int mtp_attention_tc(const mtp_attention_args* args, void* workspace, size_t workspace_bytes,
                             void* cuda_stream);

/* mtp_attention without a caller workspace and without any allocation.  The
 * paper has no counterpart: this serves callers that must not allocate GPU
 * memory while they run -- for instance a real-time audio callback, where
 * cudaMalloc/cudaFree may block on the driver or synchronise the device and
 * so stall playback, or a host application that owns every byte of GPU
 * memory and hands none to the library.
 * The split-merge scratch lives in one fixed device array of
 * MTP_ATTENTION_NOALLOC_SCRATCH_BYTES per GPU, held from library load until
 * process exit and shared by every call on that GPU.  A call whose scratch
 * need (mtp_attention_workspace_bytes) exceeds it fails with MTP_ERR_INVALID
 * before launching anything, as does any invalid argument: nothing is queued
 * then.  Every call looks up the array's device address (which allocates
 * nothing); the first call on a device may also load the library's device
 * code, so make that first call before any stream capture.  Each call clears
 * the merge counters it uses (an asynchronous memset on the stream); the
 * partial results keep the last call's contents.  Calls that
 * overlap on the GPU (other streams or threads) race on the array: order
 * them on one stream.  Arguments, outputs and errors as mtp_attention.  No
 * cudaMalloc, cudaFree or allocating library call is made. */
#define MTP_ATTENTION_NOALLOC_SCRATCH_BYTES (4u << 20)
MTP_API int mtp_attention_noalloc(const mtp_attention_args* args, void* cuda_stream);

/* The batched path's tensor-core projection (the block's linear layers,
 * Sec. III-A, for many fed rows at once):
 *   out[i][f] (+)= sum_k (a_hi[i][k] + a_lo[i][k]) * w[f][k]
 * w: device bf16 [n_w][k] row-major; a_hi, a_lo: device bf16 [m][k]
 * row-major, the two parts of fp32 activations (a_lo = a - a_hi); out:
 * device fp32 [m][n_w].  n_w a multiple of 128, k a multiple of 64 with
 * (k / 64) divisible by splits, 1 <= m <= 4096; all pointers 16-byte
 * aligned.  splits > 1 splits the reduction across CTAs and requires
 * accumulate = 1 (fp32 atomic adds into out, so the summation order and the
 * last bits vary between runs); accumulate = 0 stores.  Runs on cuda_stream
 * and synchronises it before returning.  Errors: MTP_ERR_INVALID (shapes,
 * alignment), MTP_ERR_CUDA, MTP_ERR_DEVICE (a bounded wait ran out). */
MTP_API int mtp_gemm_bf16x2(const void* w, const void* a_hi, const void* a_lo, float* out, int n_w, int k, int m,
                            int splits, int accumulate, void* cuda_stream);

#ifdef __cplusplus
}
#endif
#endif /* MTP_H */
