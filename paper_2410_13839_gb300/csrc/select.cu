// select.cu -- log-softmax + top-k of each head, Viterbi over the candidate
// lattice, and acceptance (Sec. III-B, III-C).
//
// Top-k (one warp per head): each lane holds 33 of the V <= 1056 logits;
// lse = m + log(sum exp(l - m)) with a fixed reduction order; the ranking
// score is logp = l - lse rounded to fp32; k rounds of a warp arg-max with
// the key (score descending, id ascending) pick the candidates.
//
// Viterbi (one warp per sequence, lane j = candidate j, k <= 32): max-plus
// recursion over the n positions,
//   delta_t(j) = (max_i delta_{t-1}(i) + log_q[c_{t-1,i}][c_{t,j}]) + s_t(j),
// every add a single fp32 add (no contraction), the lowest i on ties, the
// backpointers in registers; the final state is the lowest j of the max.
// Acceptance (ACCEPT_ALL): the path is cut after its first EOS and at the
// remaining budget; the slot's state (cached length, fed tokens, output
// buffer, done flag) is updated on the device, so steps need no host sync.
// Union lattice (reading B, option): the states of every position are the
// m <= n*k distinct tokens of all heads' top-k (sorted by id), each scored by
// head t's full fp32 log-softmax; the same recursion, add order and lowest-index
// tie-breaks, one thread per state, transitions read from the L2-resident
// log Q.
// Path sampling (option): instead of the best path, one path drawn from the
// lattice's posterior (forward filtering, backward sampling) with SplitMix64
// uniforms of (seed, slot, tokens generated, position); either lattice.
// VERIFY_GREEDY: verify_kernel finds the drafts kept (head 1's top-1 at each
// fed row against the next fed token); select_kernel forces position 1 of
// the lattice to its top-1 candidate, emits the kept drafts and path[0],
// advances the cached length by the kept rows only (the rest is rolled
// back) and feeds the path next step.
#include <math.h>

#include "common.cuh"
#include "kernels.cuh"

namespace mtp {
namespace {

constexpr int VPL = MAX_VOCAB / 32;  // logits per lane

// (value desc, index asc) arg-max across the warp; every lane returns the winner.
__device__ __forceinline__ void warp_argmax(float& v, int& i) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(FULL_MASK, v, o);
        const int oi = __shfl_xor_sync(FULL_MASK, i, o);
        if (ov > v || (ov == v && oi < i)) {
            v = ov;
            i = oi;
        }
    }
}

// One head: lse and the top-k (ids, scores) of a logit row.  Lanes 0..k-1 of
// out_ids/out_lp receive candidates 0..k-1 (written by lane 0).
__device__ void head_topk_warp(const float* row, int V, int k, int* out_ids, float* out_lp, float* out_lse) {
    const int lane = threadIdx.x & 31;
    float v[VPL];
    float m = -INFINITY;
#pragma unroll
    for (int c = 0; c < VPL; ++c) {
        const int idx = lane + 32 * c;
        v[c] = idx < V ? row[idx] : -INFINITY;
        m = fmaxf(m, v[c]);
    }
    m = warp_max(m);
    float sum = 0.f;  // the fast exponential keeps this once-per-step code short (lse within ~1e-7)
#pragma unroll
    for (int c = 0; c < VPL; ++c)
        if (lane + 32 * c < V) sum += __expf(v[c] - m);
    sum = warp_sum(sum);
    const float lse = m + __logf(sum);
#pragma unroll
    for (int c = 0; c < VPL; ++c) v[c] = __fsub_rn(v[c], lse);  // -inf stays -inf
    uint64_t taken = 0;
    for (int r = 0; r < k; ++r) {
        float bv = -INFINITY;
        int bi = 0x7fffffff;
#pragma unroll
        for (int c = 0; c < VPL; ++c) {
            const int idx = lane + 32 * c;
            if (idx < V && !((taken >> c) & 1ull) && (v[c] > bv || bi == 0x7fffffff)) {
                bv = v[c];
                bi = idx;
            }
        }
        warp_argmax(bv, bi);
        if ((bi & 31) == lane) taken |= 1ull << (bi >> 5);
        if (lane == 0) {
            out_ids[r] = bi;
            out_lp[r] = bv;
        }
    }
    if (lane == 0 && out_lse) *out_lse = lse;
}

// Gather the transition scores the lattice uses, lq[t-1][i][j] = log_q[c_{t-1,i}][c_{t,j}]
// for t = 1..n-1, into shared memory with all threads of the group at once
// (one memory latency instead of one per recursion step).  Each pass covers
// nthreads / kp candidate rows i (kp = k rounded up to a power of two, lane
// j of a row slice = candidate j): no integer division per element.  Ids
// outside [0, V) get -inf (never read out of range).
__device__ __forceinline__ void gather_transitions(const int* ids, int n, int k, const float* log_q, int V,
                                                   float* lq, int tid, int nthreads) {
    int kp = 1;
    while (kp < k) kp <<= 1;
    const int sh = __ffs(kp) - 1;
    const int j = tid & (kp - 1), rows_per_pass = nthreads >> sh;
    const int kk = k * k;
    for (int t = 1; t < n; ++t) {
        const int* prev = ids + (t - 1) * k;
        const int cj = ids[t * k + min(j, k - 1)];
        float* out = lq + (size_t)(t - 1) * kk;
#pragma unroll 4
        for (int i = tid >> sh; i < k && j < k; i += rows_per_pass) {
            const int ci = prev[i];
            out[i * k + j] = (ci >= 0 && ci < V && cj >= 0 && cj < V) ? __ldg(log_q + (size_t)ci * V + cj) : -INFINITY;
        }
    }
}

// Viterbi over ids/lp [n][k] with transitions lq [n-1][k][k] and backpointers
// bp [MAX_NHEADS][32] (all shared memory); lane 0 writes the results.  The
// selection kernel runs it once per step with a cold instruction cache and
// keeps the loops rolled (its time follows the instructions it fetches).
__device__ void viterbi_warp(const int* ids, const float* lp, const float* lq, int n, int k, int* bp, int* path,
                               float* score) {
    const int lane = threadIdx.x & 31;
    const bool on = lane < k;
    float delta = on ? lp[lane] : -INFINITY;
#pragma unroll 1
    for (int t = 1; t < n; ++t) {
        const float* lqt = lq + (size_t)(t - 1) * k * k + (on ? lane : 0);
        float best = 0.f;
        int arg = 0;
#pragma unroll 1
        for (int i = 0; i < k; ++i) {
            const float di = __shfl_sync(FULL_MASK, delta, i);
            const float val = __fadd_rn(di, lqt[i * k]);
            if (i == 0 || val > best) {
                best = val;
                arg = i;
            }
        }
        delta = on ? __fadd_rn(best, lp[t * k + lane]) : -INFINITY;
        bp[t * 32 + lane] = arg;
    }
    float bv = delta;
    int bj = on ? lane : 0x7fffffff;
    warp_argmax(bv, bj);
    __syncwarp();
    if (lane == 0) {
        int state = bj;
#pragma unroll 1
        for (int t = n - 1; t >= 0; --t) {
            path[t] = ids[t * k + state];
            if (t > 0) state = bp[t * 32 + state];
        }
        *score = bv;
    }
}

constexpr int MS = MAX_NHEADS * MAX_TOPK;  // most states of a union lattice
constexpr int LQ_FLOATS = (MAX_NHEADS - 1) * MAX_TOPK * MAX_TOPK;  // select_kernel's scratch
static_assert((2 + MAX_NHEADS + 2 + MAX_NHEADS) * MS <= LQ_FLOATS, "union Viterbi scratch");
static_assert((2 + MAX_NHEADS + MAX_NHEADS + 1) * MS <= LQ_FLOATS, "union sampling scratch");

// Union lattice (reading B) of one sequence in `scratch` (>= 20 KB of shared
// memory): states [MS] (the distinct ids of all heads' top-k, ascending) and
// emissions em [MAX_NHEADS][MS] (head t's fp32 logp of every state; position 1
// forced to head 1's top-1 under VERIFY_GREEDY).  Returns the state count m.
__device__ int union_states(const SelectArgs& a, int bl, int n, int k, const int* s_ids, unsigned char* scratch) {
    int* states = reinterpret_cast<int*>(scratch);            // [MS]
    int* first = states + MS;                                 // [MS]
    float* em = reinterpret_cast<float*>(first + MS);         // [MAX_NHEADS][MS]
    __shared__ int s_m;
    const int tid = threadIdx.x, N = n * k;
    for (int t = tid; t < N; t += blockDim.x) {  // first occurrence of each id
        int f = 1;
        for (int j = 0; j < t; ++j)
            if (s_ids[j] == s_ids[t]) f = 0;
        first[t] = f;
    }
    __syncthreads();
    for (int t = tid; t < N; t += blockDim.x)
        if (first[t]) {  // rank among the distinct ids = its state index (ids ascending)
            int r = 0;
            for (int j = 0; j < N; ++j) r += first[j] && s_ids[j] < s_ids[t];
            states[r] = s_ids[t];
        }
    if (tid == 0) {
        int m = 0;
        for (int j = 0; j < N; ++j) m += first[j];
        s_m = m;
    }
    __syncthreads();
    const int m = s_m;
    for (int i = tid; i < n * m; i += blockDim.x) {  // emissions: logp of every state under every head
        const int t = i / m, r = i % m;
        const size_t row = (size_t)bl * n + t;
        float v = __fsub_rn(a.logits[row * a.V + states[r]], a.lse[row]);
        if (t == 0 && a.policy == 1 && states[r] != s_ids[0]) v = -INFINITY;  // VERIFY_GREEDY: forced
        em[t * MS + r] = v;
    }
    __syncthreads();
    return m;
}

// Viterbi (reading B) over the union lattice union_states built in `scratch`.
__device__ void union_viterbi(const SelectArgs& a, int n, int m, unsigned char* scratch, int* s_path) {
    const int* states = reinterpret_cast<const int*>(scratch);
    const float* em = reinterpret_cast<const float*>(states + 2 * MS);
    float* delta = const_cast<float*>(em) + MAX_NHEADS * MS;  // [2][MS]
    int* psi = reinterpret_cast<int*>(delta + 2 * MS);        // [MAX_NHEADS][MS]
    const int tid = threadIdx.x;
    for (int r = tid; r < m; r += blockDim.x) delta[r] = em[r];
    __syncthreads();
    for (int t = 1; t < n; ++t) {
        const float* prev = delta + ((t - 1) & 1) * MS;
        float* cur = delta + (t & 1) * MS;
        for (int r = tid; r < m; r += blockDim.x) {
            const float* lq_col = a.log_q + states[r];
            float best = -INFINITY;
            int arg = 0;
            for (int i = 0; i < m; ++i) {
                const float v = __fadd_rn(prev[i], lq_col[(size_t)states[i] * a.V]);
                if (v > best) {
                    best = v;
                    arg = i;
                }
            }
            cur[r] = __fadd_rn(best, em[t * MS + r]);
            psi[t * MS + r] = arg;
        }
        __syncthreads();
    }
    if (tid == 0) {
        const float* last = delta + ((n - 1) & 1) * MS;
        int r = 0;
        for (int i = 1; i < m; ++i)
            if (last[i] > last[r]) r = i;
        for (int t = n - 1; t >= 0; --t) {
            s_path[t] = states[r];
            if (t > 0) r = psi[t * MS + r];
        }
    }
}

// SplitMix64 (Steele, Lea, Flood 2014): the output function of a 64-bit counter.
__device__ __forceinline__ unsigned long long splitmix64(unsigned long long x) {
    unsigned long long z = x + 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

// The uniform of position t of one path draw: 24 bits of SplitMix64 of the
// counter ((seed * P + slot) * P + generated) * P + t, P = 0x100000001B3,
// so it is exact in fp32.
__device__ __forceinline__ float path_uniform(unsigned long long seed, int slot, int generated, int t) {
    constexpr unsigned long long P = 0x100000001B3ull;
    const unsigned long long x = ((seed * P + (unsigned long long)slot) * P + (unsigned long long)generated) * P +
                                 (unsigned long long)t;
    return (float)(splitmix64(x) >> 40) * (1.0f / 16777216.0f);
}

// Path sampling (top-k sampling, Fig. 2): one path of a lattice of S <= MS
// states per position (ids[t * ids_t + r], emissions em[t * em_t + r]) drawn
// from P(path) ~ prod_t Q(c_{t-1}, c_t) S_t(c_t).  Forward filtering, one
// thread per state: alpha_t(r) = logsumexp_i(alpha_{t-1}(i) + log Q) + s_t(r)
// (fp32, running-max form); backward sampling by warp 0: the last state from
// alpha_{n-1}, each earlier one from alpha_t(r) + log Q(c_{t,r}, next), by the
// first index whose inclusive prefix sum of exp(w - max) exceeds u * total
// (clamped to the last index of positive weight); gen = tokens the slot has
// generated.  alpha [MAX_NHEADS][MS] and cum [MS] are shared memory.
__device__ void sample_lattice(const SelectArgs& a, int b, int gen, const int* ids, int ids_t, const float* em,
                               int em_t, int S, int n, float* alpha, float* cum, int* s_path) {
    const int tid = threadIdx.x, lane = tid & 31;
    for (int r = tid; r < S; r += blockDim.x) alpha[r] = em[r];
    __syncthreads();
    for (int t = 1; t < n; ++t) {
        for (int r = tid; r < S; r += blockDim.x) {
            const float* lq_col = a.log_q + ids[t * ids_t + r];
            float mx = -INFINITY, sum = 0.f;
            for (int i = 0; i < S; ++i) {
                const float x = __fadd_rn(alpha[(t - 1) * MS + i], lq_col[(size_t)ids[(t - 1) * ids_t + i] * a.V]);
                if (x == -INFINITY) continue;
                if (x > mx) {
                    sum = sum * expf(mx - x) + 1.f;
                    mx = x;
                } else {
                    sum += expf(x - mx);
                }
            }
            alpha[t * MS + r] = mx == -INFINITY ? -INFINITY : __fadd_rn(__fadd_rn(mx, logf(sum)), em[t * em_t + r]);
        }
        __syncthreads();
    }
    if (tid >= 32) return;
    int next = -1;
    for (int t = n - 1; t >= 0; --t) {
        auto weight = [&](int r) {
            const float al = alpha[t * MS + r];
            return next < 0 ? al : __fadd_rn(al, a.log_q[(size_t)ids[t * ids_t + r] * a.V + next]);
        };
        float mx = -INFINITY;
        for (int r = lane; r < S; r += 32) mx = fmaxf(mx, weight(r));
        mx = warp_max(mx);
        float carry = 0.f;
        int last_pos = 0;
        for (int r0 = 0; r0 < S; r0 += 32) {
            const int r = r0 + lane;
            const float x = r < S ? weight(r) : -INFINITY;
            const float w = x == -INFINITY ? 0.f : expf(x - mx);
            float c = w;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const float y = __shfl_up_sync(FULL_MASK, c, o);
                if (lane >= o) c += y;
            }
            if (r < S) cum[r] = carry + c;
            carry += __shfl_sync(FULL_MASK, c, 31);
            const unsigned pos = __ballot_sync(FULL_MASK, w > 0.f);
            if (pos) last_pos = r0 + 31 - __clz(pos);
        }
        __syncwarp();
        const float target = path_uniform(a.seed, b, gen, t) * carry;
        int pick = -1;
        for (int r0 = 0; r0 < S && pick < 0; r0 += 32) {
            const int r = r0 + lane;
            const unsigned hit = __ballot_sync(FULL_MASK, r < S && cum[r] > target);
            if (hit) pick = r0 + __ffs(hit) - 1;
        }
        if (pick < 0 || pick > last_pos) pick = last_pos;
        next = ids[t * ids_t + pick];
        if (lane == 0) s_path[t] = next;
        __syncwarp();
    }
}

__global__ void __launch_bounds__(256) select_kernel(const SelectArgs a, int do_accept) {
    __shared__ int s_ids[MAX_NHEADS * MAX_TOPK];
    __shared__ float s_lp[MAX_NHEADS * MAX_TOPK];
    __shared__ float s_lq[LQ_FLOATS];
    __shared__ int s_path[MAX_NHEADS];
    __shared__ int s_bp[MAX_NHEADS * 32];
    __shared__ int s_emit[MAX_NHEADS + 1];
    __shared__ float s_score;
    const int bl = blockIdx.x, b = a.seq_base + bl;
    const int warp = threadIdx.x >> 5;
    const int n = a.n, k = a.k;
    __shared__ int s_st[6];  // active, done, remaining, generated, fed rows, cached length
    TraceEnd trace_guard(a.trace);
    pdl_launch_dependents();
    // The slot's state, read before the wait: the kernels of a step before
    // this one do not change it.
    if (do_accept && threadIdx.x < 6) {
        const int* src = threadIdx.x == 0 ? a.active : threadIdx.x == 1 ? a.done : threadIdx.x == 2 ? a.remaining
                         : threadIdx.x == 3 ? a.gen_count : threadIdx.x == 4 ? a.n_pending : a.seq_len;
        s_st[threadIdx.x] = src[b];
    }
    __syncthreads();
    pdl_wait();
    trace_wait(a.trace);
    // a slot still running its prompt (admitted, prefilled in the lane of the steps) selects nothing yet
    const bool prefilling = do_accept && a.prompt_left && (a.prompt_left[b] > 0 || (a.lane && a.lane_take[b] > 0));
    if (do_accept && (!s_st[0] || s_st[1] || prefilling)) {
        if (threadIdx.x < a.n_max) a.out_tokens[(size_t)b * a.n_max + threadIdx.x] = -1;
        if (threadIdx.x == 0) a.out_accepted[b] = 0;
        return;
    }
    if (a.pre_topk) {  // the heads kernel ranked them already
        for (int i = threadIdx.x; i < n * k; i += blockDim.x) {
            s_ids[i] = a.cand_ids[(size_t)bl * n * k + i];
            s_lp[i] = a.cand_logp[(size_t)bl * n * k + i];
        }
    } else if (warp < n) {
        const size_t row = (size_t)bl * n + warp;
        head_topk_warp(a.logits + row * a.V, a.V, k, s_ids + warp * k, s_lp + warp * k, a.lse + row);
    }
    __syncthreads();
    trace_mark(a.trace, 0);  // candidates
    if (do_accept && a.policy == 1 && threadIdx.x > 0 && threadIdx.x < k) s_lp[threadIdx.x] = -INFINITY;  // force
    __syncthreads();
    for (int i = threadIdx.x; i < n * k; i += blockDim.x) {
        a.cand_ids[(size_t)bl * n * k + i] = s_ids[i];
        a.cand_logp[(size_t)bl * n * k + i] = s_lp[i];
    }
    if (!do_accept) return;
    if (a.lattice == 1) {
        unsigned char* scratch = reinterpret_cast<unsigned char*>(s_lq);
        const int m = union_states(a, bl, n, k, s_ids, scratch);
        if (a.sampling) {
            const int* states = reinterpret_cast<const int*>(scratch);
            float* alpha = reinterpret_cast<float*>(scratch) + (2 + MAX_NHEADS) * MS;  // past states, first, em
            sample_lattice(a, b, s_st[3], states, 0, reinterpret_cast<const float*>(states + 2 * MS), MS, m, n, alpha,
                           alpha + MAX_NHEADS * MS, s_path);
        } else {
            union_viterbi(a, n, m, scratch, s_path);
        }
    } else if (a.sampling) {
        float* alpha = s_lq;
        sample_lattice(a, b, s_st[3], s_ids, k, s_lp, k, k, n, alpha, alpha + MAX_NHEADS * MS, s_path);
    } else {
        gather_transitions(s_ids, n, k, a.log_q, a.V, s_lq, threadIdx.x, blockDim.x);
        __syncthreads();
        if (warp == 0) viterbi_warp(s_ids, s_lp, s_lq, n, k, s_bp, s_path, &s_score);
    }
    __syncthreads();
    trace_mark(a.trace, 1);  // path
    if (warp != 0) return;

    // Acceptance and the slot's bookkeeping, one lane per token (short code:
    // see viterbi_warp).
    const int lane = threadIdx.x & 31;
    const int rem = s_st[2], gc = s_st[3];
    int n_emit;  // tokens this step emits (before the EOS / budget cut), s_emit
    if (a.policy == 1) {  // kept drafts, then head 1's argmax at the last kept row
        const int fed = s_st[4];
        const int kept = fed > 0 ? a.kept[b] : 0;
        if (lane < kept) s_emit[lane] = a.pending[(size_t)b * a.n_max + 1 + lane];
        if (lane == kept) s_emit[kept] = s_path[0];
        n_emit = kept + 1;
        if (lane == 0) a.seq_len[b] = s_st[5] + (fed > 0 ? kept + 1 : 0);  // confirmed token + kept drafts stay
    } else {
        if (lane < n) s_emit[lane] = s_path[lane];
        n_emit = n;
        if (lane == 0) a.seq_len[b] = s_st[5] + s_st[4];  // the tokens fed this step are now cached
    }
    __syncwarp();
    // ACCEPT_ALL on the emitted list: cut after the first EOS and at the budget
    const int e = lane < n_emit ? s_emit[lane] : -1;
    const unsigned eos_at = __ballot_sync(FULL_MASK, lane < n_emit && e == a.eos_id);
    int acc = eos_at ? __ffs(eos_at) : n_emit;
    acc = min(acc, max(rem, 0));
    const bool done = (eos_at != 0 && acc >= 1 && s_emit[acc - 1] == a.eos_id) || rem - acc <= 0;
    if (gc + acc > a.gen_stride) {
        if (lane == 0) atomicOr(a.err, ERR_BOUNDS);
        acc = max(0, a.gen_stride - gc);
    }
    const int n_next = a.policy == 1 ? n : acc;  // VERIFY_GREEDY feeds the path: confirmed token + drafts
    if (lane < a.n_max) a.out_tokens[(size_t)b * a.n_max + lane] = lane < acc ? e : -1;
    if (lane < n) a.path[(size_t)b * n + lane] = s_path[lane];
    if (lane < acc) a.gen_tokens[(size_t)b * a.gen_stride + gc + lane] = e;
    if (lane < n_next) a.pending[(size_t)b * a.n_max + lane] = s_path[lane];
    if (lane == 0) {
        a.gen_count[b] = gc + acc;
        a.remaining[b] = rem - acc;
        a.n_pending[b] = done ? 0 : n_next;
        a.done[b] = done;
        a.out_accepted[b] = acc;
    }
}

__global__ void __launch_bounds__(256) verify_kernel(const VerifyArgs a) {
    __shared__ int s_g[MAX_NHEADS];
    __shared__ float s_lp[MAX_NHEADS], s_lse[MAX_NHEADS];
    __shared__ int s_kept;
    const int bl = blockIdx.x, b = a.seq_base + bl;
    const int warp = threadIdx.x >> 5;
    TraceEnd trace_guard(a.trace);
    pdl_launch_dependents();
    pdl_wait();
    trace_wait(a.trace);
    if (!a.active[b] || a.done[b]) return;
    const int fed = a.n_pending[b];
    if (fed == 0) {  // first step after the prompt: h_last is the prompt's last row
        if (threadIdx.x == 0) a.kept[b] = 0;
        return;
    }
    if (warp < fed) head_topk_warp(a.logits1 + ((size_t)bl * a.n + warp) * a.V, a.V, 1, s_g + warp, s_lp + warp,
                                   s_lse + warp);
    __syncthreads();
    if (threadIdx.x == 0) {
        int kept = 0;
        while (kept < fed - 1 && a.pending[(size_t)b * a.n_max + kept + 1] == s_g[kept]) ++kept;
        s_kept = kept;
        a.kept[b] = kept;
    }
    __syncthreads();
    const float* src = a.x + ((size_t)bl * a.n + s_kept) * a.d;
    for (int i = threadIdx.x; i < a.d; i += blockDim.x) a.h_last[(size_t)b * a.d + i] = src[i];
}

// Stand-alone Viterbi: a group of KP lanes per lattice (KP = k rounded up to
// a power of two, 32 / KP lattices per warp), lane j = candidate j.  Each lane
// loads its own column of the transition scores, lq[i][j] = log_q[c_{t-1,i}][c_{t,j}]
// for every i, straight into registers: k independent L2 gathers per
// position, issued one position ahead of the recursion that consumes them, and
// no shared memory to limit how many warps an SM holds.  The ids of the
// previous position come from the group's lanes by shuffle.  The recursion,
// its add order and its tie rules are those of viterbi_warp; acceptance is
// the ACCEPT_ALL rule (cut after the first EOS and at the remaining budget).
constexpr int VIT_THREADS = 256;

template <int KP>
__device__ __forceinline__ void vit_load_column(const ViterbiArgs& a, int id_prev, int id_cur, bool on,
                                                float* q) {
    const int V = a.vocab;
    const bool cj_ok = on && id_cur >= 0 && id_cur < V;
#pragma unroll
    for (int i = 0; i < KP; ++i) {
        const int ci = __shfl_sync(FULL_MASK, id_prev, i, KP);
        q[i] = (cj_ok && i < a.k && ci >= 0 && ci < V) ? __ldg(a.log_q + (size_t)ci * V + id_cur) : -INFINITY;
    }
}

template <int KP>
__global__ void __launch_bounds__(VIT_THREADS, KP >= 32 ? 2 : 4) viterbi_kernel(const ViterbiArgs a) {
    constexpr int G = 32 / KP;  // lattices per warp
    const int lane = threadIdx.x & 31, j = lane & (KP - 1);
    const int b = (blockIdx.x * (VIT_THREADS / 32) + (threadIdx.x >> 5)) * G + lane / KP;
    const bool live = b < a.batch;  // the whole warp stays for the shuffles
    const int n = a.n, k = a.k;
    const bool on = live && j < k;
    int id[MAX_NHEADS];
    float lp[MAX_NHEADS];
#pragma unroll
    for (int t = 0; t < MAX_NHEADS; ++t) {
        id[t] = -1;
        lp[t] = -INFINITY;
        if (on && t < n) {
            id[t] = a.cand_ids[((size_t)b * n + t) * k + j];
            lp[t] = a.cand_logp[((size_t)b * n + t) * k + j];
        }
    }
    float qa[KP], qb[KP];
    int bp[MAX_NHEADS];
    if (n > 1) vit_load_column<KP>(a, id[0], id[1], on, qa);
    float delta = on ? lp[0] : -INFINITY;
#pragma unroll
    for (int t = 1; t < MAX_NHEADS; ++t) {
        bp[t] = 0;
        if (t < n) {
            float* cur = (t & 1) ? qa : qb;
            if (t + 1 < n) vit_load_column<KP>(a, id[t], id[t + 1], on, (t & 1) ? qb : qa);
            float best = 0.f;
            int arg = 0;
#pragma unroll
            for (int i = 0; i < KP; ++i) {
                const float di = __shfl_sync(FULL_MASK, delta, i, KP);
                if (i < k) {
                    const float val = __fadd_rn(di, cur[i]);
                    if (i == 0 || val > best) {
                        best = val;
                        arg = i;
                    }
                }
            }
            delta = on ? __fadd_rn(best, lp[t]) : -INFINITY;
            bp[t] = arg;
        }
    }
    // best final state: the lowest j of the maximum, within the group
    float bv = delta;
    int bj = on ? j : 0x7fffffff;
#pragma unroll
    for (int o = KP / 2; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(FULL_MASK, bv, o);
        const int oi = __shfl_xor_sync(FULL_MASK, bj, o);
        if (ov > bv || (ov == bv && oi < bj)) {
            bv = ov;
            bj = oi;
        }
    }
    int state = live ? bj : 0;
    int path[MAX_NHEADS];
#pragma unroll
    for (int t = MAX_NHEADS - 1; t >= 0; --t) {
        path[t] = -1;
        if (t < n) {
            path[t] = __shfl_sync(FULL_MASK, id[t], state, KP);
            if (t > 0) state = __shfl_sync(FULL_MASK, bp[t], state, KP);
        }
    }
    if (!live || j != 0) return;
    int acc = n;
    bool cut = false;
#pragma unroll
    for (int t = 0; t < MAX_NHEADS; ++t)
        if (t < n && !cut && path[t] == a.eos_id) {
            acc = t + 1;
            cut = true;
        }
    const int rem = a.remaining ? a.remaining[b] : n;
    acc = min(acc, max(rem, 0));
#pragma unroll
    for (int t = 0; t < MAX_NHEADS; ++t)
        if (t < n) a.path[(size_t)b * n + t] = path[t];
    if (a.score) a.score[b] = bv;
    a.accepted[b] = acc;
    if (a.rollback) a.rollback[b] = 0;
}

template <int KP>
cudaError_t launch_viterbi_kp(const ViterbiArgs& a, cudaStream_t s) {
    constexpr int per_block = VIT_THREADS / 32 * (32 / KP);
    viterbi_kernel<KP><<<(a.batch + per_block - 1) / per_block, VIT_THREADS, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_select(const SelectArgs& a, int batch, bool do_accept, cudaStream_t s, bool pdl) {
    if (a.n < 1 || a.n > MAX_NHEADS || a.k < 1 || a.k > MAX_TOPK || a.V > MAX_VOCAB || a.k > a.V)
        return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(batch);
    cfg.blockDim = dim3(256);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, select_kernel, a, do_accept ? 1 : 0);
}

cudaError_t launch_verify(const VerifyArgs& a, int slots, cudaStream_t s, bool pdl) {
    if (a.n < 1 || a.n > MAX_NHEADS || a.V > MAX_VOCAB || slots < 1) return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(slots);
    cfg.blockDim = dim3(256);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, verify_kernel, a);
}

cudaError_t launch_viterbi(const ViterbiArgs& a, cudaStream_t s) {
    if (a.n < 1 || a.n > MAX_NHEADS || a.k < 1 || a.k > MAX_TOPK || a.batch < 0) return cudaErrorInvalidValue;
    if (a.batch == 0) return cudaSuccess;
    if (a.k <= 1) return launch_viterbi_kp<1>(a, s);
    if (a.k <= 2) return launch_viterbi_kp<2>(a, s);
    if (a.k <= 4) return launch_viterbi_kp<4>(a, s);
    if (a.k <= 8) return launch_viterbi_kp<8>(a, s);
    if (a.k <= 16) return launch_viterbi_kp<16>(a, s);
    return launch_viterbi_kp<32>(a, s);
}

}  // namespace mtp
