"""Oracle: MTP heads, log-softmax, top-k and Viterbi selection (Sec. III-B, III-C).

Test infrastructure only (see oracle/__init__.py).

Heads (Sec. III-B): head i (1-based) maps the latent z of the last fed
position to the distribution of token t+i; z = LN_f(h).  Head 1 is the plain
next-token head, so n = 1 is ordinary greedy AR decoding.

Scores: logp = l - (m + log sum exp(l - m)), m = max l, in float64, then
rounded to float32; every decision below is taken on those float32 values.
Top-k order: logp descending, lower token id first on equal logp.

Viterbi (Sec. III-C; the printed algorithm is missing from the source, so this
follows the prose).  Token transitions form a first-order Markov chain with
matrix Q; head t gives the emission S_t; the step from a_i at t-1 to a_j at t
has weight Q(a_i, a_j) * S_t(a_j); the best sequence A* maximises the product.
In the log domain with delta_1(j) = s_1(j):
    delta_t(j) = max_i [ delta_{t-1}(i) + LQ(c_{t-1,i}, c_{t,j}) ] + s_t(j)
The inner sum is one float32 add, then the outer one; the backpointer is the
lowest i reaching the max; the final state is the lowest j reaching the max of
delta_n.  Position 1 carries no transition from the previously accepted token
(with it, n = 1 would no longer be greedy AR).
  * reading A (hot path): states at t are head t's own top-k candidates;
  * reading B (`viterbi_union`): states at every t are the m <= n*k distinct
    tokens of all heads' top-k (the reduced m x m matrix of Sec. III-C), each
    scored at t by head t's full log-softmax; states ordered by token id.

Acceptance (ACCEPT_ALL): the whole selected sequence is accepted, cut after
the first EOS and at the remaining budget (the paper accepts every selected
token; its speed-up scales with n).

Parity pins (tests/test_oracle_select.py): brute-force enumeration of all
k^n paths, scored left to right with the same float32 adds (bit-exact), hand-worked lattices
in tests/golden/, k = 1 and uniform-Q reductions to per-head argmax, the
sticky-diagonal case, sum(exp(logp)) = 1, shift invariance, and top-k against
a stable lexicographic sort.  head_logits (tests/test_oracle_heads_embed.py):
the closed form of LN_f on an alternating hidden state through heads whose
rows select one coordinate each, with planted mistakes (LN_f or its affine
part skipped, head i reading head i + 1, bias dropped) rejected.
"""
from __future__ import annotations

import numpy as np

from .model import layer_norm


def head_logits(h_last: np.ndarray, w: dict[str, np.ndarray], n: int, eps: float) -> np.ndarray:
    """Logits [n, V] of the first n heads on z = LN_f(h_last) (float64)."""
    z = layer_norm(np.asarray(h_last, dtype=np.float64), w["lnf_g"], w["lnf_b"], eps)
    return np.stack([w["w_heads"][i] @ z + w["b_heads"][i] for i in range(n)])


def log_softmax(logits: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """(logp, lse) over the last axis in float64: logp = l - lse, lse = m + log sum exp(l - m)."""
    m = logits.max(axis=-1, keepdims=True)
    lse = m + np.log(np.exp(logits - m).sum(axis=-1, keepdims=True))
    return logits - lse, lse[..., 0]


def top_k(logp32: np.ndarray, k: int) -> tuple[np.ndarray, np.ndarray]:
    """The k best (id, score) of one float32 score row, by a plain selection loop.

    Order: score descending; among equal scores the lower id first."""
    scores = np.asarray(logp32, dtype=np.float32)
    taken = np.zeros(scores.shape[0], dtype=bool)
    ids, vals = [], []
    for _ in range(k):
        best = -1
        for a in range(scores.shape[0]):
            if taken[a]:
                continue
            if best < 0 or scores[a] > scores[best]:
                best = a
        taken[best] = True
        ids.append(best)
        vals.append(scores[best])
    return np.array(ids, dtype=np.int32), np.array(vals, dtype=np.float32)


def top_k_rows(logp32: np.ndarray, k: int) -> tuple[np.ndarray, np.ndarray]:
    """top_k over each row of a [..., V] array, vectorised over the leading axes.

    Same selection loop as top_k: at each round take the highest remaining
    score, the lowest id among equals (argmax returns the first maximum)."""
    s = np.array(logp32, dtype=np.float32, copy=True)
    lead = s.shape[:-1]
    flat = s.reshape(-1, s.shape[-1])
    ids = np.zeros((flat.shape[0], k), dtype=np.int32)
    vals = np.zeros((flat.shape[0], k), dtype=np.float32)
    rows = np.arange(flat.shape[0])
    for r in range(k):
        best = np.argmax(flat, axis=1)
        ids[:, r] = best
        vals[:, r] = flat[rows, best]
        flat[rows, best] = -np.inf
    return ids.reshape(lead + (k,)), vals.reshape(lead + (k,))


def viterbi(cand_ids: np.ndarray, cand_logp: np.ndarray, log_q: np.ndarray):
    """Reading A over a batch: ids/logp [B, n, k] -> (path ids [B, n], state idx [B, n], score [B]).

    Loops follow the recursion; each loop body is vectorised over the batch."""
    cand_ids = np.asarray(cand_ids)
    s = np.asarray(cand_logp, dtype=np.float32)
    lq = np.asarray(log_q, dtype=np.float32)
    batch, n, k = s.shape
    delta = s[:, 0, :].copy()
    back = np.zeros((batch, n, k), dtype=np.int32)
    for t in range(1, n):
        new = np.empty_like(delta)
        for j in range(k):
            best = None
            arg = np.zeros(batch, dtype=np.int32)
            for i in range(k):
                val = delta[:, i] + lq[cand_ids[:, t - 1, i], cand_ids[:, t, j]]
                if best is None:
                    best = val
                else:
                    better = val > best
                    best = np.where(better, val, best)
                    arg = np.where(better, np.int32(i), arg)
            new[:, j] = best + s[:, t, j]
            back[:, t, j] = arg
        delta = new
    state = np.zeros((batch, n), dtype=np.int32)
    last = np.zeros(batch, dtype=np.int32)
    score = delta[:, 0].copy()
    for j in range(1, k):
        better = delta[:, j] > score
        score = np.where(better, delta[:, j], score)
        last = np.where(better, np.int32(j), last)
    state[:, n - 1] = last
    for t in range(n - 1, 0, -1):
        state[:, t - 1] = back[np.arange(batch), t, state[:, t]]
    path = np.take_along_axis(cand_ids, state[:, :, None], axis=2)[:, :, 0].astype(np.int32)
    return path, state, score.astype(np.float32)


def viterbi_union(topk_ids: np.ndarray, logp32_full: np.ndarray, log_q: np.ndarray):
    """Reading B for one sequence: states = sorted distinct tokens of all heads' top-k.

    topk_ids [n, k], logp32_full [n, V] (float32 log-softmax of every head).
    Returns (path ids [n], score)."""
    states = np.unique(np.asarray(topk_ids).reshape(-1))
    n = logp32_full.shape[0]
    ids = np.broadcast_to(states, (n, states.shape[0]))[None]
    scores = np.asarray(logp32_full, dtype=np.float32)[:, states][None]
    path, _, score = viterbi(ids, scores, log_q)
    return path[0], score[0]


def viterbi_margin(cand_ids: np.ndarray, cand_logp: np.ndarray, log_q: np.ndarray) -> np.ndarray:
    """Gap [B] between the best path and the best path that differs anywhere.

    Max-marginals in float64: M(t, j) = forward(t, j) + backward(t, j); the
    runner-up is the best M over states off the best path.  Infinite when
    every position has a single candidate."""
    ids = np.asarray(cand_ids)
    s = np.asarray(cand_logp, dtype=np.float64)
    lq = np.asarray(log_q, dtype=np.float64)
    batch, n, k = s.shape
    if k == 1:
        return np.full(batch, np.inf)
    fwd = np.zeros((batch, n, k))
    bwd = np.zeros((batch, n, k))
    fwd[:, 0] = s[:, 0]
    for t in range(1, n):
        trans = lq[ids[:, t - 1, :, None], ids[:, t, None, :]]        # [B, k_prev, k]
        fwd[:, t] = (fwd[:, t - 1, :, None] + trans).max(axis=1) + s[:, t]
    for t in range(n - 2, -1, -1):
        trans = lq[ids[:, t, :, None], ids[:, t + 1, None, :]]        # [B, k, k_next]
        bwd[:, t] = (trans + s[:, t + 1, None, :] + bwd[:, t + 1, None, :]).max(axis=2)
    marg = fwd + bwd
    best = marg[:, n - 1].max(axis=1)
    _, state, _ = viterbi(ids, s.astype(np.float32), log_q)
    off = marg.copy()
    off[np.arange(batch)[:, None], np.arange(n)[None, :], state] = -np.inf
    return best - off.reshape(batch, -1).max(axis=1)


def topk_gap(logp32: np.ndarray, k: int) -> np.ndarray:
    """Gap between the k-th and (k+1)-th best float32 score of each row (inf if k = V)."""
    s = -np.sort(-np.asarray(logp32, dtype=np.float64), axis=-1)
    if k >= s.shape[-1]:
        return np.full(s.shape[:-1], np.inf)
    return s[..., k - 1] - s[..., k]


def accept_all(path: np.ndarray, eos_id: int, remaining: int) -> tuple[int, bool]:
    """Accepted count and done flag: cut after the first EOS and at the budget."""
    n = len(path)
    a = n
    hits = np.nonzero(np.asarray(path) == eos_id)[0]
    if hits.size:
        a = int(hits[0]) + 1
    a = min(a, remaining)
    done = bool(hits.size and hits[0] < a) or remaining - a <= 0
    return a, done


# ---- path sampling (top-k sampling over the lattice, the diversity option of Fig. 2) ----
_M64 = (1 << 64) - 1


def splitmix64(x: int) -> int:
    """SplitMix64 output function (Steele, Lea, Flood 2014) of a 64-bit counter."""
    z = (x + 0x9E3779B97F4A7C15) & _M64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _M64
    return z ^ (z >> 31)


def path_uniform(seed: int, slot: int, generated: int, t: int) -> float:
    """The uniform in [0, 1) (24 bits) drawn for position t of a sampling step of
    `slot` when it has generated `generated` tokens: SplitMix64 of the counter
    ((seed * P + slot) * P + generated) * P + t, P = 0x100000001B3, top 24 bits."""
    p = 0x100000001B3
    x = (((((seed & _M64) * p + slot) & _M64) * p + generated) & _M64) * p + t
    return (splitmix64(x & _M64) >> 40) * (1.0 / (1 << 24))


def _categorical(logw: np.ndarray, u: float) -> tuple[int, float]:
    """(index, margin) of one draw with probabilities proportional to exp(logw):
    the first index whose cumulative weight (index order, float64) exceeds
    u times the total, clamped to the last index of positive weight.  margin
    is the distance of u * total from the nearest boundary that separates the
    drawn index from another index of positive weight, over the total (1 when
    only one index has positive weight)."""
    m = logw.max()
    w = np.where(np.isfinite(logw), np.exp(logw - m), 0.0)
    c = np.cumsum(w)
    total = c[-1]
    target = u * total
    pos = np.flatnonzero(w > 0)
    i = int(np.searchsorted(c, target, side="right"))
    i = min(i, int(pos[-1]))
    margin = 1.0
    if pos[0] < i:       # a positive-weight index below: the lower boundary counts
        margin = min(margin, (target - (c[i - 1] if i > 0 else 0.0)) / total)
    if pos[-1] > i:      # one above: the upper boundary counts
        margin = min(margin, (c[i] - target) / total)
    return i, max(margin, 0.0)


def sample_path(cand_ids: np.ndarray, cand_logp: np.ndarray, log_q: np.ndarray, uniforms):
    """(path [n], margin) of one lattice drawn from P(path) proportional to
    prod_t Q(c_{t-1}, c_t) S_t(c_t) (the quantity Viterbi maximises), by forward
    filtering (log-sum-exp, float64) and backward sampling: the last state with
    uniforms[n-1], then each earlier state given its successor with uniforms[t].
    margin: the smallest draw margin (see _categorical) along the way."""
    ids = np.asarray(cand_ids)
    s = np.asarray(cand_logp, dtype=np.float64)
    lq = np.asarray(log_q, dtype=np.float64)
    n, k = s.shape
    alpha = np.zeros((n, k))
    alpha[0] = s[0]
    for t in range(1, n):
        x = alpha[t - 1][:, None] + lq[ids[t - 1][:, None], ids[t][None, :]]   # [k_prev, k]
        mx = x.max(axis=0)
        safe = np.where(np.isfinite(mx), mx, 0.0)
        with np.errstate(divide="ignore"):
            lse = np.where(np.isfinite(mx), safe + np.log(np.exp(x - safe).sum(axis=0)), -np.inf)
        alpha[t] = lse + s[t]
    state = np.zeros(n, dtype=np.int64)
    state[n - 1], margin = _categorical(alpha[n - 1], uniforms[n - 1])
    for t in range(n - 2, -1, -1):
        state[t], mg = _categorical(alpha[t] + lq[ids[t], ids[t + 1][state[t + 1]]], uniforms[t])
        margin = min(margin, mg)
    return ids[np.arange(n), state].astype(np.int32), float(margin)


def sample_path_union(cand_ids: np.ndarray, logp32: np.ndarray, log_q: np.ndarray, uniforms):
    """sample_path over the union lattice (reading B): the states of every
    position are the distinct ids of all heads' top-k, ascending, each scored
    at position t by head t's float32 log-softmax."""
    states = np.unique(np.asarray(cand_ids).reshape(-1))
    n = logp32.shape[0]
    return sample_path(np.tile(states, (n, 1)), np.asarray(logp32)[:, states], log_q, uniforms)
