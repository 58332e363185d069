"""Oracle: the multi-token inference loop (Fig. 1 caption, Sec. III-B, III-C).

Test infrastructure only (see oracle/__init__.py).

One sequence.  Prefill runs the prompt [phonemes ; acoustic codes] through the
decoder and keeps the hidden state of its last position.  Each step then
  1. feeds the tokens accepted by the previous step (none on the first step)
     through the decoder, appending their keys/values to the cache;
  2. applies the first n heads to LN_f of the last fed position's hidden state;
  3. takes each head's top-k as the candidates of its position and selects the
     path with Viterbi (reading A, select.viterbi);
  4. accepts the path under ACCEPT_ALL (select.accept_all); the accepted
     tokens are output and become the next step's fed tokens.
Each step selects min(n, remaining) tokens unless EOS ends the sequence, so
the number of steps is ceil(budget / n) -- the O(L/n + alpha) of Sec. III-B.

Parity pins (tests/test_oracle_mtp.py): n = 1 equals a plain greedy AR loop
written separately, token for token; the first i heads at n = N give the same
distributions as a run at n = i; the KV cache equals a cache-free recompute;
append-rollback-append equals append.

VERIFY_GREEDY (policy 1; speculative decoding with the heads as drafter,
the paper's "speculative decoding" framing, Sec. I, II): each step feeds the
confirmed token c and the drafts d_1..d_m proposed by the previous step.
Head 1's argmax g_j at fed row j (c for j = 0, d_j after) is the greedy
token after that row, so the drafts are kept while d_{j+1} = g_j; with a kept
drafts, the other m - a cache rows are rolled back and the step emits
d_1..d_a and then g_a.  The next drafts are the Viterbi path over the heads
at the last kept row with position 1 forced to g_a (its top-1 candidate), so
c' = g_a and d'_t = path[t].  The emitted sequence is the greedy AR
sequence for every n and k (pinned in tests/test_oracle_verify.py).

Path sampling (sample = (seed, slot); the top-k sampling of the Fig. 2
caption): step 3 draws the path from the lattice's posterior instead of
taking its maximum (select.sample_path), with the uniforms of
select.path_uniform(seed, slot, tokens generated so far, position).  Under
VERIFY_GREEDY only the drafts are drawn (position 1 stays forced), so the
emitted sequence is still the greedy one.
"""
from __future__ import annotations

import dataclasses

import numpy as np

from .model import ARDecoder
from .select import (accept_all, head_logits, log_softmax, path_uniform, sample_path, sample_path_union,
                     top_k_rows, topk_gap, viterbi, viterbi_margin, viterbi_union)


@dataclasses.dataclass
class StepRecord:
    """Everything one step decided, for comparison with the CUDA path."""
    fed: np.ndarray          # tokens fed this step (int32)
    logits: np.ndarray       # [n, V] float64
    lse: np.ndarray          # [n] float64
    logp32: np.ndarray       # [n, V] float32 scores the decisions use
    cand_ids: np.ndarray     # [n, k] int32
    cand_logp: np.ndarray    # [n, k] float32
    path: np.ndarray         # [n] int32
    accepted: int
    done: bool
    margin: float            # min(top-k gap over heads, Viterbi runner-up gap)


@dataclasses.dataclass
class VerifyRecord:
    """One VERIFY_GREEDY step."""
    fed: np.ndarray          # [c, d_1..d_m] (empty on the first step)
    greedy: np.ndarray       # head 1's argmax at every fed row (float32 scores)
    kept: int                # drafts kept (a)
    rollback: int            # cache rows rolled back (m - a)
    emitted: np.ndarray      # d_1..d_a, g_a (cut at EOS / budget)
    logits: np.ndarray       # [n, V] float64 heads at the last kept row
    lse: np.ndarray
    logp32: np.ndarray
    cand_ids: np.ndarray     # [n, k]
    cand_logp: np.ndarray    # [n, k], position 1 forced to its top-1
    path: np.ndarray         # [n]: next step's confirmed token and drafts
    done: bool


class MTPOracle:
    def __init__(self, cfg, weights: dict[str, np.ndarray]):
        self.cfg = cfg
        self.model = ARDecoder(cfg, weights)
        self.w = self.model.w
        self.log_q = np.asarray(weights["log_q"], dtype=np.float32)

    def prefill(self, phonemes, acoustic, max_new: int) -> None:
        ph = np.asarray(phonemes, dtype=np.int64)
        ac = np.asarray(acoustic, dtype=np.int64)
        self.cache = self.model.new_cache()
        tokens = np.concatenate([ph, ac])
        is_phone = np.concatenate([np.ones(ph.shape[0], bool), np.zeros(ac.shape[0], bool)])
        self.h_last = self.model.forward(tokens, is_phone, self.cache)[-1]
        self.pending = np.zeros(0, dtype=np.int32)
        self.remaining = int(max_new)
        self.generated: list[int] = []
        self.done = False

    def feed(self, tokens) -> None:
        """Run fed codec tokens through the decoder (extends the cache, moves h_last)."""
        tokens = np.asarray(tokens, dtype=np.int64)
        if tokens.shape[0]:
            h = self.model.forward(tokens, np.zeros(tokens.shape[0], bool), self.cache)
            self.h_last = h[-1]

    def uniforms(self, sample, n: int) -> list[float]:
        """The n uniforms of this step's path draw: sample = (seed, slot), the
        counter also holds the number of tokens generated so far."""
        seed, slot = sample
        return [path_uniform(seed, slot, len(self.generated), t) for t in range(n)]

    def select(self, n: int, k: int, lattice: str = "A", sample=None):
        """Heads, log-softmax, top-k and Viterbi on the current h_last.

        lattice "A": each position's states are its own head's top-k; "B": the
        union of all heads' top-k at every position (select.viterbi_union).
        sample = (seed, slot): draw the path from the lattice's posterior
        (select.sample_path) instead of taking its maximum; margin is then the
        smallest draw margin."""
        logits = head_logits(self.h_last, self.w, n, self.cfg.ln_eps)
        logp, lse = log_softmax(logits)
        logp32 = logp.astype(np.float32)
        ids, vals = top_k_rows(logp32, k)
        if sample is not None:
            u = self.uniforms(sample, n)
            if lattice == "B":
                path, margin = sample_path_union(ids, logp32, self.log_q, u)
            else:
                path, margin = sample_path(ids, vals, self.log_q, u)
            return logits, lse, logp32, ids, vals, path, min(margin, float(topk_gap(logp32, k).min()))
        if lattice == "B":
            path, _ = viterbi_union(ids, logp32, self.log_q)
            margin = float(topk_gap(logp32, k).min())
            return logits, lse, logp32, ids, vals, path, margin
        path, _, _ = viterbi(ids[None], vals[None], self.log_q)
        margin = min(float(topk_gap(logp32, k).min()),
                     float(viterbi_margin(ids[None], vals[None], self.log_q)[0]))
        return logits, lse, logp32, ids, vals, path[0], margin

    def step(self, n: int, k: int, teacher=None, lattice: str = "A", sample=None) -> StepRecord:
        """One decode step; `teacher` overrides the fed tokens (teacher forcing)."""
        fed = self.pending if teacher is None else np.asarray(teacher, dtype=np.int32)
        self.feed(fed)
        logits, lse, logp32, ids, vals, path, margin = self.select(n, k, lattice, sample)
        a, done = accept_all(path, self.cfg.eos_id, self.remaining)
        self.pending = path[:a].astype(np.int32)
        self.generated.extend(int(t) for t in self.pending)
        self.remaining -= a
        self.done = done
        return StepRecord(np.asarray(fed, np.int32), logits, lse, logp32, ids, vals, path,
                          a, done, margin)

    # ---- VERIFY_GREEDY ----
    def propose(self, n: int, k: int, sample=None):
        """Heads at h_last with position 1 forced to head 1's top-1 (the greedy token);
        the drafts are the Viterbi path, or a drawn path with sample = (seed, slot)."""
        logits = head_logits(self.h_last, self.w, n, self.cfg.ln_eps)
        logp, lse = log_softmax(logits)
        logp32 = logp.astype(np.float32)
        ids, vals = top_k_rows(logp32, k)
        vals = vals.copy()
        vals[0, 1:] = -np.inf  # position 1: the greedy token only
        if sample is not None:
            path, self.last_margin = sample_path(ids, vals, self.log_q, self.uniforms(sample, n))
            return logits, lse, logp32, ids, vals, path
        path, _, _ = viterbi(ids[None], vals[None], self.log_q)
        return logits, lse, logp32, ids, vals, path[0]

    def step_verify(self, n: int, k: int, sample=None) -> "VerifyRecord":
        """One VERIFY_GREEDY step (see the module docstring)."""
        fed = self.pending
        m = max(0, len(fed) - 1)  # drafts fed
        g = np.zeros(0, np.int32)
        if len(fed):
            h = self.model.forward(np.asarray(fed, np.int64), np.zeros(len(fed), bool), self.cache)
            l1 = np.stack([head_logits(h[j], self.w, 1, self.cfg.ln_eps)[0] for j in range(len(fed))])  # head 1
            lp1 = log_softmax(l1)[0].astype(np.float32)
            g = np.array([top_k_rows(lp1[j:j + 1], 1)[0][0, 0] for j in range(len(fed))], np.int32)
            a = 0
            while a < m and int(fed[a + 1]) == int(g[a]):
                a += 1
            self.cache.rollback(m - a)
            self.h_last = h[a]
        else:
            a = 0
        logits, lse, logp32, ids, vals, path = self.propose(n, k, sample)
        emit = [int(t) for t in fed[1:a + 1]] + [int(path[0])]
        e, done = accept_all(np.asarray(emit, np.int32), self.cfg.eos_id, self.remaining)
        emitted = np.asarray(emit[:e], np.int32)
        self.generated.extend(int(t) for t in emitted)
        self.remaining -= e
        self.done = done
        self.pending = np.zeros(0, np.int32) if done else path.astype(np.int32)
        return VerifyRecord(np.asarray(fed, np.int32), g, a, m - a, emitted, logits, lse, logp32, ids, vals,
                            path, done)

    def generate_verify(self, n: int, k: int, max_steps: int | None = None) -> list["VerifyRecord"]:
        records = []
        while not self.done and (max_steps is None or len(records) < max_steps):
            records.append(self.step_verify(n, k))
        return records

    def generate(self, n: int, k: int, max_steps: int | None = None) -> list[StepRecord]:
        records = []
        while not self.done and (max_steps is None or len(records) < max_steps):
            records.append(self.step(n, k))
        return records
