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
"""
from __future__ import annotations

import dataclasses

import numpy as np

from .model import ARDecoder
from .select import (accept_all, head_logits, log_softmax, top_k_rows, topk_gap,
                     viterbi, viterbi_margin)


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

    def select(self, n: int, k: int):
        """Heads, log-softmax, top-k and Viterbi on the current h_last."""
        logits = head_logits(self.h_last, self.w, n, self.cfg.ln_eps)
        logp, lse = log_softmax(logits)
        logp32 = logp.astype(np.float32)
        ids, vals = top_k_rows(logp32, k)
        path, _, _ = viterbi(ids[None], vals[None], self.log_q)
        margin = min(float(topk_gap(logp32, k).min()),
                     float(viterbi_margin(ids[None], vals[None], self.log_q)[0]))
        return logits, lse, logp32, ids, vals, path[0], margin

    def step(self, n: int, k: int, teacher=None) -> StepRecord:
        """One decode step; `teacher` overrides the fed tokens (teacher forcing)."""
        fed = self.pending if teacher is None else np.asarray(teacher, dtype=np.int32)
        self.feed(fed)
        logits, lse, logp32, ids, vals, path, margin = self.select(n, k)
        a, done = accept_all(path, self.cfg.eos_id, self.remaining)
        self.pending = path[:a].astype(np.int32)
        self.generated.extend(int(t) for t in self.pending)
        self.remaining -= a
        self.done = done
        return StepRecord(np.asarray(fed, np.int32), logits, lse, logp32, ids, vals, path,
                          a, done, margin)

    def generate(self, n: int, k: int, max_steps: int | None = None) -> list[StepRecord]:
        records = []
        while not self.done and (max_steps is None or len(records) < max_steps):
            records.append(self.step(n, k))
        return records
