"""Pins of the oracle's VERIFY_GREEDY policy (speculative decoding with the
MTP heads as drafter): its output must equal plain greedy AR decoding token
for token, whatever n and k; the bookkeeping must hold."""
import numpy as np
import pytest

import synth
from oracle.mtp import MTPOracle
from oracle.select import head_logits, log_softmax


def _greedy(model, w, ph, ac, budget):
    """Plain greedy AR written from the definition: argmax of head 1 (float32 scores, lowest id)."""
    o = MTPOracle(model, w)
    o.prefill(ph, ac, budget)
    out = []
    while len(out) < budget:
        lp = log_softmax(head_logits(o.h_last, o.w, 1, model.ln_eps))[0].astype(np.float32)[0]
        t = int(np.flatnonzero(lp == lp.max())[0])
        out.append(t)
        if t == model.eos_id:
            break
        o.feed([t])
    return out


@pytest.fixture(scope="module")
def tiny():
    w = synth.make_weights(synth.TINY)
    ph, ac = synth.make_prompt(3, 12, 30, synth.TINY.phone_vocab)
    return w, ph, ac


@pytest.mark.parametrize("n,k", [(1, 1), (2, 3), (4, 4), (6, 2)])
def test_verify_greedy_equals_greedy_ar(tiny, n, k):
    w, ph, ac = tiny
    budget = 40
    ref = _greedy(synth.TINY, w, ph, ac, budget)
    o = MTPOracle(synth.TINY, w)
    o.prefill(ph, ac, budget)
    recs = o.generate_verify(n, k)
    assert o.generated == ref
    assert sum(len(r.emitted) for r in recs) == len(ref)


def test_verify_bookkeeping(tiny):
    w, ph, ac = tiny
    o = MTPOracle(synth.TINY, w)
    o.prefill(ph, ac, 50)
    T = len(ph) + len(ac)
    emitted = 0
    steps = 0
    while not o.done:
        r = o.step_verify(4, 4)
        steps += 1
        m = max(0, len(r.fed) - 1)
        assert 0 <= r.kept <= m and r.rollback == m - r.kept
        assert len(r.emitted) <= r.kept + 1
        assert np.all(r.greedy[:r.kept] == r.fed[1:r.kept + 1])     # kept drafts are the greedy tokens
        if r.kept < m:
            assert r.greedy[r.kept] != r.fed[r.kept + 1]              # the first rejected draft is not
        assert r.path[0] == r.cand_ids[0, 0]                           # position 1 forced to its top-1
        emitted += len(r.emitted)
        if not r.done:
            # every emitted token but the last (the next confirmed token, fed next step) is cached
            assert o.cache.length == T + emitted - 1
    # random-init heads rarely propose the greedy continuation (about 1 in V per draft),
    # so about one token per step is expected here; the perfect-drafter test covers keeping
    assert emitted == 50 and steps <= 50


def test_verify_with_a_perfect_drafter_keeps_every_draft(tiny):
    """Drafts equal to the greedy continuation are all kept: feed the greedy tokens as drafts."""
    w, ph, ac = tiny
    ref = _greedy(synth.TINY, w, ph, ac, 30)
    o = MTPOracle(synth.TINY, w)
    o.prefill(ph, ac, 30)
    o.step_verify(4, 4)                      # emits ref[0]
    o.pending = np.asarray(ref[0:4], np.int32)  # c = ref[0], drafts = ref[1:4]
    r = o.step_verify(4, 4)
    assert r.kept == 3 and r.rollback == 0
    assert list(r.emitted) == ref[1:5]


@pytest.mark.parametrize("n,k", [(4, 4), (6, 3)])
def test_verify_with_sampled_drafts_is_still_greedy(tiny, n, k):
    """Drawn drafts (path sampling) change which drafts are kept, never the output."""
    w, ph, ac = tiny
    budget = 40
    ref = _greedy(synth.TINY, w, ph, ac, budget)
    o = MTPOracle(synth.TINY, w)
    o.prefill(ph, ac, budget)
    while not o.done:
        o.step_verify(n, k, sample=(12345, 0))
    assert o.generated == ref
