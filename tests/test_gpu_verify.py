"""VERIFY_GREEDY on the GPU (speculative decoding with the heads as drafter).

Teacher-forced (the main parity tests): every step both the GPU and the
oracle are fed the same confirmed token and drafts, built from the oracle's
greedy continuation so that the number of drafts that must be kept is known
in advance: j correct drafts, then a draft that is the lowest-scored token of
head 1 at that row (never the greedy token on either side).  j cycles over
0..n-1 and is cut at the first row whose greedy decision is a near-tie
(oracle top-1 margin <= 5e-2), so that every kept/rejected decision is one
both sides must take alike.  Per step and slot: the oracle keeps j drafts
and rolls back n-1-j rows; the GPU accepts j + 1 tokens, emits the j drafts
and the greedy token after them (compared where its margin is clear), its
cached length equals the oracle's, and the heads' logits at the last kept
row are within the bf16 bar of the oracle's.

Free-running: mtp_generate's emitted sequence equals the oracle's greedy AR
sequence up to the first near-tie, with a minimum compared length asserted.
"""
import copy

import numpy as np
import pytest

import synth
from oracle.mtp import MTPOracle
from oracle.select import head_logits, log_softmax

from gpu_util import MARGIN, assert_logits_close, decoder, lib_module

pytestmark = pytest.mark.gpu


def greedy_trace(o, budget, eos_id):
    """From the oracle's current state (left untouched): greedy tokens, the
    float32 top-1 margin of each decision and head 1's lowest-scored token at
    each decision."""
    o = copy.copy(o)
    o.cache = copy.deepcopy(o.cache)
    toks, margins, worst = [], [], []
    while len(toks) < budget:
        lp = log_softmax(head_logits(o.h_last, o.w, 1, o.cfg.ln_eps))[0].astype(np.float32)[0]
        order = np.lexsort((np.arange(lp.shape[0]), -lp))
        toks.append(int(order[0]))
        margins.append(float(lp[order[0]] - lp[order[1]]))
        worst.append(int(order[-1]))
        if toks[-1] == eos_id:
            break
        o.feed([toks[-1]])
    return toks, margins, worst


def _prompts(model, batch, seed0):
    return [synth.make_prompt(seed0 + b, 10 + 3 * b, 30 + 5 * b, model.phone_vocab) for b in range(batch)]


def _teacher_forced_verify(model, batch, n, k, tokens, seed0, batched=1):
    """Teacher-forced VERIFY_GREEDY run of about `tokens` emitted tokens per slot."""
    mtp = lib_module()
    m = n - 1
    prompts = _prompts(model, batch, seed0)
    budget = tokens + 2 * n
    max_ctx = max(len(p) + len(a) for p, a in prompts) + budget + model.n_heads_max + 4
    dec, w = decoder(model, max_batch=batch, max_ctx=max_ctx, accept_policy=1)
    kept_seen = set()
    compared_tokens = 0
    try:
        mtp.mtp_set_option(dec.ctx, 4, batched)
        oracles, plans = [], []
        for b, (ph, ac) in enumerate(prompts):
            dec.prefill(b, ph, ac, budget)
            o = MTPOracle(model, w) if b == 0 else copy.copy(oracles[0])
            o.prefill(ph, ac, budget)
            oracles.append(o)
            plans.append(greedy_trace(o, budget, model.eos_id))
        pos = [0] * batch  # greedy tokens emitted so far per slot
        step = 0
        while True:
            feds, js = [], []
            for b in range(batch):
                G, margins, worst = plans[b]
                if step == 0:
                    feds.append(None)
                    js.append(0)
                    continue
                p = pos[b]
                if p + n >= len(G):
                    feds.append(None)
                    js.append(None)
                    continue
                j = (step * 3 + b) % (m + 1)
                for r in range(j):  # draft r + 1 is kept only where row r's greedy decision is clear
                    if margins[p + r] <= MARGIN:
                        j = r
                        break
                drafts = G[p:p + j] + [worst[p + j]] * (m - j)
                feds.append(np.asarray([G[p - 1]] + drafts, np.int32))
                js.append(j)
            if step > 0 and all(j is None for j in js):
                break
            for b in range(batch):
                if feds[b] is not None:
                    mtp.mtp_set_teacher_tokens(dec.ctx, b, feds[b])
            toks, acc, _ = dec.decode_step(n, k)
            lg, _ = dec.logits(n)
            for b in range(batch):
                j = js[b]
                if j is None:
                    continue
                G, margins, _ = plans[b]
                o, p = oracles[b], pos[b]
                if feds[b] is not None:
                    o.pending = feds[b]
                rec = o.step_verify(n, k)
                assert rec.kept == j and rec.rollback == (m - j if step else 0), f"step {step} slot {b}: oracle"
                assert rec.emitted.tolist() == G[p:p + j + 1], f"step {step} slot {b}: oracle emitted"
                assert int(acc[b]) == j + 1, f"step {step} slot {b}: accepted {acc[b]}, expected {j + 1}"
                got = toks[b, :j + 1].tolist()
                assert got[:j] == G[p:p + j], f"step {step} slot {b}: kept drafts"
                if margins[p + j] > MARGIN:
                    assert got[j] == G[p + j], f"step {step} slot {b}: greedy token after the kept drafts"
                    compared_tokens += 1
                compared_tokens += j
                assert dec.state(b)["len"] == o.cache.length, f"step {step} slot {b}: cached length"
                assert_logits_close(lg[b], rec.logits, f"step {step} slot {b}")
                kept_seen.add(j)
                pos[b] = p + j + 1
            step += 1
    finally:
        dec.close()
    return step, kept_seen, compared_tokens, pos


def test_verify_teacher_forced_tiny_fused():
    steps, kept, compared, pos = _teacher_forced_verify(synth.TINY, 1, 4, 4, 120, 7)
    assert kept == {0, 1, 2, 3} and pos[0] >= 100 and compared >= 60


def test_verify_teacher_forced_batched_tiny_bf16():
    steps, kept, compared, pos = _teacher_forced_verify(synth.TINY_BF16, 5, 4, 4, 60, 20, batched=1)
    assert kept == {0, 1, 2, 3} and min(pos) >= 50 and compared >= 120


def test_verify_teacher_forced_valle():
    steps, kept, compared, pos = _teacher_forced_verify(synth.VALLE, 1, 4, 4, 210, 3)
    assert kept == {0, 1, 2, 3} and pos[0] >= 200 and compared >= 120


# ---- free-running: mtp_generate against the oracle's greedy sequence ----

def clear_prefix(margins):
    low = [i for i, m in enumerate(margins) if m <= MARGIN]
    return low[0] if low else len(margins)


def _run_verify(model, batch, n, k, budget, seed0, batched=1, options=()):
    mtp = lib_module()
    prompts = _prompts(model, batch, seed0)
    max_ctx = max(len(p) + len(a) for p, a in prompts) + budget + model.n_heads_max + 4
    dec, w = decoder(model, max_batch=batch, max_ctx=max_ctx, accept_policy=1)
    try:
        mtp.mtp_set_option(dec.ctx, 4, batched)
        for opt, val in options:
            mtp.mtp_set_option(dec.ctx, opt, val)
        for b, (ph, ac) in enumerate(prompts):
            dec.prefill(b, ph, ac, budget)
        out, steps = dec.generate(n, k, budget)
    finally:
        dec.close()
    compared = []
    o = MTPOracle(model, w)
    for b, (ph, ac) in enumerate(prompts):
        o.prefill(ph, ac, budget)
        ref, margins, _ = greedy_trace(o, budget, model.eos_id)
        upto = clear_prefix(margins)
        assert len(out[b]) == len(ref) or upto < len(ref)
        assert out[b][:upto + 1] == ref[:upto + 1], f"slot {b}: diverges before the first near-tie at {upto}"
        compared.append(upto)
    return out, steps, compared


def test_verify_greedy_free_running_valle():
    out, steps, compared = _run_verify(synth.VALLE, 1, 4, 4, 40, 3)
    assert len(out[0]) == 40 and compared[0] >= 20


def test_verify_greedy_free_running_batched_tiny_bf16():
    out, steps, compared = _run_verify(synth.TINY_BF16, 5, 4, 4, 24, 20, batched=1)
    assert all(len(t) == 24 for t in out) and sum(compared) >= 10
