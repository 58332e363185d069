"""VERIFY_GREEDY on the GPU (speculative decoding with the heads as drafter):
the emitted sequence equals the oracle's greedy AR sequence up to the first
near-tie (oracle top-1 margin <= 5e-2, where float rounding may legitimately
pick the other token); drafts equal to the greedy continuation are all kept;
rejected drafts are rolled back (later steps would diverge otherwise)."""
import numpy as np
import pytest

import synth
from oracle.mtp import MTPOracle
from oracle.select import head_logits, log_softmax

from gpu_util import MARGIN, decoder, lib_module

pytestmark = pytest.mark.gpu


def oracle_greedy(model, w, ph, ac, budget):
    """Greedy AR tokens and, per token, the float32 top-1 margin of its decision."""
    o = MTPOracle(model, w)
    o.prefill(ph, ac, budget)
    toks, margins = [], []
    while len(toks) < budget:
        lp = log_softmax(head_logits(o.h_last, o.w, 1, model.ln_eps))[0].astype(np.float32)[0]
        order = np.lexsort((np.arange(lp.shape[0]), -lp))
        toks.append(int(order[0]))
        margins.append(float(lp[order[0]] - lp[order[1]]))
        if toks[-1] == model.eos_id:
            break
        o.feed([toks[-1]])
    return toks, margins


def clear_prefix(margins):
    low = [i for i, m in enumerate(margins) if m <= MARGIN]
    return low[0] if low else len(margins)


def _run_verify(model, batch, n, k, budget, seed0, batched=1, options=()):
    mtp = lib_module()
    prompts = [synth.make_prompt(seed0 + b, 10 + 3 * b, 30 + 5 * b, model.phone_vocab) for b in range(batch)]
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
    for b, (ph, ac) in enumerate(prompts):
        ref, margins = oracle_greedy(model, w, ph, ac, budget)
        upto = clear_prefix(margins)
        assert len(out[b]) == len(ref) or upto < len(ref)
        assert out[b][:upto + 1] == ref[:upto + 1], f"slot {b}: diverges before the first near-tie at {upto}"
    return out, steps


def test_verify_greedy_tiny():
    out, steps = _run_verify(synth.TINY, 1, 4, 4, 40, 7)
    assert len(out[0]) == 40


def test_verify_greedy_batched_tiny_bf16():
    _run_verify(synth.TINY_BF16, 5, 4, 4, 24, 20, batched=1)


def test_verify_greedy_valle():
    _run_verify(synth.VALLE, 1, 4, 4, 40, 3)


def test_correct_drafts_are_kept():
    mtp = lib_module()
    model = synth.TINY
    dec, w = decoder(model, max_batch=1, max_ctx=200, accept_policy=1)
    try:
        ph, ac = synth.make_prompt(11, 12, 30, model.phone_vocab)
        ref, margins = oracle_greedy(model, w, ph, ac, 12)
        dec.prefill(0, ph, ac, 12)
        toks, acc, _ = dec.decode_step(4, 4)              # emits the first greedy token
        assert acc[0] == 1 and toks[0, 0] == ref[0]
        mtp.mtp_set_teacher_tokens(dec.ctx, 0, np.asarray(ref[0:4], np.int32))  # c + 3 correct drafts
        toks, acc, _ = dec.decode_step(4, 4)
        if min(margins[:5]) > MARGIN:
            assert acc[0] == 4 and toks[0, :4].tolist() == ref[1:5]
        st = dec.state(0)
        assert st["len"] == len(ph) + len(ac) + 4           # c and three kept drafts are cached
    finally:
        dec.close()
