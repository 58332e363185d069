"""GPU parity of the persistent step kernel (the embedding and every block of a
pass of <= 8 fed rows in one kernel, bf16 weights) against the oracle, and
against the two-kernel-per-layer path.

Teacher-forced as in test_gpu_decode: per step and slot the logits are within
the bf16 bar, top-k and the Viterbi path are bit-exact given the GPU's own
scores, and the path equals the oracle's wherever its decision margin is
clear.  Cases: 1, 2, 4 and 8 fed rows, two and more slots in one pass (several
attention groups), page sizes 16, 32, 64 and 128, contexts that end inside and
on the edge of a 64-key stage, the VALLE-sized model."""
import numpy as np
import pytest

import synth
from oracle import select as S
from oracle.mtp import MTPOracle

from gpu_util import MARGIN, assert_logits_close, decoder, lib_module, logp32

pytestmark = pytest.mark.gpu

OPT_PERSISTENT = 9


def _teacher_forced(model, batch, n, k, max_new, max_steps, page_size=64, seed0=0, n_ph=10, n_ac=40,
                    persistent=1):
    mtp = lib_module()
    prompts = [synth.make_prompt(seed0 + b, n_ph + 3 * b, n_ac + 7 * b, model.phone_vocab) for b in range(batch)]
    max_ctx = max(len(p) + len(a) for p, a in prompts) + max_new + model.n_heads_max + 3
    dec, w = decoder(model, max_batch=batch, max_ctx=max_ctx, page_size=page_size)
    steps = clear = 0
    try:
        mtp.mtp_set_option(dec.ctx, OPT_PERSISTENT, persistent)
        assert mtp.mtp_get_option(dec.ctx, OPT_PERSISTENT) == persistent
        oracles = []
        for b, (ph, ac) in enumerate(prompts):
            o = MTPOracle(model, w) if b == 0 else _share(oracles[0])
            o.prefill(ph, ac, max_new)
            dec.prefill(b, ph, ac, max_new)
            oracles.append(o)
        while steps < max_steps and not all(o.done for o in oracles):
            recs = []
            for b, o in enumerate(oracles):
                if o.done:
                    recs.append(None)
                    continue
                fed = o.pending.copy()
                recs.append(o.step(n, k))
                if len(fed):
                    mtp.mtp_set_teacher_tokens(dec.ctx, b, fed)
            toks, acc, done = dec.decode_step(n, k)
            lg, lse = dec.logits(n)
            ids, lp, path = dec.lattice(n, k)
            for b, rec in enumerate(recs):
                if rec is None:
                    continue
                what = f"step {steps} slot {b}"
                assert_logits_close(lg[b], rec.logits, what)
                r_ids, r_vals = S.top_k_rows(logp32(lg[b], lse[b]), k)
                assert np.array_equal(ids[b], r_ids) and np.array_equal(lp[b], r_vals), what
                r_path, _, _ = S.viterbi(ids[b:b + 1], lp[b:b + 1], oracles[b].log_q)
                assert np.array_equal(path[b], r_path[0]), what
                if rec.margin > MARGIN:
                    clear += 1
                    assert np.array_equal(path[b], rec.path), f"{what}: clear decision differs"
            steps += 1
    finally:
        dec.close()
    return steps, clear


def _share(o):
    """A second oracle sharing the first one's (float64) weights."""
    import copy
    return copy.copy(o)


@pytest.mark.parametrize("n", [1, 2, 4, 8])
def test_rows_per_pass_tiny_bf16(n):
    steps, _ = _teacher_forced(synth.TINY_BF16, 1, n, 4, 40, 8)
    assert steps == min(8, -(-40 // n))


@pytest.mark.parametrize("batch,n", [(2, 4), (4, 2), (8, 1), (3, 2)])
def test_several_slots_per_pass_tiny_bf16(batch, n):
    _teacher_forced(synth.TINY_BF16, batch, n, 4, 30, 6, seed0=5)


@pytest.mark.parametrize("page_size", [16, 32, 128])
def test_page_sizes_tiny_bf16(page_size):
    _teacher_forced(synth.TINY_BF16, 2, 4, 4, 40, 8, page_size=page_size, seed0=11)


@pytest.mark.parametrize("n_ac", [44, 45, 50, 118])
def test_stage_edges_tiny_bf16(n_ac):
    """Prompts of 10 + n_ac positions: cached lengths just below, at and past a 64-key stage edge."""
    _teacher_forced(synth.TINY_BF16, 1, 4, 4, 16, 5, n_ac=n_ac, seed0=2)


def test_valle_teacher_forced():
    steps, clear = _teacher_forced(synth.VALLE, 1, 4, 4, 200, 50, n_ph=64, n_ac=225)
    assert steps == 50


def test_persistent_equals_block_kernels_valle():
    """The same steps through both paths: logits within 1e-3 (same arithmetic, other summation order)."""
    mtp = lib_module()
    model = synth.VALLE
    ph, ac = synth.make_prompt(0, 64, 225, model.phone_vocab)
    outs = []
    for persistent in (1, 0):
        dec, _ = decoder(model, max_batch=1, max_ctx=400)
        try:
            mtp.mtp_set_option(dec.ctx, OPT_PERSISTENT, persistent)
            dec.prefill(0, ph, ac, 80)
            lgs, toks = [], []
            for step in range(6):
                if step:
                    mtp.mtp_set_teacher_tokens(dec.ctx, 0, np.array([5 + step, 900, 17, 333], np.int32))
                dec.decode_step(4, 4)
                lgs.append(dec.logits(4)[0][0].copy())
            outs.append(lgs)
        finally:
            dec.close()
    for a, b in zip(outs[0], outs[1]):
        assert np.abs(a - b).max() <= 1e-3


def test_generate_graphs_equal_stepping_valle():
    """mtp_generate (graphs of chained persistent steps) = step-by-step decoding."""
    mtp = lib_module()
    model = synth.VALLE
    ph, ac = synth.make_prompt(1, 64, 225, model.phone_vocab)
    res = []
    for stepwise in (False, True):
        dec, _ = decoder(model, max_batch=1, max_ctx=700)
        try:
            mtp.mtp_set_option(dec.ctx, OPT_PERSISTENT, 1)
            dec.prefill(0, ph, ac, 300)
            if stepwise:
                toks = []
                while not dec.state(0)["done"]:
                    t, a, _ = dec.decode_step(4, 4)
                    toks += t[0, :a[0]].tolist()
            else:
                out, steps = dec.generate(4, 4, 300)
                toks = out[0]
            res.append(toks)
        finally:
            dec.close()
    assert len(res[0]) == 300 and res[0] == res[1]
