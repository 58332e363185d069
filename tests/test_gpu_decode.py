"""End-to-end GPU parity of the MTP decode path against the oracle (teacher-forced).

Each step both sides feed the same tokens (the oracle's accepted ones).  Per
step: logits within the bf16 bar; top-k, Viterbi path and accepted count
bit-exact given the GPU's own scores; the path equal to the oracle's wherever
the oracle's decision margin exceeds 5e-2."""
import numpy as np
import pytest

import synth
from oracle import select as S
from oracle.mtp import MTPOracle

from gpu_util import MARGIN, assert_logits_close, decoder, lib_module, logp32

pytestmark = pytest.mark.gpu


def teacher_forced(model, n, k, n_ph, n_ac, max_new, max_steps=None, page_size=64, seq=0):
    mtp = lib_module()
    max_ctx = n_ph + n_ac + max_new + model.n_heads_max + 3
    dec, w = decoder(model, max_batch=1, max_ctx=max_ctx, page_size=page_size)
    try:
        ph, ac = synth.make_prompt(seq, n_ph, n_ac, model.phone_vocab)
        o = MTPOracle(model, w)
        o.prefill(ph, ac, max_new)
        dec.prefill(0, ph, ac, max_new)
        steps = clear = 0
        while not o.done and (max_steps is None or steps < max_steps):
            fed = o.pending.copy()
            rec = o.step(n, k)
            if len(fed):
                mtp.mtp_set_teacher_tokens(dec.ctx, 0, fed)
            toks, acc, done = dec.decode_step(n, k)
            lg, lse = dec.logits(n)
            ids, lp, path = dec.lattice(n, k)
            assert_logits_close(lg[0], rec.logits, f"step {steps}")
            r_ids, r_vals = S.top_k_rows(logp32(lg[0], lse[0]), k)
            assert np.array_equal(ids[0], r_ids) and np.array_equal(lp[0], r_vals), f"step {steps}"
            r_path, _, _ = S.viterbi(ids, lp, o.log_q)
            assert np.array_equal(path[0], r_path[0]), f"step {steps}"
            if rec.margin > MARGIN:
                clear += 1
                assert np.array_equal(path[0], rec.path), f"step {steps}: clear decision differs"
            a = int(acc[0])
            assert toks[0, :a].tolist() == path[0, :a].tolist() and np.all(toks[0, a:] == -1)
            steps += 1
        return steps, clear
    finally:
        dec.close()


def test_tiny_full_generation():
    steps, _ = teacher_forced(synth.TINY, 4, 4, 32, 75, 150)
    assert steps == 38


def test_valle_full_generation():
    steps, clear = teacher_forced(synth.VALLE, 4, 4, 64, 225, 750)
    assert steps == 188


@pytest.mark.parametrize("n,k", [(1, 1), (1, 8), (2, 4), (8, 16), (8, 25), (3, 32)])
def test_valle_head_and_beam_sweep(n, k):
    teacher_forced(synth.VALLE, n, k, 64, 225, 1500, max_steps=6)


@pytest.mark.parametrize("page_size", [16, 128])
def test_page_sizes(page_size):
    teacher_forced(synth.TINY, 4, 4, 20, 50, 40, max_steps=6, page_size=page_size)


def test_generate_equals_stepping_and_launch_modes():
    """mtp_generate (graph, no host sync) = repeated mtp_decode_step = eager launches."""
    mtp = lib_module()
    model = synth.TINY
    ph, ac = synth.make_prompt(5, 16, 40, model.phone_vocab)
    results = []
    for graphs, pdl, stepwise in [(1, 1, False), (1, 1, True), (0, 0, False), (0, 1, True)]:
        dec, _ = decoder(model, max_batch=1, max_ctx=200)
        try:
            mtp.mtp_set_option(dec.ctx, 0, graphs)
            mtp.mtp_set_option(dec.ctx, 1, pdl)
            dec.prefill(0, ph, ac, 61)
            if stepwise:
                toks = []
                while not dec.state(0)["done"]:
                    t, a, _ = dec.decode_step(4, 4)
                    toks += t[0, :a[0]].tolist()
            else:
                out, steps = dec.generate(4, 4, 61)
                toks = out[0]
                assert steps == 16
            results.append(toks)
        finally:
            dec.close()
    assert len(results[0]) == 61
    assert all(r == results[0] for r in results)


def test_n1_is_greedy_on_gpu_scores():
    dec, _ = decoder(synth.TINY, max_batch=1, max_ctx=160)
    try:
        ph, ac = synth.make_prompt(2, 10, 30, synth.TINY.phone_vocab)
        dec.prefill(0, ph, ac, 20)
        for _ in range(20):
            toks, acc, _ = dec.decode_step(1, 4)
            lg, lse = dec.logits(1)
            sc = logp32(lg[0], lse[0])[0]
            assert acc[0] == 1 and toks[0, 0] == int(np.argmax(sc))
    finally:
        dec.close()


# The block kernels add residual contributions from many CTAs with float
# atomics, so two runs of the same step may differ in the last bits; the
# cache-bookkeeping checks below therefore compare to 1e-5 (a wrong page,
# position or length moves logits by O(0.1)).
REPEAT_ATOL = 1e-5


def test_rollback_then_append():
    """append(A); rollback(|A|); append(C) gives the logits of append(C) on a fresh cache."""
    mtp = lib_module()
    ph, ac = synth.make_prompt(3, 12, 30, synth.TINY.phone_vocab)
    dec, _ = decoder(synth.TINY, max_batch=1, max_ctx=200)
    ref, _ = decoder(synth.TINY, max_batch=1, max_ctx=200)
    try:
        dec.prefill(0, ph, ac, 100)
        a_toks, _, _ = dec.decode_step(4, 4)        # selects A
        dec.decode_step(4, 4)                       # feeds A
        lg_a, _ = dec.logits(4)
        t = dec.state(0)["len"]
        mtp.mtp_rollback(dec.ctx, 0, 4)
        assert dec.state(0)["len"] == t - 4
        mtp.mtp_set_teacher_tokens(dec.ctx, 0, a_toks[0])   # A again: same logits
        dec.decode_step(4, 4)
        lg_a2, _ = dec.logits(4)
        assert np.abs(lg_a - lg_a2).max() <= REPEAT_ATOL
        c = np.array([7, 1000, 3, 512], np.int32)
        mtp.mtp_rollback(dec.ctx, 0, 4)
        mtp.mtp_set_teacher_tokens(dec.ctx, 0, c)
        dec.decode_step(4, 4)
        lg_c, _ = dec.logits(4)
        ref.prefill(0, ph, ac, 100)
        ref.decode_step(4, 4)
        mtp.mtp_set_teacher_tokens(ref.ctx, 0, c)
        ref.decode_step(4, 4)
        lg_ref, _ = ref.logits(4)
        assert np.abs(lg_c - lg_ref).max() <= REPEAT_ATOL
    finally:
        dec.close()
        ref.close()


def test_page_placement():
    """The same sequence on other physical pages gives identical logits."""
    ph, ac = synth.make_prompt(4, 12, 40, synth.TINY.phone_vocab)
    other_ph, other_ac = synth.make_prompt(9, 30, 60, synth.TINY.phone_vocab)
    out = []
    for first_other in (False, True):
        dec, _ = decoder(synth.TINY, max_batch=2, max_ctx=240)
        try:
            if first_other:
                dec.prefill(1, other_ph, other_ac, 50)   # takes the first pages
                from paper_2410_13839_gb300 import mtp as M
                M.mtp_release(dec.ctx, 1)
                dec.prefill(1, other_ph[:5], other_ac[:5], 150)
            dec.prefill(0, ph, ac, 30)
            logits = []
            for _ in range(4):
                dec.decode_step(4, 4)
                logits.append(dec.logits(4)[0][0].copy())
            out.append(logits)
        finally:
            dec.close()
    for a, b in zip(out[0], out[1]):
        assert np.abs(a - b).max() <= REPEAT_ATOL


def test_eos_finishes_a_slot():
    dec, _ = decoder(synth.TINY, max_batch=1, max_ctx=200, eos_bias=40.0)
    try:
        ph, ac = synth.make_prompt(1, 10, 20, synth.TINY.phone_vocab)
        dec.prefill(0, ph, ac, 100)
        toks, acc, done = dec.decode_step(4, 4)
        assert acc[0] == 1 and toks[0, 0] == synth.TINY.eos_id and done[0] == 1
        toks, acc, done = dec.decode_step(4, 4)     # a finished slot stays idle
        assert acc[0] == 0 and np.all(toks[0] == -1)
    finally:
        dec.close()


def test_invalid_calls_are_rejected():
    mtp = lib_module()
    dec, _ = decoder(synth.TINY, max_batch=1, max_ctx=100)
    try:
        ph, ac = synth.make_prompt(1, 10, 20, synth.TINY.phone_vocab)
        with pytest.raises(mtp.MTPError):
            dec.prefill(0, ph, ac, 90)               # exceeds max_ctx
        with pytest.raises(mtp.MTPError):
            dec.prefill(1, ph, ac, 10)               # no such slot
        bad = ac.copy()
        bad[3] = 5000
        with pytest.raises(mtp.MTPError):
            dec.prefill(0, ph, bad, 10)              # id out of range
        dec.prefill(0, ph, ac, 10)
        with pytest.raises(mtp.MTPError):
            dec.decode_step(9, 4)                    # more heads than stored
        with pytest.raises(mtp.MTPError):
            dec.decode_step(4, 33)
        with pytest.raises(mtp.MTPError):
            mtp.mtp_rollback(dec.ctx, 0, 1000)
    finally:
        dec.close()
