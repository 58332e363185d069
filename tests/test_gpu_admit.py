"""Admitted prompts prefilled inside the decode steps (chunked prefill in the
batched pass's lane, Sec. III-A prompt; Sec. III-B/C steps) against the oracle.

A slot admitted mid-generation (mtp_admit) runs its prompt in the prefill lane
of the next steps, 128 positions per step, beside the other slots' fed rows;
it selects nothing until its prompt is done, then decodes.  Every slot,
teacher-forced, matches its own oracle: logits within the bf16 bar at every
step, top-k and Viterbi path bit-exact given the GPU's scores.  Also:
mtp_prefill_pending (many slots' prompt rows per pass) against sequential
prefill, and mtp_generate over admitted prompts."""
import copy

import numpy as np
import pytest

import synth
from oracle import select as S
from oracle.mtp import MTPOracle

from gpu_util import assert_logits_close, decoder, lib_module, logp32

pytestmark = pytest.mark.gpu

LANE = 128


def _check_step(dec, recs, n, k, log_q, step):
    lg, lse = dec.logits(n)
    ids, lp, path = dec.lattice(n, k)
    for b, rec in recs.items():
        what = f"step {step} slot {b}"
        assert_logits_close(lg[b], rec.logits, what)
        r_ids, r_vals = S.top_k_rows(logp32(lg[b], lse[b]), k)
        assert np.array_equal(ids[b], r_ids) and np.array_equal(lp[b], r_vals), what
        r_path, _, _ = S.viterbi(ids[b:b + 1], lp[b:b + 1], log_q)
        assert np.array_equal(path[b], r_path[0]), what


def _admit_mid_generation(model, batch, n, k, admit_len, steps_before, steps_after, seed0):
    mtp = lib_module()
    prompts = [synth.make_prompt(seed0 + b, 12 + 3 * b, 40 + 5 * b, model.phone_vocab) for b in range(batch - 1)]
    late = synth.make_prompt(seed0 + 99, 20, admit_len - 20, model.phone_vocab)
    max_new = 4 * (steps_before + steps_after) + 8
    max_ctx = max(len(p) + len(a) for p, a in prompts + [late]) + max_new + model.n_heads_max + 4
    dec, w = decoder(model, max_batch=batch, max_ctx=max_ctx)
    oracles = {}
    try:
        for b, (ph, ac) in enumerate(prompts):
            dec.prefill(b, ph, ac, max_new)
            o = MTPOracle(model, w) if not oracles else copy.copy(next(iter(oracles.values())))
            o.prefill(ph, ac, max_new)
            oracles[b] = o
        late_slot = batch - 1
        log_q = oracles[0].log_q
        lane_steps = -(-admit_len // (LANE // n * n))
        waited = None
        accepted_late = []
        for step in range(steps_before + steps_after):
            if step == steps_before:
                dec.admit(late_slot, *late, max_new)
                waited = 0
            recs = {}
            for b, o in oracles.items():
                fed = o.pending.copy()
                recs[b] = o.step(n, k)
                if len(fed):
                    mtp.mtp_set_teacher_tokens(dec.ctx, b, fed)
            _, acc, _ = dec.decode_step(n, k)
            _check_step(dec, recs, n, k, log_q, step)
            if waited is not None and late_slot not in oracles:
                accepted_late.append(int(acc[late_slot]))
                waited += 1
                st = dec.state(late_slot)
                if waited == lane_steps:  # the prompt ran in the lane of these steps
                    assert st["len"] == admit_len and st["pending"] == 0
                    o = copy.copy(oracles[0])
                    o.prefill(*late, max_new)
                    oracles[late_slot] = o
                else:
                    assert st["len"] == min(admit_len, waited * (LANE // n * n))
        assert accepted_late == [0] * lane_steps  # nothing selected while the prompt ran
        assert late_slot in oracles
    finally:
        dec.close()
    return oracles


def test_admit_mid_generation_tiny_bf16():
    oracles = _admit_mid_generation(synth.TINY_BF16, 5, 4, 4, admit_len=230, steps_before=4, steps_after=8,
                                    seed0=40)
    assert len(oracles[4].generated) > 0


def test_admit_mid_generation_valle():
    _admit_mid_generation(synth.VALLE, 9, 4, 4, admit_len=289, steps_before=3, steps_after=7, seed0=60)


def test_admit_single_slot_uses_the_lane():
    """B = 1 (the fused path otherwise): an admitted prompt runs in the batched pass's lane."""
    _admit_mid_generation(synth.TINY_BF16, 2, 4, 4, admit_len=140, steps_before=2, steps_after=5, seed0=70)


def test_prefill_pending_equals_sequential_prefill():
    mtp = lib_module()
    model = synth.TINY_BF16
    prompts = [synth.make_prompt(80 + b, 20 + 7 * b, 90 + 31 * b, model.phone_vocab) for b in range(4)]
    outs = []
    for admitted in (True, False):
        dec, w = decoder(model, max_batch=4, max_ctx=400)
        try:
            for b, (ph, ac) in enumerate(prompts):
                (dec.admit if admitted else dec.prefill)(b, ph, ac, 40)
            if admitted:
                assert mtp.mtp_prefill_pending(dec.ctx) >= 1
                assert mtp.mtp_prefill_pending(dec.ctx) == 0
            lgs = []
            for step in range(3):
                if step:
                    for b in range(4):
                        mtp.mtp_set_teacher_tokens(dec.ctx, b, np.array([3 + b, 700, 17, 1000 - step], np.int32))
                dec.decode_step(4, 4)
                lgs.append(dec.logits(4)[0].copy())
            outs.append(lgs)
            for b, (ph, ac) in enumerate(prompts):
                assert dec.state(b)["len"] == len(ph) + len(ac) + 8
        finally:
            dec.close()
        if admitted:  # the admitted run against the oracle at the first step
            o = MTPOracle(model, w)
            for b, (ph, ac) in enumerate(prompts):
                o.prefill(ph, ac, 40)
                assert_logits_close(outs[0][0][b], o.step(4, 4).logits, f"slot {b}")
    for a, b in zip(outs[0], outs[1]):
        assert np.abs(a - b).max() <= 1e-3


def test_generate_runs_admitted_prompts():
    model = synth.TINY_BF16
    prompts = [synth.make_prompt(90 + b, 15, 60 + 40 * b, model.phone_vocab) for b in range(6)]
    dec, _ = decoder(model, max_batch=6, max_ctx=400)
    try:
        dec.prefill(0, *prompts[0], 30)
        for b in range(1, 6):
            dec.admit(b, *prompts[b], 30 + b)
        out, steps = dec.generate(4, 4, 40)
        assert [len(t) for t in out] == [30, 31, 32, 33, 34, 35]
        assert all(0 <= t < model.codec_vocab for toks in out for t in toks)
        for b in range(6):
            st = dec.state(b)
            assert st["done"] == 1 and st["generated"] == 30 + b
    finally:
        dec.close()
