"""GPU parity of the batched path (all slots' fed rows in one pass through the
tensor-core projections) against one oracle per sequence, teacher-forced.

Per slot and step: logits within the bf16 bar; top-k bit-exact given the
GPU's own scores; Viterbi path bit-exact given the GPU's lattice; the path
equal to the oracle's wherever the oracle's decision margin exceeds 5e-2.
The fused path (8-row passes) must give the same logits to float tolerance."""
import numpy as np
import pytest

import synth
from oracle import select as S
from oracle.mtp import MTPOracle

from gpu_util import MARGIN, assert_logits_close, decoder, lib_module, logp32

pytestmark = pytest.mark.gpu


def _prompts(model, batch, seed0):
    out = []
    for b in range(batch):
        lens = synth.uniform(seed0 + b, "batched_len", 2)
        n_ph = 8 + int(lens[0] * 24)
        n_ac = 20 + int(lens[1] * 40)
        out.append(synth.make_prompt(seed0 + b, n_ph, n_ac, model.phone_vocab))
    return out


def _serving_prompts(model, batch):
    """The batched-serving recipe: U[32,128] phonemes + U[150,450] acoustic tokens (seeds 2000 + i)."""
    out = []
    for i in range(batch):
        n_ph = synth.make_lengths(i, 32, 128, "serve_phonemes")
        n_ac = synth.make_lengths(i, 150, 450, "serve_acoustic")
        out.append(synth.make_prompt(i, n_ph, n_ac, model.phone_vocab))
    return out


def batched_teacher_forced(model, batch, n, k, max_new, max_steps, seed0=300, batched=1, prompts=None):
    mtp = lib_module()
    prompts = prompts if prompts is not None else _prompts(model, batch, seed0)
    max_ctx = max(len(p) + len(a) for p, a in prompts) + max_new + model.n_heads_max + 3
    dec, w = decoder(model, max_batch=batch, max_ctx=max_ctx)
    logs = []
    try:
        mtp.mtp_set_option(dec.ctx, 4, batched)
        assert mtp.mtp_get_option(dec.ctx, 4) == batched, "batched path not available"
        oracles = []
        for b, (ph, ac) in enumerate(prompts):
            o = MTPOracle(model, w)
            o.prefill(ph, ac, max_new)
            dec.prefill(b, ph, ac, max_new)
            oracles.append(o)
        for step in range(max_steps):
            recs = []
            for b, o in enumerate(oracles):
                fed = o.pending.copy()
                recs.append(o.step(n, k) if not o.done else None)
                if len(fed):
                    mtp.mtp_set_teacher_tokens(dec.ctx, b, fed)
            toks, acc, done = dec.decode_step(n, k)
            lg, lse = dec.logits(n)
            ids, lp, path = dec.lattice(n, k)
            logs.append(lg.copy())
            for b, rec in enumerate(recs):
                if rec is None:
                    continue
                assert_logits_close(lg[b], rec.logits, f"slot {b} step {step}")
                r_ids, r_vals = S.top_k_rows(logp32(lg[b], lse[b]), k)
                assert np.array_equal(ids[b], r_ids) and np.array_equal(lp[b], r_vals), f"slot {b} step {step}"
                r_path, _, _ = S.viterbi(ids[b:b + 1], lp[b:b + 1], oracles[b].log_q)
                assert np.array_equal(path[b], r_path[0]), f"slot {b} step {step}"
                if rec.margin > MARGIN:
                    assert np.array_equal(path[b], rec.path), f"slot {b} step {step}: clear decision differs"
        return np.stack(logs)
    finally:
        dec.close()


def test_batched_tiny_bf16_matches_oracle():
    batched_teacher_forced(synth.TINY_BF16, batch=5, n=4, k=4, max_new=40, max_steps=8)


def test_batched_tiny_bf16_n8_k8():
    batched_teacher_forced(synth.TINY_BF16, batch=3, n=8, k=8, max_new=40, max_steps=4)


def test_batched_equals_fused_passes():
    a = batched_teacher_forced(synth.TINY_BF16, batch=4, n=3, k=4, max_new=24, max_steps=4, batched=1)
    b = batched_teacher_forced(synth.TINY_BF16, batch=4, n=3, k=4, max_new=24, max_steps=4, batched=0)
    assert np.abs(a - b).max() <= 1e-3


def test_batched_valle_b32():
    batched_teacher_forced(synth.VALLE, batch=32, n=4, k=4, max_new=16, max_steps=2, seed0=500)


def test_batched_valle_b32_serving_prompts():
    """VALL-E-sized B=32 with the serving workload's prompt lengths (182-578 positions: two to
    five 128-position prefill chunks per slot; decode contexts of several key pages per split)."""
    prompts = _serving_prompts(synth.VALLE, 32)
    lens = [len(p) + len(a) for p, a in prompts]
    assert min(lens) > 128 and max(lens) > 3 * 128
    batched_teacher_forced(synth.VALLE, batch=32, n=4, k=4, max_new=8, max_steps=2, prompts=prompts)


def test_batched_tiny_bf16_b128():
    """The batch-128 serving shape: 512 fed rows per step (several activation tiles per
    projection, 128 attention groups)."""
    batched_teacher_forced(synth.TINY_BF16, batch=128, n=4, k=4, max_new=16, max_steps=3, seed0=700)
