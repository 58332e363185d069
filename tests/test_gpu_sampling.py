"""Path sampling on the GPU (the top-k sampling of Fig. 2: a path drawn from
the lattice's posterior).  Per step, teacher-forced on the oracle's fed
tokens: the logits stay within the bar, and the drawn path equals the
oracle's draw (float64 forward filtering) on the GPU's own float32 scores
with the same SplitMix64 uniforms wherever every draw of the path is clear of
a sampling boundary by SAMPLE_MARGIN of its total weight (the GPU filters in
float32; its weight errors are ~1e-5 relative).  Also: draws are reproducible
for a seed and vary across seeds, and under VERIFY_GREEDY sampled drafts leave
the greedy output unchanged."""
import numpy as np
import pytest

import synth
from oracle import select as S
from oracle.mtp import MTPOracle

from gpu_util import assert_logits_close, decoder, lib_module, logp32
from test_gpu_verify import _run_verify

pytestmark = pytest.mark.gpu

OPT_BATCHED, OPT_LATTICE, OPT_SAMPLING, OPT_SEED = 4, 6, 7, 8
SAMPLE_MARGIN = 1e-3


@pytest.mark.parametrize("model,batch,n,k,lattice,steps", [
    (synth.TINY, 2, 4, 4, "A", 10),
    (synth.TINY, 1, 8, 32, "A", 5),
    (synth.TINY, 1, 6, 8, "B", 6),
    (synth.VALLE, 1, 4, 8, "A", 4),
])
def test_sampled_path_matches_oracle(model, batch, n, k, lattice, steps):
    mtp = lib_module()
    seed = 0xC0FFEE
    prompts = [synth.make_prompt(21 + b, 12 + b, 40, model.phone_vocab) for b in range(batch)]
    max_ctx = max(len(p) + len(a) for p, a in prompts) + 120
    dec, w = decoder(model, max_batch=batch, max_ctx=max_ctx)
    compared = 0
    try:
        mtp.mtp_set_option(dec.ctx, OPT_SAMPLING, 1)
        mtp.mtp_set_option(dec.ctx, OPT_SEED, seed)
        mtp.mtp_set_option(dec.ctx, OPT_LATTICE, 1 if lattice == "B" else 0)
        assert mtp.mtp_get_option(dec.ctx, OPT_SAMPLING) == 1
        oracles = []
        for b, (ph, ac) in enumerate(prompts):
            o = MTPOracle(model, w)
            o.prefill(ph, ac, 80)
            dec.prefill(b, ph, ac, 80)
            oracles.append(o)
        generated = [0] * batch
        for step in range(steps):
            recs = []
            for b, o in enumerate(oracles):
                fed = o.pending.copy()
                recs.append(o.step(n, k, lattice=lattice, sample=(seed, b)))
                if len(fed):
                    mtp.mtp_set_teacher_tokens(dec.ctx, b, fed)
            toks, acc, _ = dec.decode_step(n, k)
            lg, lse = dec.logits(n)
            _, _, path = dec.lattice(n, k)
            for b in range(batch):
                assert_logits_close(lg[b], recs[b].logits, f"step {step} slot {b}")
                sc = logp32(lg[b], lse[b])
                ids, vals = S.top_k_rows(sc, k)
                u = [S.path_uniform(seed, b, generated[b], t) for t in range(n)]
                if lattice == "B":
                    r_path, margin = S.sample_path_union(ids, sc, oracles[b].log_q, u)
                else:
                    r_path, margin = S.sample_path(ids, vals, oracles[b].log_q, u)
                if margin > SAMPLE_MARGIN:
                    assert np.array_equal(path[b], r_path), f"step {step} slot {b} margin {margin:.2e}"
                    compared += 1
                a = int(acc[b])
                assert toks[b, :a].tolist() == path[b, :a].tolist()
                generated[b] += a
    finally:
        dec.close()
    assert compared >= batch * steps // 2


def _generate(model, n, k, seed, budget=60):
    mtp = lib_module()
    ph, ac = synth.make_prompt(31, 14, 40, model.phone_vocab)
    dec, _ = decoder(model, max_batch=1, max_ctx=len(ph) + len(ac) + budget + 16)
    try:
        mtp.mtp_set_option(dec.ctx, OPT_SAMPLING, 1)
        mtp.mtp_set_option(dec.ctx, OPT_SEED, seed)
        dec.prefill(0, ph, ac, budget)
        out, _ = dec.generate(n, k, budget)
    finally:
        dec.close()
    return out[0]


def test_draws_are_reproducible_and_seeded():
    a = _generate(synth.TINY, 4, 8, 5)
    assert _generate(synth.TINY, 4, 8, 5) == a
    others = [_generate(synth.TINY, 4, 8, s) for s in (6, 7, 8)]
    assert any(o != a for o in others)


@pytest.mark.parametrize("batched", [0, 1])
def test_sampled_drafts_keep_greedy_output(batched):
    """VALLE-sized, 3 slots: the greedy sequence up to each slot's first near-tie (23, 15 and 7
    tokens on these prompts) is emitted whatever drafts the sampler draws."""
    _, _, compared = _run_verify(synth.VALLE, 3, 4, 8, 40, 51, batched=batched,
                                 options=((OPT_SAMPLING, 1), (OPT_SEED, 99)))
    assert sum(compared) >= 40
