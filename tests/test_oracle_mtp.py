"""Pins of the oracle's multi-token inference loop (Fig. 1 caption, Sec. III-B)."""
import numpy as np

import synth
from oracle import model as M
from oracle.mtp import MTPOracle


def _prompt():
    return synth.make_prompt(0, 32, 75, synth.TINY.phone_vocab)


def test_n1_equals_plain_greedy_ar(tiny_weights):
    """With one head the MTP loop is greedy AR (Eq. 1): compare with a cache-free loop."""
    cfg = synth.TINY
    ph, ac = _prompt()
    o = MTPOracle(cfg, tiny_weights)
    o.prefill(ph, ac, 24)
    o.generate(1, 4)
    w = {n: np.asarray(t, np.float64) for n, t in tiny_weights.items()}
    dec = M.ARDecoder(cfg, tiny_weights)
    seq = list(ph) + list(ac)
    n_ph = len(ph)
    greedy = []
    for _ in range(24):
        is_phone = np.arange(len(seq)) < n_ph
        h = dec.forward(np.array(seq), is_phone, dec.new_cache())[-1]
        z = M.layer_norm(h, w["lnf_g"], w["lnf_b"], cfg.ln_eps)
        logits = w["w_heads"][0] @ z + w["b_heads"][0]
        tok = int(np.argmax(logits))
        greedy.append(tok)
        seq.append(tok)
    assert o.generated == greedy


def test_first_heads_do_not_depend_on_n(tiny_weights):
    cfg = synth.TINY
    ph, ac = _prompt()
    recs = {}
    for n in (1, 2, 4, 8):
        o = MTPOracle(cfg, tiny_weights)
        o.prefill(ph, ac, 40)
        recs[n] = o.step(n, 4)
    for n in (2, 4, 8):
        for i in (1, 2, 4):
            if i <= n:
                assert np.array_equal(recs[n].logits[:i], recs[i].logits[:i])


def test_budget_and_step_count(tiny_weights):
    ph, ac = _prompt()
    o = MTPOracle(synth.TINY, tiny_weights)
    o.prefill(ph, ac, 10)
    recs = o.generate(4, 4)
    assert [r.accepted for r in recs] == [4, 4, 2]
    assert len(o.generated) == 10 and recs[-1].done


def test_eos_ends_the_sequence():
    cfg = synth.TINY
    w = synth.make_weights(cfg, eos_bias=40.0)
    ph, ac = _prompt()
    o = MTPOracle(cfg, w)
    o.prefill(ph, ac, 100)
    recs = o.generate(4, 4)
    assert len(recs) == 1 and recs[0].accepted == 1 and o.generated == [cfg.eos_id]


def test_teacher_forcing_feeds_given_tokens(tiny_weights):
    ph, ac = _prompt()
    a = MTPOracle(synth.TINY, tiny_weights)
    a.prefill(ph, ac, 100)
    a.step(4, 4)
    ra = a.step(4, 4, teacher=[1, 2, 3])
    b = MTPOracle(synth.TINY, tiny_weights)
    b.prefill(np.asarray(ph), np.concatenate([ac, [1, 2, 3]]), 100)
    rb = b.step(4, 4)
    assert np.allclose(ra.logits, rb.logits, atol=1e-12)
