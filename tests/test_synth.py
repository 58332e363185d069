"""The seeded input generators hold the recipe the inputs are said to follow:
the transition matrix Q (rows sum to 1, self-transition mass about 0.3), bf16
rounding (ties to even, as torch rounds), counter-based streams that are
deterministic and independent per (seed, name), prompt and length ranges, and
the weight recipe (N(0, 0.02), LayerNorm gains near 1, EOS bias, bf16 matrices)."""
import numpy as np
import pytest

import synth


def test_transition_matrix_rows_and_self_mass():
    lq = synth.transition_log_q(257)
    q = np.exp(lq.astype(np.float64))
    assert lq.dtype == np.float32 and np.isfinite(lq).all()
    assert np.abs(q.sum(axis=1) - 1.0).max() < 1e-5
    diag = np.diag(q)
    assert 0.3 <= diag.min() and diag.mean() < 0.32   # 0.3 plus the row's own exp(g) share
    off = q[~np.eye(257, dtype=bool)]
    assert off.max() < 0.3


def test_round_bf16_matches_torch():
    torch = pytest.importorskip("torch")
    x = synth.normal(5, "bf16_check", 4096).astype(np.float32) * 3.0
    x[:4] = [1.00390625, 1.01171875, -1.00390625, 0.0]   # exact ties: round to even
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(synth.round_bf16(x), ref)
    assert np.array_equal(synth.round_bf16(synth.round_bf16(x)), synth.round_bf16(x))


def test_streams_are_deterministic_and_independent():
    a = synth.uniform(1, "s", 1000)
    assert np.array_equal(a, synth.uniform(1, "s", 1000))
    assert not np.allclose(a, synth.uniform(2, "s", 1000))
    assert not np.allclose(a, synth.uniform(1, "t", 1000))
    assert 0.0 <= a.min() and a.max() < 1.0
    # a prefix of a longer draw is the shorter draw (counter-based)
    assert np.array_equal(synth.uniform(1, "s", 10), a[:10])
    n = synth.normal(3, "n", 200000)
    assert abs(n.mean()) < 0.01 and abs(n.std() - 1.0) < 0.01


def test_prompt_and_length_ranges():
    ph, ac = synth.make_prompt(7, 50, 300, 512)
    assert ph.shape == (50,) and ac.shape == (300,)
    assert 0 <= ph.min() and ph.max() < 512 and 0 <= ac.min() and ac.max() < 1024
    lens = [synth.make_lengths(i, 32, 128, "serve_phonemes") for i in range(400)]
    assert min(lens) >= 32 and max(lens) <= 128 and len(set(lens)) > 50


def test_weight_recipe():
    w = synth.make_weights(synth.TINY_BF16)
    shapes = synth.weight_shapes(synth.TINY_BF16)
    assert set(w) == set(synth.weight_names(synth.TINY_BF16))
    for name, arr in w.items():
        assert arr.shape == shapes[name] and arr.dtype == np.float32
        if synth.is_matrix(name):
            assert np.array_equal(synth.round_bf16(arr), arr), name   # bf16-representable
    g = w["layers.0.ln1_g"]
    assert abs(g.mean() - 1.0) < 0.01 and abs(g.std() - 0.02) < 0.005
    wq = w["layers.0.wqkv"]
    assert abs(wq.std() - 0.02) < 0.001
    b = w["b_heads"]
    assert (b[:, synth.TINY_BF16.eos_id] < -3.5).all()   # the EOS bias keeps EOS rare
