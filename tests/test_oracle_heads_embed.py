"""Pins of the oracle's heads (Sec. III-B) and of its embedding-table choice (Sec. III-A).

Both functions are checked against closed forms computed here with scalar
arithmetic, on weights built so that every term of the definition leaves a
distinct trace:

  * heads: z = LN_f(h) with h = a * (+1, -1, +1, ...) has the closed form
    z_c = s_c a / sqrt(a^2 + eps) g_c + b_c; head i's row j selects one
    coordinate of z (a different coordinate per head), so
    logits[i][j] = z[(3 j + i) mod d] + b_heads[i][j];
  * embedding: with every block matrix and bias zero the decoder is the
    identity, so its output is the embedding itself, tok_phone[id] + PE(p)
    on the phoneme span and tok_codec[id] + PE(p) on the codec span, PE the
    sinusoid written out with math.sin / math.cos.

Each pin is also run on planted mistakes (LN_f skipped, head i reading head
i + 1's matrix, the bias dropped, the two tables swapped or shared) and must
reject every one of them.
"""
import dataclasses
import math

import numpy as np
import pytest

import synth
from oracle import model as M
from oracle import select as S
from oracle.mtp import MTPOracle

CFG = synth.ModelConfig(layers=2, d_model=64, n_attn_heads=2, d_ffn=128, phone_vocab=16,
                        codec_vocab=16, eos_id=15, n_heads_max=4, top_k_max=4, weight_dtype="f32")
A = 3.0  # amplitude of the alternating hidden state


def _head_weights():
    d, V, nh = CFG.d_model, CFG.codec_vocab, CFG.n_heads_max
    w = {k: np.asarray(v, np.float64) for k, v in synth.make_weights(CFG).items()}
    w["lnf_g"] = np.linspace(0.5, 1.5, d)
    w["lnf_b"] = np.linspace(-0.3, 0.2, d)
    wh = np.zeros((nh, V, d))
    for i in range(nh):
        for j in range(V):
            wh[i, j, (3 * j + i) % d] = 1.0
    w["w_heads"] = wh
    w["b_heads"] = 0.01 * np.arange(nh * V, dtype=np.float64).reshape(nh, V)
    return w


def _hidden():
    return np.array([A if c % 2 == 0 else -A for c in range(CFG.d_model)])


def _expected_head_logits(w, n):
    d, V = CFG.d_model, CFG.codec_vocab
    scale = A / math.sqrt(A * A + CFG.ln_eps)
    z = [(1.0 if c % 2 == 0 else -1.0) * scale * w["lnf_g"][c] + w["lnf_b"][c] for c in range(d)]
    return np.array([[z[(3 * j + i) % d] + w["b_heads"][i][j] for j in range(V)] for i in range(n)])


def _head_pin_holds(fn) -> bool:
    w = _head_weights()
    got = fn(_hidden(), w, CFG.n_heads_max, CFG.ln_eps)
    return got.shape == (CFG.n_heads_max, CFG.codec_vocab) and bool(
        np.allclose(got, _expected_head_logits(w, CFG.n_heads_max), rtol=0, atol=1e-12))


def test_head_logits_closed_form():
    assert _head_pin_holds(S.head_logits)


def test_head_logits_first_n_heads_only():
    w = _head_weights()
    got = S.head_logits(_hidden(), w, 2, CFG.ln_eps)
    assert np.allclose(got, _expected_head_logits(w, 2), rtol=0, atol=1e-12)


def _no_lnf(h, w, n, eps):
    return np.stack([w["w_heads"][i] @ np.asarray(h, np.float64) + w["b_heads"][i] for i in range(n)])


def _next_head(h, w, n, eps):
    shifted = dict(w, w_heads=np.roll(w["w_heads"], -1, axis=0))
    return S.head_logits(h, shifted, n, eps)


def _no_bias(h, w, n, eps):
    return S.head_logits(h, dict(w, b_heads=np.zeros_like(w["b_heads"])), n, eps)


def _no_affine(h, w, n, eps):
    return S.head_logits(h, dict(w, lnf_g=np.ones_like(w["lnf_g"]), lnf_b=np.zeros_like(w["lnf_b"])), n, eps)


def _transposed_rows(h, w, n, eps):
    # a head matrix read as [d][V] instead of [V][d] (only shape-compatible on a square slice)
    z = M.layer_norm(np.asarray(h, np.float64), w["lnf_g"], w["lnf_b"], eps)
    V = w["w_heads"].shape[1]
    return np.stack([w["w_heads"][i][:, :V].T @ z[:V] + w["b_heads"][i] for i in range(n)])


@pytest.mark.parametrize("planted", [_no_lnf, _next_head, _no_bias, _no_affine, _transposed_rows])
def test_head_pin_rejects_planted_mistakes(planted):
    assert not _head_pin_holds(planted)


# ---- embedding: phoneme ids read tok_phone, codec ids read tok_codec ----

def _identity_block_weights():
    w = {k: np.array(v, np.float64) for k, v in synth.make_weights(CFG).items()}
    for name in list(w):
        leaf = name.split(".")[-1]
        if name.startswith("layers.") and leaf in ("wqkv", "bqkv", "wo", "bo", "w1", "b1", "w2", "b2"):
            w[name] = np.zeros_like(w[name])
    # two clearly different tables of the same shape, so a swap stays in range
    d = CFG.d_model
    w["tok_phone"] = 1.0 + 0.001 * np.arange(CFG.phone_vocab * d, dtype=np.float64).reshape(-1, d)
    w["tok_codec"] = -1.0 - 0.002 * np.arange(CFG.codec_vocab * d, dtype=np.float64).reshape(-1, d)
    return w


def _pe(p, d):
    row = []
    for c in range(d):
        freq = 10000.0 ** (-(2 * (c // 2)) / d)
        row.append(math.sin(p * freq) if c % 2 == 0 else math.cos(p * freq))
    return np.array(row)


PH = [5, 2, 7, 2]
AC = [3, 9, 1, 0, 12]


def _expected_rows(w):
    d = CFG.d_model
    rows = [w["tok_phone"][t] + _pe(p, d) for p, t in enumerate(PH)]
    rows += [w["tok_codec"][t] + _pe(len(PH) + p, d) for p, t in enumerate(AC)]
    return np.stack(rows)


def _embed_pin_holds(w_used) -> bool:
    w = _identity_block_weights()
    dec = M.ARDecoder(CFG, w_used)
    tokens = np.array(PH + AC)
    is_phone = np.arange(len(tokens)) < len(PH)
    out = dec.forward(tokens, is_phone, dec.new_cache())
    return bool(np.allclose(out, _expected_rows(w), rtol=0, atol=1e-9))


def test_identity_blocks_return_the_embedding():
    assert _embed_pin_holds(_identity_block_weights())


def test_prefill_keeps_the_last_codec_row():
    w = _identity_block_weights()
    o = MTPOracle(CFG, w)
    o.prefill(PH, AC, 4)
    assert np.allclose(o.h_last, _expected_rows(w)[-1], rtol=0, atol=1e-9)
    # a fed codec token embeds through the codec table at the next position
    o.feed([6])
    expect = w["tok_codec"][6] + _pe(len(PH) + len(AC), CFG.d_model)
    assert np.allclose(o.h_last, expect, rtol=0, atol=1e-9)


@pytest.mark.parametrize("variant", ["swapped", "phone_shared", "codec_shared"])
def test_embed_pin_rejects_planted_tables(variant):
    w = _identity_block_weights()
    if variant == "swapped":
        w = dict(w, tok_phone=w["tok_codec"], tok_codec=w["tok_phone"])
    elif variant == "phone_shared":
        w = dict(w, tok_codec=w["tok_phone"])
    else:
        w = dict(w, tok_phone=w["tok_codec"])
    assert not _embed_pin_holds(w)


def test_embed_pin_rejects_a_shifted_position():
    w = _identity_block_weights()
    tokens = np.array(PH + AC)
    is_phone = np.arange(len(tokens)) < len(PH)
    dec = M.ARDecoder(CFG, w)
    shifted = dec.embed(tokens, is_phone, np.arange(len(tokens)) + 1)
    assert not np.allclose(shifted, _expected_rows(w), rtol=0, atol=1e-9)
