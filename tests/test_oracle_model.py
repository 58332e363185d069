"""Pins of the oracle's decoder (Sec. III-A, Eq. 1) by closed forms and special cases."""
import math

import numpy as np
import pytest

import synth
from oracle import model as M


def test_sinusoid_closed_forms():
    d = 64
    pe = M.sinusoidal_position(np.array([0, 1, 7, 500]), d)
    assert np.array_equal(pe[0, 0::2], np.zeros(d // 2))
    assert np.array_equal(pe[0, 1::2], np.ones(d // 2))
    assert pe[2, 0] == pytest.approx(math.sin(7.0), abs=1e-15)
    assert pe[2, 1] == pytest.approx(math.cos(7.0), abs=1e-15)
    # the slowest pair turns at 10000^(-(d-2)/d) radians per position
    assert pe[3, d - 2] == pytest.approx(math.sin(500 * 10000.0 ** (-(d - 2) / d)), abs=1e-12)


def test_sinusoid_angle_addition():
    d, p, q = 32, 37, 91
    a, b, ab = M.sinusoidal_position(np.array([p, q, p + q]), d)
    sin_ab = a[0::2] * b[1::2] + a[1::2] * b[0::2]
    cos_ab = a[1::2] * b[1::2] - a[0::2] * b[0::2]
    assert np.allclose(ab[0::2], sin_ab, atol=1e-12)
    assert np.allclose(ab[1::2], cos_ab, atol=1e-12)


def test_layer_norm_moments_and_scale_invariance():
    x = synth.normal(3, "ln", 5 * 96).reshape(5, 96) * 3.0 + 2.0
    y = M.layer_norm(x, np.ones(96), np.zeros(96), 0.0)
    assert np.allclose(y.mean(axis=1), 0.0, atol=1e-12)
    assert np.allclose(y.var(axis=1), 1.0, atol=1e-12)
    assert np.allclose(M.layer_norm(7.5 * x - 3.0, np.ones(96), np.zeros(96), 0.0), y, atol=1e-12)
    g, b = np.linspace(0.5, 2.0, 96), np.linspace(-1, 1, 96)
    assert np.allclose(M.layer_norm(x, g, b, 0.0), y * g + b, atol=1e-12)


def test_gelu_against_normal_cdf_table():
    # Phi(1) = 0.8413447460685429, Phi(-1) = 0.15865525393145707, Phi(2) = 0.9772498680518208
    x = np.array([0.0, 1.0, -1.0, 2.0])
    expect = np.array([0.0, 0.8413447460685429, -0.15865525393145707, 2 * 0.9772498680518208])
    assert np.allclose(M.gelu(x), expect, atol=1e-14)


def test_attention_special_cases():
    h, hd = 3, 8
    rng_q = synth.normal(4, "q", 4 * h * hd).reshape(4, h, hd)
    k = synth.normal(4, "k", 6 * h * hd).reshape(6, h, hd)
    v = synth.normal(4, "v", 6 * h * hd).reshape(6, h, hd)
    kpos = np.arange(6)
    # one visible key returns its value
    out = M.causal_attention(rng_q[:1], k, v, np.array([0]), kpos)
    assert np.allclose(out[0], v[0], atol=1e-14)
    # a zero query weighs the visible keys equally
    out = M.causal_attention(np.zeros((1, h, hd)), k, v, np.array([3]), kpos)
    assert np.allclose(out[0], v[:4].mean(axis=0), atol=1e-14)
    # keys after the query's position change nothing
    k2, v2 = k.copy(), v.copy()
    k2[4:] += 100.0
    v2[4:] -= 50.0
    a = M.causal_attention(rng_q, k, v, np.array([0, 1, 2, 3]), kpos)
    b = M.causal_attention(rng_q, k2, v2, np.array([0, 1, 2, 3]), kpos)
    assert np.allclose(a, b, atol=1e-14)
    # a dominant score selects its key's value
    q = np.zeros((1, h, hd))
    q[0, :, 0] = 1e3
    kk = np.zeros((6, h, hd))
    kk[2, :, 0] = 1.0
    out = M.causal_attention(q, kk, v, np.array([5]), kpos)
    assert np.allclose(out[0], v[2], atol=1e-12)


def _zero_cfg_weights(cfg):
    w = {n: np.array(t, dtype=np.float64) for n, t in synth.make_weights(cfg).items()}
    return w


def test_block_with_zero_projections_adds_only_biases():
    cfg = synth.TINY
    w = _zero_cfg_weights(cfg)
    for layer in range(cfg.layers):
        p = f"layers.{layer}."
        w[p + "wo"][:] = 0.0
        w[p + "w2"][:] = 0.0
    dec = M.ARDecoder(cfg, w)
    cache = dec.new_cache()
    x = synth.normal(5, "x", 3 * cfg.d_model).reshape(3, cfg.d_model)
    y = dec.block(0, x, np.arange(3), cache)
    assert np.allclose(y, x + w["layers.0.bo"] + w["layers.0.b2"], atol=1e-14)


def test_single_token_block_closed_form():
    """With one key the attention output is v (rows 2d..3d of the QKV projection)."""
    cfg = synth.TINY
    w = _zero_cfg_weights(cfg)
    d, p = cfg.d_model, "layers.1."
    dec = M.ARDecoder(cfg, w)
    x = synth.normal(6, "x1", d)[None]
    y = dec.block(1, x, np.array([0]), dec.new_cache())
    ln1 = M.layer_norm(x, w[p + "ln1_g"], w[p + "ln1_b"], cfg.ln_eps)
    v = ln1 @ w[p + "wqkv"][2 * d:].T + w[p + "bqkv"][2 * d:]
    x1 = x + v @ w[p + "wo"].T + w[p + "bo"]
    ln2 = M.layer_norm(x1, w[p + "ln2_g"], w[p + "ln2_b"], cfg.ln_eps)
    hid = ln2 @ w[p + "w1"].T + w[p + "b1"]
    ref = x1 + M.gelu(hid) @ w[p + "w2"].T + w[p + "b2"]      # GELU pinned separately
    assert np.allclose(y, ref, atol=1e-12)


def test_zero_query_section_averages_values():
    """Zeroing the query rows (0..d) of W_qkv and their bias makes every head average v."""
    cfg = synth.TINY
    w = _zero_cfg_weights(cfg)
    d, p = cfg.d_model, "layers.0."
    w[p + "wqkv"][:d] = 0.0
    w[p + "bqkv"][:d] = 0.0
    w[p + "wo"][:] = np.eye(d)
    w[p + "bo"][:] = 0.0
    w[p + "w2"][:] = 0.0
    w[p + "b2"][:] = 0.0
    dec = M.ARDecoder(cfg, w)
    x = synth.normal(7, "x2", 5 * d).reshape(5, d)
    y = dec.block(0, x, np.arange(5), dec.new_cache())
    ln1 = M.layer_norm(x, w[p + "ln1_g"], w[p + "ln1_b"], cfg.ln_eps)
    v = ln1 @ w[p + "wqkv"][2 * d:].T + w[p + "bqkv"][2 * d:]
    mean_v = np.cumsum(v, axis=0) / np.arange(1, 6)[:, None]
    assert np.allclose(y - x, mean_v, atol=1e-12)


def test_cached_chunked_decode_equals_full_recompute(tiny_weights):
    cfg = synth.TINY
    dec = M.ARDecoder(cfg, tiny_weights)
    ph, ac = synth.make_prompt(3, 10, 20, cfg.phone_vocab)
    tokens = np.concatenate([ph, ac])
    is_phone = np.arange(30) < 10
    full = dec.forward(tokens, is_phone, dec.new_cache())
    cache = dec.new_cache()
    parts, start = [], 0
    for size in (1, 7, 3, 11, 8):
        parts.append(dec.forward(tokens[start:start + size], is_phone[start:start + size], cache))
        start += size
    assert np.allclose(np.concatenate(parts), full, atol=1e-12)


def test_rollback_then_append_equals_append(tiny_weights):
    cfg = synth.TINY
    dec = M.ARDecoder(cfg, tiny_weights)
    ph, ac = synth.make_prompt(4, 8, 12, cfg.phone_vocab)
    prompt = np.concatenate([ph, ac])
    is_phone = np.arange(20) < 8
    c1 = dec.new_cache()
    dec.forward(prompt, is_phone, c1)
    dec.forward(np.array([5, 6, 7]), np.zeros(3, bool), c1)
    c1.rollback(3)
    y1 = dec.forward(np.array([9, 10]), np.zeros(2, bool), c1)
    c2 = dec.new_cache()
    dec.forward(prompt, is_phone, c2)
    y2 = dec.forward(np.array([9, 10]), np.zeros(2, bool), c2)
    assert np.array_equal(y1, y2)


# ---- permutation invariances of the block: a transposed operand or a wrong head /
# feature layout in the oracle breaks at least one of them ----

def _forward(cfg, w, seed=11):
    dec = M.ARDecoder(cfg, w)
    ph, ac = synth.make_prompt(seed, 6, 14, cfg.phone_vocab)
    tokens = np.concatenate([ph, ac])
    return dec.forward(tokens, np.arange(20) < 6, dec.new_cache())


def _permute_heads(cfg, w, perm, fix_wo=True):
    """Heads reordered: q, k and v row blocks of W_qkv (and b_qkv) and W_o's column blocks."""
    d, H = cfg.d_model, cfg.n_attn_heads
    hd = d // H
    rows = np.concatenate([np.arange(p * hd, (p + 1) * hd) for p in perm])
    out = {k: v.copy() for k, v in w.items()}
    for layer in range(cfg.layers):
        p = f"layers.{layer}."
        idx = np.concatenate([sec * d + rows for sec in range(3)])
        out[p + "wqkv"] = w[p + "wqkv"][idx]
        out[p + "bqkv"] = w[p + "bqkv"][idx]
        if fix_wo:
            out[p + "wo"] = w[p + "wo"][:, rows]
    return out


def test_block_is_invariant_to_a_head_permutation(tiny_weights):
    cfg = synth.TINY
    perm = np.array([2, 0, 3, 1])
    base = _forward(cfg, tiny_weights)
    assert np.allclose(_forward(cfg, _permute_heads(cfg, tiny_weights, perm)), base, atol=1e-10)
    # the same reordering without W_o's columns is a different model
    assert not np.allclose(_forward(cfg, _permute_heads(cfg, tiny_weights, perm, fix_wo=False)), base, atol=1e-3)


def test_block_is_invariant_to_an_ffn_unit_permutation(tiny_weights):
    cfg = synth.TINY
    sigma = np.random.default_rng(3).permutation(cfg.d_ffn)
    w = {k: v.copy() for k, v in tiny_weights.items()}
    broken = {k: v.copy() for k, v in tiny_weights.items()}
    for layer in range(cfg.layers):
        p = f"layers.{layer}."
        w[p + "w1"] = tiny_weights[p + "w1"][sigma]
        w[p + "b1"] = tiny_weights[p + "b1"][sigma]
        w[p + "w2"] = tiny_weights[p + "w2"][:, sigma]
        broken[p + "w1"] = w[p + "w1"]
        broken[p + "b1"] = w[p + "b1"]
    base = _forward(cfg, tiny_weights)
    assert np.allclose(_forward(cfg, w), base, atol=1e-10)
    assert not np.allclose(_forward(cfg, broken), base, atol=1e-3)


def test_block_is_invariant_to_a_dimension_permutation_within_heads(tiny_weights):
    """q and k dimensions of every head reordered alike (scores unchanged); v dimensions
    reordered with W_o's matching columns (outputs unchanged)."""
    cfg = synth.TINY
    d, H = cfg.d_model, cfg.n_attn_heads
    hd = d // H
    rng = np.random.default_rng(4)
    tau, rho = rng.permutation(hd), rng.permutation(hd)
    qk = np.concatenate([h * hd + tau for h in range(H)])
    vv = np.concatenate([h * hd + rho for h in range(H)])
    w = {k: v.copy() for k, v in tiny_weights.items()}
    for layer in range(cfg.layers):
        p = f"layers.{layer}."
        idx = np.concatenate([qk, d + qk, 2 * d + vv])
        w[p + "wqkv"] = tiny_weights[p + "wqkv"][idx]
        w[p + "bqkv"] = tiny_weights[p + "bqkv"][idx]
        w[p + "wo"] = tiny_weights[p + "wo"][:, vv]
    assert np.allclose(_forward(cfg, w), _forward(cfg, tiny_weights), atol=1e-10)


def test_a_transposed_output_projection_breaks_the_head_pin(tiny_weights):
    """Planted mistake: an oracle that applies W_o untransposed (x += att W_o instead of
    att W_o^T).  It still runs, but the head-permutation invariance fails."""
    cfg = synth.TINY

    class Planted(M.ARDecoder):
        def block(self, layer, x, positions, cache):
            key = f"layers.{layer}.wo"
            wo = self.w[key]
            self.w[key] = wo.T
            try:
                return super().block(layer, x, positions, cache)
            finally:
                self.w[key] = wo

    def fwd(w):
        dec = Planted(cfg, w)
        ph, ac = synth.make_prompt(11, 6, 14, cfg.phone_vocab)
        return dec.forward(np.concatenate([ph, ac]), np.arange(20) < 6, dec.new_cache())

    perm = np.array([2, 0, 3, 1])
    assert not np.allclose(fwd(_permute_heads(cfg, tiny_weights, perm)), fwd(tiny_weights), atol=1e-3)
