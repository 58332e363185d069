"""Oracle pin: the decoder's block stack (Sec. III-A, Eq. 1) against PyTorch's pre-LN
transformer encoder layer, an implementation of the same textbook block that shares no
code with the oracle.

The paper does not print the block's internals; the reading both sides use is the
standard pre-LN layer: x += W_o MHA(LN1 x) + b_o, then x += W_2 GELU(W_1 LN2 x + b_1) + b_2,
with exact-erf GELU, causal attention scaled by 1/sqrt(head_dim), biased linears and the
LayerNorm eps of the config.  torch.nn.TransformerEncoderLayer(norm_first=True) computes
exactly that; loaded with the oracle's weights (q, k, v row blocks stacked as its in_proj,
each head a contiguous 64-wide chunk) and run over a prompt with a causal mask, it must give
ARDecoder.forward's hidden states to float64 rounding, for a whole prompt and for a prompt
fed in chunks through the cache.  Planted mistakes in the oracle (a transposed W_o, heads
split across the wrong axis, the tanh GELU, LN2 skipped) must break the agreement.
"""
import math

import numpy as np
import pytest

import synth
from oracle import model as M

torch = pytest.importorskip("torch")

MODEL = synth.TINY
TOL = 1e-9  # float64 on both sides; different summation orders


def _prompt():
    ph, ac = synth.make_prompt(3, 12, 21, MODEL.phone_vocab)
    tokens = np.concatenate([ph, ac]).astype(np.int64)
    is_phone = np.arange(tokens.shape[0]) < ph.shape[0]
    return tokens, is_phone


def _torch_layers(w):
    c = MODEL
    layers = []
    for l in range(c.layers):
        p = f"layers.{l}."
        layer = torch.nn.TransformerEncoderLayer(c.d_model, c.n_attn_heads, c.d_ffn, dropout=0.0,
                                                 activation="gelu", layer_norm_eps=c.ln_eps, batch_first=True,
                                                 norm_first=True, dtype=torch.float64)
        t = lambda name: torch.from_numpy(np.asarray(w[p + name], dtype=np.float64))  # noqa: E731
        with torch.no_grad():
            layer.self_attn.in_proj_weight.copy_(t("wqkv"))
            layer.self_attn.in_proj_bias.copy_(t("bqkv"))
            layer.self_attn.out_proj.weight.copy_(t("wo"))
            layer.self_attn.out_proj.bias.copy_(t("bo"))
            layer.linear1.weight.copy_(t("w1"))
            layer.linear1.bias.copy_(t("b1"))
            layer.linear2.weight.copy_(t("w2"))
            layer.linear2.bias.copy_(t("b2"))
            layer.norm1.weight.copy_(t("ln1_g"))
            layer.norm1.bias.copy_(t("ln1_b"))
            layer.norm2.weight.copy_(t("ln2_g"))
            layer.norm2.bias.copy_(t("ln2_b"))
        layer.train()  # dropout 0: the standard (non-fused) path of the layer
        layers.append(layer)
    return layers


def _torch_forward(layers, x0):
    T = x0.shape[0]
    mask = torch.triu(torch.full((T, T), float("-inf"), dtype=torch.float64), diagonal=1)
    x = torch.from_numpy(x0)[None]
    with torch.no_grad():
        for layer in layers:
            x = layer(x, src_mask=mask)
    return x[0].numpy()


@pytest.fixture(scope="module")
def setup():
    w = synth.make_weights(MODEL)
    tokens, is_phone = _prompt()
    dec = M.ARDecoder(MODEL, w)
    x0 = dec.embed(tokens, is_phone, np.arange(tokens.shape[0]))
    ref = _torch_forward(_torch_layers(w), x0)
    return w, tokens, is_phone, ref


def test_block_stack_equals_torch_pre_ln_layers(setup):
    w, tokens, is_phone, ref = setup
    dec = M.ARDecoder(MODEL, w)
    out = dec.forward(tokens, is_phone, dec.new_cache())
    assert np.abs(out - ref).max() <= TOL * max(1.0, np.abs(ref).max())
    assert np.abs(ref).max() > 0.1  # the comparison is not on vanishing values


def test_chunked_prompt_through_the_cache_equals_torch(setup):
    w, tokens, is_phone, ref = setup
    dec = M.ARDecoder(MODEL, w)
    cache = dec.new_cache()
    outs = [dec.forward(tokens[a:b], is_phone[a:b], cache) for a, b in ((0, 7), (7, 8), (8, 20), (20, 33))]
    assert np.abs(np.concatenate(outs) - ref).max() <= TOL * max(1.0, np.abs(ref).max())


class _TransposedWo(M.ARDecoder):
    def block(self, layer, x, positions, cache):
        p = f"layers.{layer}."
        saved = self.w[p + "wo"]
        self.w[p + "wo"] = saved.T.copy()
        try:
            return super().block(layer, x, positions, cache)
        finally:
            self.w[p + "wo"] = saved


class _HeadsAcrossDims(M.ARDecoder):
    """Heads taken as strided rather than contiguous chunks of q, k and v."""

    def block(self, layer, x, positions, cache):
        c, w, p = self.cfg, self.w, f"layers.{layer}."
        m, d = x.shape
        H, hd = c.n_attn_heads, d // c.n_attn_heads
        h = M.layer_norm(x, w[p + "ln1_g"], w[p + "ln1_b"], c.ln_eps)
        qkv = h @ w[p + "wqkv"].T + w[p + "bqkv"]
        split = [qkv[:, i * d:(i + 1) * d].reshape(m, hd, H).transpose(0, 2, 1) for i in range(3)]
        cache.append(layer, split[1], split[2])
        att = M.causal_attention(split[0], cache.k[layer], cache.v[layer], positions,
                                 np.arange(cache.k[layer].shape[0]))
        x = x + att.transpose(0, 2, 1).reshape(m, d) @ w[p + "wo"].T + w[p + "bo"]
        h = M.layer_norm(x, w[p + "ln2_g"], w[p + "ln2_b"], c.ln_eps)
        return x + M.gelu(h @ w[p + "w1"].T + w[p + "b1"]) @ w[p + "w2"].T + w[p + "b2"]


class _TanhGelu(M.ARDecoder):
    def block(self, layer, x, positions, cache):
        keep = M.gelu
        M.gelu = lambda z: 0.5 * z * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (z + 0.044715 * z ** 3)))
        try:
            return super().block(layer, x, positions, cache)
        finally:
            M.gelu = keep


class _NoLn2(M.ARDecoder):
    def block(self, layer, x, positions, cache):
        keep = M.layer_norm
        calls = []

        def ln(v, g, b, eps):
            calls.append(1)
            return keep(v, g, b, eps) if len(calls) == 1 else v
        M.layer_norm = ln
        try:
            return super().block(layer, x, positions, cache)
        finally:
            M.layer_norm = keep


@pytest.mark.parametrize("variant", [_TransposedWo, _HeadsAcrossDims, _TanhGelu, _NoLn2])
def test_planted_mistakes_break_the_agreement(setup, variant):
    w, tokens, is_phone, ref = setup
    dec = variant(MODEL, w)
    out = dec.forward(tokens, is_phone, dec.new_cache())
    assert np.abs(out - ref).max() > 1e3 * TOL * max(1.0, np.abs(ref).max())
