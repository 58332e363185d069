"""Oracle: the autoregressive codec-token decoder theta_AR (Sec. III-A, Eq. 1).

Test infrastructure only (see oracle/__init__.py).  Float64 throughout.

Readings of the paper (it is silent on the block internals):
  * Sec. III-A: phonemes, acoustic prompt and generated codes are concatenated
    into one sequence with no separator; phonemes embed through their own
    table, codec ids (prompt and generated) through the codec table.
  * positions: sinusoidal absolute encoding over the one continuous index
    0..T-1, added to the token embedding;
  * attention: fully causal over the whole sequence, scale 1/sqrt(head_dim);
  * block: pre-LN, x += W_o MHA(LN1 x) + b_o ; x += W_2 GELU(W_1 LN2 x + b_1) + b_2,
    exact erf GELU, LayerNorm eps from the config (1e-5), biased linears;
  * the final LayerNorm LN_f is applied by the heads (select.py), not here.

Parity pins (tests/test_oracle_model.py): sinusoid closed forms and the
angle-addition identity; LayerNorm moments; GELU against printed normal-CDF
values; attention special cases (one key returns v, zero query averages,
future keys have no effect); the block with zeroed weights is the identity
plus biases; a one-token block against its closed form; cached chunked decode
against a cache-free full recompute; invariance to permutations of the
attention heads, of the FFN units and of the dimensions within a head (which
a transposed operand or a wrong head layout breaks); with every block matrix
and bias zero the decoder returns tok_phone[id] + PE(p) on the phoneme span
and tok_codec[id] + PE(p) on the codec span, the sinusoid written out in
scalar form (tests/test_oracle_heads_embed.py; swapped or shared tables
rejected); the whole block stack against PyTorch's pre-LN transformer
encoder layer (torch.nn.TransformerEncoderLayer, norm_first, exact GELU)
loaded with the same weights, for a whole prompt and a prompt fed in chunks
through the cache, to float64 rounding (tests/test_oracle_block_torch.py;
a transposed W_o, heads split across the wrong axis, the tanh GELU and a
skipped LN2 rejected).  No pin ties the block to printed values: the paper
prints no activation, logit or worked example of the model, so what these
pins fix is the reading above, not numbers from the paper.
"""
from __future__ import annotations

import math

import numpy as np
from scipy.special import erf


def sinusoidal_position(positions: np.ndarray, d: int) -> np.ndarray:
    """PE[p, 2i] = sin(p / 10000^(2i/d)), PE[p, 2i+1] = cos(p / 10000^(2i/d))."""
    positions = np.asarray(positions, dtype=np.float64)
    i = np.arange(d // 2, dtype=np.float64)
    inv_freq = 1.0 / np.power(10000.0, 2.0 * i / d)
    angle = positions[:, None] * inv_freq[None, :]
    pe = np.empty((positions.shape[0], d), dtype=np.float64)
    pe[:, 0::2] = np.sin(angle)
    pe[:, 1::2] = np.cos(angle)
    return pe


def layer_norm(x: np.ndarray, g: np.ndarray, b: np.ndarray, eps: float) -> np.ndarray:
    """(x - mean) / sqrt(var + eps) * g + b over the last axis (biased variance)."""
    mean = x.mean(axis=-1, keepdims=True)
    var = ((x - mean) ** 2).mean(axis=-1, keepdims=True)
    return (x - mean) / np.sqrt(var + eps) * g + b


def gelu(x: np.ndarray) -> np.ndarray:
    """Exact GELU: x * Phi(x) = 0.5 x (1 + erf(x / sqrt 2))."""
    return 0.5 * x * (1.0 + erf(x / math.sqrt(2.0)))


def causal_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray,
                     q_pos: np.ndarray, k_pos: np.ndarray) -> np.ndarray:
    """Multi-head attention of queries [m, H, hd] over keys/values [T, H, hd].

    Query j sees exactly the keys with k_pos <= q_pos[j]; weights are the
    softmax of q.k / sqrt(hd) over those keys."""
    m, n_heads, hd = q.shape
    out = np.zeros((m, n_heads, hd), dtype=np.float64)
    scale = 1.0 / math.sqrt(hd)
    for j in range(m):
        visible = k_pos <= q_pos[j]
        for h in range(n_heads):
            s = (k[visible, h, :] @ q[j, h, :]) * scale
            w = np.exp(s - s.max())
            w /= w.sum()
            out[j, h, :] = w @ v[visible, h, :]
    return out


class KVCache:
    """Per-layer keys and values of every cached position (a plain growing array)."""

    def __init__(self, layers: int, n_heads: int, hd: int):
        self.k = [np.zeros((0, n_heads, hd)) for _ in range(layers)]
        self.v = [np.zeros((0, n_heads, hd)) for _ in range(layers)]

    @property
    def length(self) -> int:
        return self.k[0].shape[0]

    def append(self, layer: int, k: np.ndarray, v: np.ndarray) -> None:
        self.k[layer] = np.concatenate([self.k[layer], k], axis=0)
        self.v[layer] = np.concatenate([self.v[layer], v], axis=0)

    def rollback(self, count: int) -> None:
        """Drop the last `count` cached positions (rejected tokens)."""
        keep = self.length - count
        assert 0 <= keep
        self.k = [k[:keep] for k in self.k]
        self.v = [v[:keep] for v in self.v]


class ARDecoder:
    """theta_AR: embeds rows of the concatenated sequence and runs the L blocks."""

    def __init__(self, cfg, weights: dict[str, np.ndarray]):
        self.cfg = cfg
        self.w = {name: np.asarray(t, dtype=np.float64) for name, t in weights.items()}

    def new_cache(self) -> KVCache:
        c = self.cfg
        return KVCache(c.layers, c.n_attn_heads, c.d_model // c.n_attn_heads)

    def embed(self, tokens: np.ndarray, is_phone: np.ndarray, positions: np.ndarray) -> np.ndarray:
        """x = E[token] + PE(position), E the phoneme or codec table (Sec. III-A)."""
        rows = np.where(is_phone[:, None], self.w["tok_phone"][np.where(is_phone, tokens, 0)],
                        self.w["tok_codec"][np.where(is_phone, 0, tokens)])
        return rows + sinusoidal_position(positions, self.cfg.d_model)

    def block(self, layer: int, x: np.ndarray, positions: np.ndarray, cache: KVCache) -> np.ndarray:
        """One pre-LN block on rows x [m, d] at `positions`; appends their K/V first."""
        c, w, p = self.cfg, self.w, f"layers.{layer}."
        m, d = x.shape
        n_heads, hd = c.n_attn_heads, d // c.n_attn_heads
        h = layer_norm(x, w[p + "ln1_g"], w[p + "ln1_b"], c.ln_eps)
        qkv = h @ w[p + "wqkv"].T + w[p + "bqkv"]
        q = qkv[:, 0:d].reshape(m, n_heads, hd)
        k = qkv[:, d:2 * d].reshape(m, n_heads, hd)
        v = qkv[:, 2 * d:3 * d].reshape(m, n_heads, hd)
        cache.append(layer, k, v)
        k_pos = np.arange(cache.k[layer].shape[0])
        att = causal_attention(q, cache.k[layer], cache.v[layer], positions, k_pos)
        x = x + att.reshape(m, d) @ w[p + "wo"].T + w[p + "bo"]
        h = layer_norm(x, w[p + "ln2_g"], w[p + "ln2_b"], c.ln_eps)
        u = gelu(h @ w[p + "w1"].T + w[p + "b1"])
        return x + u @ w[p + "w2"].T + w[p + "b2"]

    def forward(self, tokens, is_phone, cache: KVCache) -> np.ndarray:
        """Hidden states [m, d] (before LN_f) of the next m rows of the sequence.

        The rows take positions cache.length .. cache.length + m - 1."""
        tokens = np.asarray(tokens, dtype=np.int64)
        is_phone = np.asarray(is_phone, dtype=bool)
        positions = cache.length + np.arange(tokens.shape[0])
        x = self.embed(tokens, is_phone, positions)
        for layer in range(self.cfg.layers):
            x = self.block(layer, x, positions, cache)
        return x
