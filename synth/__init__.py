"""Seeded synthetic inputs shared by the CUDA path's tests/bench and the CPU oracle.

This module holds no arithmetic of the method (no model step, no heads, no
Viterbi).  It only draws numbers: model weights, prompts, a token-transition
matrix and standalone candidate lattices, all from a counter-based generator so
that the same (seed, name, index) gives the same value on any machine.

Generator: the SplitMix64 output function (Steele, Lea, Flood, "Fast
splittable pseudorandom number generators", OOPSLA 2014) applied to a counter.
Element i of stream (seed, name) is mix64(key + (i + 1) * GAMMA) with
key = mix64(seed * GAMMA ^ fnv1a64(name)).  Uniforms take the top 53 bits;
normals use both branches of the Box-Muller transform on each pair of uniforms.

Recipe (the paper trains on LibriTTS with SpeechTokenizer codes, Sec. IV-A;
none of that data or any trained weight is available, so these stand in):
  * every matrix, embedding and bias ~ N(0, 0.02); LayerNorm gain 1 + N(0, 0.02),
    LayerNorm bias N(0, 0.02); for bf16 models, matrices and embeddings are
    rounded to bf16 (round-to-nearest-even) and the rounded values are the
    weights both sides use;
  * prompts: phoneme ids uniform in [0, phone_vocab), acoustic ids uniform in
    [0, 1024), seeded 1000 + sequence index;
  * the transition matrix Q of Sec. III-C ("derived from the dataset") is
    synthetic: Q[i, :] proportional to exp(g[i, :]) + beta_i * e_i with
    g ~ N(0, 1) and beta_i chosen so the self-transition mass is about 0.3,
    mimicking that consecutive speech tokens are often alike (Sec. I);
  * EOS: with random weights EOS would be as likely as any code and would cut
    generations short of the fixed lengths the workloads ask for, so the EOS
    logit of every head gets an extra bias EOS_BIAS = -4 (about 6 logit
    standard deviations at d = 1024); tests that need EOS raise it instead.
"""
from __future__ import annotations

import dataclasses
import functools
import math

import numpy as np

EOS_BIAS = -4.0

_GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)


def _mix64(z: np.ndarray) -> np.ndarray:
    z = (z ^ (z >> np.uint64(30))) * _M1
    z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def _fnv1a64(name: str) -> int:
    h = 0xCBF29CE484222325
    for byte in name.encode("utf-8"):
        h ^= byte
        h = (h * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    return h


def _stream_key(seed: int, name: str) -> np.uint64:
    with np.errstate(over="ignore"):
        base = np.uint64((seed * 0x9E3779B97F4A7C15) & 0xFFFFFFFFFFFFFFFF)
        return _mix64(np.array([base ^ np.uint64(_fnv1a64(name))], dtype=np.uint64))[0]


def uint64s(seed: int, name: str, count: int, offset: int = 0) -> np.ndarray:
    """`count` raw 64-bit draws of stream (seed, name), starting at index `offset`."""
    key = _stream_key(seed, name)
    idx = np.arange(offset + 1, offset + count + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return _mix64(key + idx * _GAMMA)


def uniform(seed: int, name: str, count: int) -> np.ndarray:
    """Uniform doubles in [0, 1)."""
    return (uint64s(seed, name, count) >> np.uint64(11)).astype(np.float64) * (2.0 ** -53)


def normal(seed: int, name: str, count: int) -> np.ndarray:
    """Standard normal doubles: Box-Muller on draw pairs (2p, 2p+1) gives elements 2p, 2p+1."""
    pairs = (count + 1) // 2
    out = np.empty(2 * pairs, dtype=np.float64)
    key = _stream_key(seed, name)
    chunk = 1 << 18
    with np.errstate(over="ignore"):
        for start in range(0, pairs, chunk):
            stop = min(pairs, start + chunk)
            idx = np.arange(2 * start + 1, 2 * stop + 1, dtype=np.uint64)
            u = (_mix64(key + idx * _GAMMA) >> np.uint64(11)).astype(np.float64) * (2.0 ** -53)
            r = np.sqrt(-2.0 * np.log(1.0 - u[0::2]))     # 1 - u in (0, 1]
            theta = (2.0 * math.pi) * u[1::2]
            out[2 * start:2 * stop:2] = r * np.cos(theta)
            out[2 * start + 1:2 * stop:2] = r * np.sin(theta)
    return out[:count]


def integers(seed: int, name: str, count: int, lo: int, hi: int) -> np.ndarray:
    """Integers uniform in [lo, hi) as int32."""
    u = uniform(seed, name, count)
    return (lo + np.floor(u * (hi - lo))).astype(np.int64).clip(lo, hi - 1).astype(np.int32)


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bf16 (ties to even); returns fp32 holding them."""
    bits = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    lsb = (bits >> np.uint64(16)) & np.uint64(1)
    bits = (bits + np.uint64(0x7FFF) + lsb) & np.uint64(0xFFFF0000)
    return bits.astype(np.uint32).view(np.float32).reshape(np.shape(x))


@dataclasses.dataclass(frozen=True)
class ModelConfig:
    """Shape of the AR decoder with MTP heads (field names follow include/mtp.h)."""
    layers: int
    d_model: int
    n_attn_heads: int
    d_ffn: int
    phone_vocab: int
    codec_vocab: int = 1025          # 1024 codec ids + EOS
    eos_id: int = 1024
    n_heads_max: int = 8
    top_k_max: int = 32
    weight_dtype: str = "bf16"       # "f32" or "bf16" for matrices and embeddings
    ln_eps: float = 1e-5

    @property
    def head_dim(self) -> int:
        return self.d_model // self.n_attn_heads


TINY = ModelConfig(layers=2, d_model=256, n_attn_heads=4, d_ffn=1024, phone_vocab=128,
                   weight_dtype="f32")
VALLE = ModelConfig(layers=12, d_model=1024, n_attn_heads=16, d_ffn=4096, phone_vocab=512,
                    weight_dtype="bf16")
# the tiny model with bf16 matrices: small batched-path (tensor-core) parity cases
TINY_BF16 = ModelConfig(layers=2, d_model=256, n_attn_heads=4, d_ffn=1024, phone_vocab=128,
                        weight_dtype="bf16")


def weight_names(cfg: ModelConfig) -> list[str]:
    """Tensor order of the weight blob (include/mtp.h documents the same order)."""
    names = ["tok_phone", "tok_codec"]
    for layer in range(cfg.layers):
        p = f"layers.{layer}."
        names += [p + s for s in ("ln1_g", "ln1_b", "wqkv", "bqkv", "wo", "bo",
                                  "ln2_g", "ln2_b", "w1", "b1", "w2", "b2")]
    names += ["lnf_g", "lnf_b", "w_heads", "b_heads", "log_q"]
    return names


def weight_shapes(cfg: ModelConfig) -> dict[str, tuple[int, ...]]:
    d, f, v = cfg.d_model, cfg.d_ffn, cfg.codec_vocab
    shapes = {"tok_phone": (cfg.phone_vocab, d), "tok_codec": (v, d)}
    for layer in range(cfg.layers):
        p = f"layers.{layer}."
        shapes.update({p + "ln1_g": (d,), p + "ln1_b": (d,), p + "wqkv": (3 * d, d),
                       p + "bqkv": (3 * d,), p + "wo": (d, d), p + "bo": (d,),
                       p + "ln2_g": (d,), p + "ln2_b": (d,), p + "w1": (f, d),
                       p + "b1": (f,), p + "w2": (d, f), p + "b2": (d,)})
    shapes.update({"lnf_g": (d,), "lnf_b": (d,), "w_heads": (cfg.n_heads_max, v, d),
                   "b_heads": (cfg.n_heads_max, v), "log_q": (v, v)})
    return shapes


def is_matrix(name: str) -> bool:
    """Matrices and embeddings are stored in the model's weight dtype; the rest in fp32."""
    leaf = name.split(".")[-1]
    return leaf in ("tok_phone", "tok_codec", "wqkv", "wo", "w1", "w2", "w_heads")


def transition_log_q(v: int, seed: int = 7, self_mass: float = 0.3) -> np.ndarray:
    """Synthetic log Q [v, v] (fp32); rows of Q sum to 1 in float64 before the log."""
    g = normal(seed, "transition_g", v * v).reshape(v, v)
    e = np.exp(g)
    row = e.sum(axis=1)
    beta = self_mass / (1.0 - self_mass) * row
    q = e / (row + beta)[:, None]
    q[np.arange(v), np.arange(v)] += beta / (row + beta)
    return np.log(q).astype(np.float32)


@functools.lru_cache(maxsize=4)
def _weights_cached(cfg: ModelConfig, seed: int, eos_bias: float) -> tuple:
    shapes = weight_shapes(cfg)
    out = {}
    for name in weight_names(cfg):
        shape = shapes[name]
        count = int(np.prod(shape))
        if name == "log_q":
            out[name] = transition_log_q(cfg.codec_vocab)
            continue
        w = 0.02 * normal(seed, name, count)
        if name.endswith("_g"):
            w = 1.0 + w
        w = w.astype(np.float32).reshape(shape)
        if name == "b_heads" and eos_bias != 0.0:
            w[:, cfg.eos_id] += np.float32(eos_bias)
        if cfg.weight_dtype == "bf16" and is_matrix(name):
            w = round_bf16(w)
        w.setflags(write=False)
        out[name] = w
    return tuple(out.items())


def make_weights(cfg: ModelConfig, seed: int = 0, eos_bias: float = EOS_BIAS) -> dict[str, np.ndarray]:
    """All weights of `cfg` as read-only fp32 arrays (bf16-representable where bf16)."""
    return dict(_weights_cached(cfg, seed, float(eos_bias)))


def make_prompt(seq_index: int, n_phone: int, n_acoustic: int, phone_vocab: int,
                codec_ids: int = 1024) -> tuple[np.ndarray, np.ndarray]:
    """Phoneme ids and acoustic-prompt codec ids of one sequence (seed 1000 + index)."""
    seed = 1000 + seq_index
    ph = integers(seed, "phonemes", n_phone, 0, phone_vocab)
    ac = integers(seed, "acoustic", n_acoustic, 0, codec_ids)
    return ph, ac


def make_lengths(seq_index: int, lo: int, hi: int, name: str) -> int:
    """One integer uniform in [lo, hi] (inclusive), seeded 2000 + index."""
    return int(integers(2000 + seq_index, name, 1, lo, hi + 1)[0])


def make_lattice(batch: int, n: int, k: int, vocab: int, seed: int,
                 quantum: float = 0.0) -> tuple[np.ndarray, np.ndarray]:
    """Standalone candidate lattices: ids [B, n, k] distinct per (b, t), log-scores [B, n, k].

    Scores are log-uniform draws sorted in descending order, as the top-k of a
    distribution would be.  With `quantum` > 0 they are rounded to multiples of
    it, which makes ties frequent (for tie-break tests)."""
    u = uniform(seed, "lattice_ids", batch * n * vocab).reshape(batch, n, vocab)
    ids = np.argsort(u, axis=2, kind="stable")[:, :, :k].astype(np.int32)
    s = np.log(1.0 - uniform(seed, "lattice_scores", batch * n * k)).reshape(batch, n, k)
    s = -np.sort(-s, axis=2)
    if quantum > 0.0:
        s = np.round(s / quantum) * quantum
    return ids, s.astype(np.float32)


def make_hidden(batch: int, d: int, seed: int) -> np.ndarray:
    """Hidden states N(0, 1) [batch, d] rounded to bf16 (head microbenchmark input)."""
    return round_bf16(normal(seed, "hidden", batch * d).astype(np.float32).reshape(batch, d))
