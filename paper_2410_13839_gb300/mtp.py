"""Python binding of include/mtp.h: same names, argument marshalling only.

Buffers are torch tensors (device memory, from PyTorch's allocator) or numpy
arrays (host memory); streams are torch CUDA streams.  Every computation runs
in libmtp's kernels.
"""
from __future__ import annotations

import ctypes
import struct

import numpy as np

from . import _lib
from ._lib import MTP_OPT_BATCHED, MTPError, MtpAttentionArgs, MtpConfig, check, lib  # noqa: F401

BLOB_MAGIC = b"MTPWGT01"


def _ptr(x):
    """Address of a contiguous torch tensor or numpy array (None -> NULL)."""
    if x is None:
        return None
    if isinstance(x, np.ndarray):
        if not x.flags["C_CONTIGUOUS"]:
            raise ValueError("numpy buffer must be C-contiguous")
        return x.ctypes.data
    if hasattr(x, "data_ptr"):
        if not x.is_contiguous():
            raise ValueError("tensor buffer must be contiguous")
        return x.data_ptr()
    if isinstance(x, int):
        return x
    raise TypeError(f"unsupported buffer type {type(x)}")


def _stream_handle(stream) -> int | None:
    if stream is None:
        return None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def make_config(model, max_batch: int, max_ctx: int, page_size: int = 64, n_pages: int = 0,
                accept_policy: int = 0) -> MtpConfig:
    """mtp_config of a synth.ModelConfig-like object plus capacity."""
    return MtpConfig(layers=model.layers, d_model=model.d_model, n_attn_heads=model.n_attn_heads,
                     d_ffn=model.d_ffn, phone_vocab=model.phone_vocab, codec_vocab=model.codec_vocab,
                     eos_id=model.eos_id, n_heads_max=model.n_heads_max, top_k_max=model.top_k_max,
                     max_batch=max_batch, max_ctx=max_ctx, page_size=page_size, n_pages=n_pages,
                     weight_dtype=_lib.MTP_BF16 if model.weight_dtype == "bf16" else _lib.MTP_F32,
                     accept_policy=accept_policy, ln_eps=model.ln_eps)


def pack_weights(tensors: list[tuple[np.ndarray, bool]], bf16: bool) -> bytes:
    """Serialise tensors (array, is_matrix) in blob order into the mtp.h weight format.

    Matrices are written as bf16 (their values must already be bf16-exact) or
    fp32; everything else as fp32."""
    header = 24 + 16 * len(tensors)
    offset = (header + 255) // 256 * 256
    table, chunks = [], []
    for arr, is_matrix in tensors:
        a = np.ascontiguousarray(arr, dtype=np.float32)
        if bf16 and is_matrix:
            bits = a.view(np.uint32)
            if np.any(bits & 0xFFFF):
                raise ValueError("matrix values are not bf16-representable")
            raw = (bits >> 16).astype(np.uint16).tobytes()
        else:
            raw = a.tobytes()
        table.append((offset, len(raw)))
        chunks.append((offset, raw))
        offset = (offset + len(raw) + 255) // 256 * 256
    blob = bytearray(offset)
    blob[0:8] = BLOB_MAGIC
    blob[8:24] = struct.pack("<IIQ", 1, len(tensors), 0)
    for i, (off, nb) in enumerate(table):
        blob[24 + 16 * i:40 + 16 * i] = struct.pack("<QQ", off, nb)
    for off, raw in chunks:
        blob[off:off + len(raw)] = raw
    return bytes(blob)


# ---- C-ABI calls, same names ------------------------------------------------

def mtp_create(config: MtpConfig, blob: bytes, stream=None) -> int:
    handle = ctypes.c_void_p()
    buf = ctypes.create_string_buffer(blob, len(blob))
    check(lib.mtp_create(ctypes.byref(config), buf, len(blob), _stream_handle(stream), ctypes.byref(handle)))
    return handle.value


def mtp_destroy(ctx: int) -> None:
    lib.mtp_destroy(ctx)


def mtp_last_error() -> str:
    return lib.mtp_last_error().decode(errors="replace")


def mtp_prefill(ctx: int, slot: int, phonemes, acoustic, max_new_tokens: int) -> None:
    ph = _as_i32(phonemes)
    ac = _as_i32(acoustic)
    check(lib.mtp_prefill(ctx, slot, _ptr(ph), _len(ph), _ptr(ac), _len(ac), max_new_tokens))


def mtp_release(ctx: int, slot: int) -> None:
    check(lib.mtp_release(ctx, slot))


def mtp_admit(ctx: int, slot: int, phonemes, acoustic, max_new_tokens: int) -> None:
    """Admit a prompt without running it: the next decode steps prefill it in their lane."""
    ph = _as_i32(phonemes)
    ac = _as_i32(acoustic)
    check(lib.mtp_admit(ctx, slot, _ptr(ph), _len(ph), _ptr(ac), _len(ac), max_new_tokens))


def mtp_prefill_pending(ctx: int) -> int:
    """Run every admitted prompt now, many slots' prompt rows per pass; returns the passes."""
    return check(lib.mtp_prefill_pending(ctx))


def mtp_decode_step(ctx: int, n_heads: int, top_k: int, out_tokens=None, out_accepted=None,
                    out_done=None) -> None:
    check(lib.mtp_decode_step(ctx, n_heads, top_k, _ptr(out_tokens), _ptr(out_accepted), _ptr(out_done)))


def mtp_generate(ctx: int, n_heads: int, top_k: int, out_tokens=None, out_stride: int = 0,
                 out_lens=None) -> int:
    return check(lib.mtp_generate(ctx, n_heads, top_k, _ptr(out_tokens), out_stride, _ptr(out_lens)))


def mtp_rollback(ctx: int, slot: int, n_tokens: int) -> None:
    check(lib.mtp_rollback(ctx, slot, n_tokens))


def mtp_set_teacher_tokens(ctx: int, slot: int, tokens) -> None:
    t = np.ascontiguousarray(tokens, dtype=np.int32)
    check(lib.mtp_set_teacher_tokens(ctx, slot, _ptr(t), t.shape[0]))


def mtp_seq_state(ctx: int, slot: int) -> dict:
    out = np.zeros(6, np.int32)
    check(lib.mtp_seq_state(ctx, slot, _ptr(out)))
    return dict(zip(("len", "pending", "remaining", "done", "active", "generated"), out.tolist()))


def mtp_debug_logits(ctx: int, out_logits=None, out_lse=None) -> None:
    check(lib.mtp_debug_logits(ctx, _ptr(out_logits), _ptr(out_lse)))


def mtp_debug_lattice(ctx: int, out_ids=None, out_logp=None, out_path=None) -> None:
    check(lib.mtp_debug_lattice(ctx, _ptr(out_ids), _ptr(out_logp), _ptr(out_path)))


def mtp_set_option(ctx: int, option: int, value: int) -> None:
    check(lib.mtp_set_option(ctx, option, value))


def mtp_get_option(ctx: int, option: int) -> int:
    out = ctypes.c_int32()
    check(lib.mtp_get_option(ctx, option, ctypes.byref(out)))
    return int(out.value)


def mtp_profile_step(ctx: int, n_heads: int, top_k: int) -> dict:
    ms = np.zeros(len(_lib.KERNEL_KINDS), np.float32)
    launches = np.zeros(len(_lib.KERNEL_KINDS), np.int32)
    check(lib.mtp_profile_step(ctx, n_heads, top_k, _ptr(ms), _ptr(launches)))
    return {k: (float(ms[i]), int(launches[i])) for i, k in enumerate(_lib.KERNEL_KINDS)}


def mtp_trace_step(ctx: int, n_heads: int, top_k: int, cap: int = 4096) -> np.ndarray:
    """Timeline of one decode step: rows (kind, start_ns, wait_ns, end_ns, 8 phase marks)."""
    out = np.zeros((cap, 12), np.int64)
    count = check(lib.mtp_trace_step(ctx, n_heads, top_k, _ptr(out), cap))
    return out[:count]


def mtp_step_bytes(ctx: int, n_heads: int) -> int:
    out = ctypes.c_uint64()
    check(lib.mtp_step_bytes(ctx, n_heads, ctypes.byref(out)))
    return int(out.value)


def mtp_viterbi(batch, n, k, vocab, eos_id, cand_ids, cand_logp, log_q, remaining, out_path,
                out_score, out_accepted, out_rollback, stream=None) -> None:
    check(lib.mtp_viterbi(batch, n, k, vocab, eos_id, _ptr(cand_ids), _ptr(cand_logp), _ptr(log_q),
                          _ptr(remaining), _ptr(out_path), _ptr(out_score), _ptr(out_accepted),
                          _ptr(out_rollback), _stream_handle(stream)))


def mtp_selftest_bounded_wait(err_word, stream=None) -> None:
    check(lib.mtp_selftest_bounded_wait(_ptr(err_word), _stream_handle(stream)))


def mtp_selftest_grid_barrier(err_word, stream=None) -> None:
    """One CTA at a grid barrier that never completes; its bounded wait sets err_word."""
    check(lib.mtp_selftest_grid_barrier(_ptr(err_word), _stream_handle(stream)))


def mtp_heads_topk(ctx, batch, hidden, hidden_dtype, n_heads, top_k, out_ids, out_logp,
                   out_logits=None, out_lse=None) -> None:
    check(lib.mtp_heads_topk(ctx, batch, _ptr(hidden), hidden_dtype, n_heads, top_k, _ptr(out_ids),
                             _ptr(out_logp), _ptr(out_logits), _ptr(out_lse)))


def attention_args(**kw) -> MtpAttentionArgs:
    a = MtpAttentionArgs()
    for key, val in kw.items():
        setattr(a, key, _ptr(val) if key in ("q", "kv_pool", "block_table", "row_seq", "row_pos", "out")
                else val)
    return a


def mtp_attention_workspace_bytes(args: MtpAttentionArgs) -> int:
    return int(lib.mtp_attention_workspace_bytes(ctypes.byref(args)))


def mtp_attention(args: MtpAttentionArgs, workspace, workspace_bytes: int, stream=None) -> None:
    check(lib.mtp_attention(ctypes.byref(args), _ptr(workspace), workspace_bytes, _stream_handle(stream)))


def mtp_attention_tc_workspace_bytes(args: MtpAttentionArgs) -> int:
    return int(lib.mtp_attention_tc_workspace_bytes(ctypes.byref(args)))


def mtp_attention_tc(args: MtpAttentionArgs, workspace, workspace_bytes: int, stream=None) -> None:
    """Tensor-core attention of prompt rows (tiles of 128 rows); the pool in the cache's swizzled layout."""
    check(lib.mtp_attention_tc(ctypes.byref(args), _ptr(workspace), workspace_bytes, _stream_handle(stream)))


def mtp_attention_noalloc(args: MtpAttentionArgs, stream=None) -> None:
    """mtp_attention with the library's fixed scratch array: no workspace, no allocation."""
    check(lib.mtp_attention_noalloc(ctypes.byref(args), _stream_handle(stream)))


def mtp_gemm_bf16x2(w, a_hi, a_lo, out, n_w, k, m, splits=1, accumulate=0, stream=None) -> None:
    """out (+)= (a_hi + a_lo) @ w.T on the tensor cores (the batched path's projection)."""
    check(lib.mtp_gemm_bf16x2(_ptr(w), _ptr(a_hi), _ptr(a_lo), _ptr(out), n_w, k, m, splits, accumulate,
                              _stream_handle(stream)))


def _as_i32(x):
    if x is None:
        return None
    if hasattr(x, "data_ptr"):
        return x.contiguous()
    return np.ascontiguousarray(x, dtype=np.int32)


def _len(x) -> int:
    return 0 if x is None else int(x.shape[0])


class MTPDecoder:
    """Owns one mtp_ctx: weights on the device, KV pages, slot state."""

    def __init__(self, model, weights: dict[str, np.ndarray], names: list[str], is_matrix,
                 max_batch: int, max_ctx: int, page_size: int = 64, n_pages: int = 0, stream=None,
                 accept_policy: int = 0):
        self.model = model
        self.config = make_config(model, max_batch, max_ctx, page_size, n_pages, accept_policy)
        blob = pack_weights([(weights[n], is_matrix(n)) for n in names], model.weight_dtype == "bf16")
        self.ctx = mtp_create(self.config, blob, stream)

    def close(self) -> None:
        if self.ctx:
            mtp_destroy(self.ctx)
            self.ctx = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def prefill(self, slot, phonemes, acoustic, max_new_tokens):
        mtp_prefill(self.ctx, slot, phonemes, acoustic, max_new_tokens)

    def admit(self, slot, phonemes, acoustic, max_new_tokens):
        mtp_admit(self.ctx, slot, phonemes, acoustic, max_new_tokens)

    def decode_step(self, n_heads, top_k):
        b = self.config.max_batch
        toks = np.zeros((b, n_heads), np.int32)
        acc = np.zeros(b, np.int32)
        done = np.zeros(b, np.int32)
        mtp_decode_step(self.ctx, n_heads, top_k, toks, acc, done)
        return toks, acc, done

    def generate(self, n_heads, top_k, max_new):
        b = self.config.max_batch
        toks = np.zeros((b, max_new), np.int32)
        lens = np.zeros(b, np.int32)
        steps = mtp_generate(self.ctx, n_heads, top_k, toks, max_new, lens)
        return [toks[i, :lens[i]].tolist() for i in range(b)], steps

    def logits(self, n_heads):
        b, v = self.config.max_batch, self.config.codec_vocab
        lg = np.zeros((b, n_heads, v), np.float32)
        lse = np.zeros((b, n_heads), np.float32)
        mtp_debug_logits(self.ctx, lg, lse)
        return lg, lse

    def lattice(self, n_heads, top_k):
        b = self.config.max_batch
        ids = np.zeros((b, n_heads, top_k), np.int32)
        lp = np.zeros((b, n_heads, top_k), np.float32)
        path = np.zeros((b, n_heads), np.int32)
        mtp_debug_lattice(self.ctx, ids, lp, path)
        return ids, lp, path

    def state(self, slot):
        return mtp_seq_state(self.ctx, slot)


__all__ = [n for n in dir() if n.startswith("mtp_")] + ["MTPDecoder", "MTPError", "pack_weights",
                                                         "make_config", "attention_args"]
