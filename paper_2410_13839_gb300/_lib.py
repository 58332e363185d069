"""ctypes declarations of libmtp.so (include/mtp.h).  Argument marshalling only.

Importing this module loads the in-tree library and fails loudly when it has
not been built: there is no other implementation of the path.
"""
from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libmtp.so")

MTP_OK = 0
MTP_ERR_INVALID = -1
MTP_ERR_NO_PAGES = -2
MTP_ERR_CUDA = -3
MTP_ERR_WEIGHTS = -4
MTP_ERR_DEVICE = -5
MTP_F32 = 0
MTP_BF16 = 1
MTP_ACCEPT_ALL = 0
MTP_VERIFY_GREEDY = 1
MTP_OPT_GRAPHS = 0
MTP_OPT_PDL = 1
MTP_OPT_L2_PREFETCH = 2
MTP_OPT_MLP_CLUSTERS = 3
MTP_OPT_BATCHED = 4
MTP_OPT_GEMM_SPLITS = 5
MTP_OPT_LATTICE = 6
MTP_OPT_SAMPLING = 7
MTP_OPT_SEED = 8
MTP_OPT_PERSISTENT = 9
MTP_OPT_PREFILL_TC = 10
MTP_OPT_HEADS_FUSED = 11
MTP_OPT_GEMM_CLUSTER = 12
KERNEL_KINDS = ("embed", "attn_block", "mlp", "heads", "select", "save", "pack", "gemm", "qkv", "attn", "step", "step_attn",
                "step_mlp", "step_cta", "attn_tc")


class MtpConfig(ctypes.Structure):
    _fields_ = [(name, ctypes.c_int32) for name in (
        "layers", "d_model", "n_attn_heads", "d_ffn", "phone_vocab", "codec_vocab", "eos_id",
        "n_heads_max", "top_k_max", "max_batch", "max_ctx", "page_size", "n_pages",
        "weight_dtype", "accept_policy")] + [("ln_eps", ctypes.c_float)]


class MtpAttentionArgs(ctypes.Structure):
    _fields_ = [(name, ctypes.c_int32) for name in (
        "rows", "rows_per_group", "n_heads", "page_size", "layers", "layer", "bt_stride",
        "max_keys")] + [(name, ctypes.c_void_p) for name in (
            "q", "kv_pool", "block_table", "row_seq", "row_pos", "out")]


class MTPError(RuntimeError):
    def __init__(self, code: int, message: str):
        super().__init__(f"libmtp error {code}: {message}")
        self.code = code


def _load() -> ctypes.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it first "
                          "(python -c 'import __graft_entry__ as g; g.build()')")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i32, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
    sig = {
        "mtp_create": (i32, [ctypes.POINTER(MtpConfig), vp, sz, vp, ctypes.POINTER(vp)]),
        "mtp_destroy": (None, [vp]),
        "mtp_last_error": (ctypes.c_char_p, []),
        "mtp_prefill": (i32, [vp, i32, vp, i32, vp, i32, i32]),
        "mtp_release": (i32, [vp, i32]),
        "mtp_admit": (i32, [vp, i32, vp, i32, vp, i32, i32]),
        "mtp_prefill_pending": (i32, [vp]),
        "mtp_decode_step": (i32, [vp, i32, i32, vp, vp, vp]),
        "mtp_generate": (i32, [vp, i32, i32, vp, i32, vp]),
        "mtp_rollback": (i32, [vp, i32, i32]),
        "mtp_set_teacher_tokens": (i32, [vp, i32, vp, i32]),
        "mtp_seq_state": (i32, [vp, i32, vp]),
        "mtp_debug_logits": (i32, [vp, vp, vp]),
        "mtp_debug_lattice": (i32, [vp, vp, vp, vp]),
        "mtp_set_option": (i32, [vp, i32, i32]),
        "mtp_get_option": (i32, [vp, i32, vp]),
        "mtp_profile_step": (i32, [vp, i32, i32, vp, vp]),
        "mtp_step_bytes": (i32, [vp, i32, vp]),
        "mtp_trace_step": (i32, [vp, i32, i32, vp, i32]),
        "mtp_viterbi": (i32, [i32, i32, i32, i32, i32, vp, vp, vp, vp, vp, vp, vp, vp, vp]),
        "mtp_heads_topk": (i32, [vp, i32, vp, i32, i32, i32, vp, vp, vp, vp]),
        "mtp_selftest_bounded_wait": (i32, [vp, vp]),
        "mtp_selftest_grid_barrier": (i32, [vp, vp]),
        "mtp_attention_workspace_bytes": (sz, [ctypes.POINTER(MtpAttentionArgs)]),
        "mtp_attention": (i32, [ctypes.POINTER(MtpAttentionArgs), vp, sz, vp]),
        "mtp_attention_noalloc": (i32, [ctypes.POINTER(MtpAttentionArgs), vp]),
        "mtp_attention_tc_workspace_bytes": (sz, [ctypes.POINTER(MtpAttentionArgs)]),
        "mtp_attention_tc": (i32, [ctypes.POINTER(MtpAttentionArgs), vp, sz, vp]),
        "mtp_gemm_bf16x2": (i32, [vp, vp, vp, vp, i32, i32, i32, i32, i32, vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


lib = _load()


def check(code: int) -> int:
    """Raise MTPError for a negative status; return non-negative results unchanged."""
    if code < 0:
        raise MTPError(code, lib.mtp_last_error().decode(errors="replace"))
    return code
