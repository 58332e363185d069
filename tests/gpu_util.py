"""Shared helpers of the GPU parity tests (build/load libmtp, seeded decoders)."""
import functools

import numpy as np
import pytest

import synth

# Parity bars (bf16 weights and KV cache against the float64 oracle)
LOGIT_ATOL = 2e-2          # elementwise |gpu - oracle|
LOGIT_REL = 1e-2           # max |gpu - oracle| / max |oracle|
MARGIN = 5e-2              # token decisions must agree where the oracle's margin exceeds this


@functools.lru_cache(maxsize=1)
def lib_module():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2410_13839_gb300 import build
    build.build()
    from paper_2410_13839_gb300 import mtp
    return mtp


def decoder(model, max_batch=1, max_ctx=512, page_size=64, n_pages=0, eos_bias=synth.EOS_BIAS, seed=0,
            accept_policy=0):
    mtp = lib_module()
    w = synth.make_weights(model, seed=seed, eos_bias=eos_bias)
    dec = mtp.MTPDecoder(model, w, synth.weight_names(model), synth.is_matrix, max_batch, max_ctx,
                         page_size=page_size, n_pages=n_pages, accept_policy=accept_policy)
    return dec, w


def assert_logits_close(gpu, ref, what=""):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    err = np.abs(gpu - ref)
    assert err.max() <= LOGIT_ATOL, f"{what}: max abs err {err.max():.3e}"
    assert err.max() / np.abs(ref).max() <= LOGIT_REL, f"{what}: rel err {err.max() / np.abs(ref).max():.3e}"


def logp32(logits32, lse32):
    """The kernels' ranking score: logits - lse as one float32 subtraction."""
    return (np.asarray(logits32, np.float32) - np.asarray(lse32, np.float32)[..., None]).astype(np.float32)
