"""CPU checks of the C-ABI library: it builds, loads without a GPU and exports
every function include/mtp.h declares; the weight-blob writer follows the
header's format."""
import ctypes
import os
import re
import struct

import numpy as np
import pytest

import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mtp.h")


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"MTP_API\s+[\w\s\*]+?\b(mtp_\w+)\s*\(", text)))


@pytest.fixture(scope="module")
def libpath():
    from paper_2410_13839_gb300 import build
    try:
        return build.build()
    except RuntimeError as e:       # no nvcc on this machine
        pytest.skip(str(e))


def test_header_declares_the_abi():
    names = declared_functions()
    for must in ("mtp_create", "mtp_prefill", "mtp_decode_step", "mtp_viterbi", "mtp_generate",
                 "mtp_rollback", "mtp_destroy", "mtp_last_error"):
        assert must in names


def test_library_exports_every_declared_symbol(libpath):
    lib = ctypes.CDLL(libpath)
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_binding_wraps_every_symbol(libpath):
    from paper_2410_13839_gb300 import mtp
    missing = [n for n in declared_functions() if not hasattr(mtp, n)]
    assert not missing, missing


def test_create_without_gpu_fails_cleanly(libpath):
    from paper_2410_13839_gb300 import mtp
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    cfg = mtp.make_config(synth.TINY, 1, 64)
    with pytest.raises(mtp.MTPError):
        mtp.mtp_create(cfg, b"MTPWGT01" + bytes(16))


def test_invalid_config_is_rejected_before_any_device_call(libpath):
    from paper_2410_13839_gb300 import mtp
    cfg = mtp.make_config(synth.TINY, 1, 64)
    cfg.d_model = 300
    with pytest.raises(mtp.MTPError) as e:
        mtp.mtp_create(cfg, b"")
    assert e.value.code == -1


def test_blob_layout():
    from paper_2410_13839_gb300.mtp import pack_weights
    a = np.arange(6, dtype=np.float32).reshape(2, 3)
    m = synth.round_bf16(np.array([1.5, -2.25, 3.0], np.float32))
    blob = pack_weights([(a, False), (m, True)], bf16=True)
    assert blob[:8] == b"MTPWGT01"
    version, count, _ = struct.unpack("<IIQ", blob[8:24])
    assert (version, count) == (1, 2)
    (o1, n1), (o2, n2) = struct.unpack("<QQ", blob[24:40]), struct.unpack("<QQ", blob[40:56])
    assert o1 % 256 == 0 and o2 % 256 == 0 and n1 == 24 and n2 == 6
    assert np.array_equal(np.frombuffer(blob[o1:o1 + n1], np.float32).reshape(2, 3), a)
    bits = np.frombuffer(blob[o2:o2 + n2], np.uint16).astype(np.uint32) << 16
    assert np.array_equal(bits.view(np.float32), m)
    with pytest.raises(ValueError):
        pack_weights([(np.array([1.1], np.float32), True)], bf16=True)
