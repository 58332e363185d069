"""Failure detection without a GPU fault: a bounded wait on a barrier that
nothing completes runs out by itself, reports through the device error word,
and the CUDA context stays usable (a decode step runs afterwards)."""
import time

import pytest

import synth

from gpu_util import decoder, lib_module

pytestmark = pytest.mark.gpu


def test_bounded_wait_runs_out_and_reports():
    import torch
    mtp = lib_module()
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    t0 = time.time()
    mtp.mtp_selftest_bounded_wait(err, torch.cuda.current_stream())
    torch.cuda.synchronize()
    assert int(err.item()) == 1          # MTP_DEVICE_ERR_WAIT
    assert time.time() - t0 < 60
    dec, _ = decoder(synth.TINY, max_batch=1, max_ctx=64)
    try:
        ph, ac = synth.make_prompt(1, 8, 8, synth.TINY.phone_vocab)
        dec.prefill(0, ph, ac, 8)
        toks, acc, _ = dec.decode_step(4, 4)
        assert int(acc[0]) == 4
    finally:
        dec.close()


def test_selftest_rejects_null():
    mtp = lib_module()
    with pytest.raises(mtp.MTPError):
        mtp.mtp_selftest_bounded_wait(None)
