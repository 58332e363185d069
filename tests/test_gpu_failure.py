"""Failure detection without a GPU fault: a bounded wait on a barrier that
nothing completes (a shared-memory mbarrier; the persistent step kernel's grid
barrier) runs out by itself, reports through the device error word, and the
CUDA context stays usable (a decode step runs afterwards)."""
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


def test_grid_barrier_runs_out_and_reports():
    import torch
    mtp = lib_module()
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    t0 = time.time()
    for _ in range(2):  # the barrier's counter is left at zero: a second call behaves the same
        err.zero_()
        mtp.mtp_selftest_grid_barrier(err, torch.cuda.current_stream())
        torch.cuda.synchronize()
        assert int(err.item()) == 1      # MTP_DEVICE_ERR_WAIT
    assert time.time() - t0 < 60
    dec, _ = decoder(synth.TINY_BF16, max_batch=1, max_ctx=80)
    try:
        mtp.mtp_set_option(dec.ctx, 9, 1)  # the persistent step kernel still runs
        ph, ac = synth.make_prompt(1, 8, 8, synth.TINY_BF16.phone_vocab)
        dec.prefill(0, ph, ac, 8)
        toks, acc, _ = dec.decode_step(4, 4)
        assert 1 <= int(acc[0]) <= 4 and dec.state(0)["len"] == 16
    finally:
        dec.close()


def test_selftest_rejects_null():
    mtp = lib_module()
    with pytest.raises(mtp.MTPError):
        mtp.mtp_selftest_bounded_wait(None)
    with pytest.raises(mtp.MTPError):
        mtp.mtp_selftest_grid_barrier(None)
