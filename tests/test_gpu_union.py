"""The union lattice (reading B) on the GPU: per step the path equals the
oracle's reading-B Viterbi run on the GPU's own float32 scores (bit-exact),
and the logits stay within the bar of the oracle run teacher-forced under the
same reading."""
import numpy as np
import pytest

import synth
from oracle import select as S
from oracle.mtp import MTPOracle

from gpu_util import assert_logits_close, decoder, lib_module, logp32

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("model,n,k,steps", [(synth.TINY, 4, 4, 10), (synth.TINY, 8, 32, 4), (synth.VALLE, 4, 8, 4)])
def test_union_lattice_matches_oracle(model, n, k, steps):
    mtp = lib_module()
    ph, ac = synth.make_prompt(9, 16, 40, model.phone_vocab)
    dec, w = decoder(model, max_batch=1, max_ctx=len(ph) + len(ac) + 100)
    try:
        mtp.mtp_set_option(dec.ctx, 6, 1)
        assert mtp.mtp_get_option(dec.ctx, 6) == 1
        o = MTPOracle(model, w)
        o.prefill(ph, ac, 60)
        dec.prefill(0, ph, ac, 60)
        for step in range(steps):
            fed = o.pending.copy()
            rec = o.step(n, k, lattice="B")
            if len(fed):
                mtp.mtp_set_teacher_tokens(dec.ctx, 0, fed)
            toks, acc, _ = dec.decode_step(n, k)
            lg, lse = dec.logits(n)
            ids, lp, path = dec.lattice(n, k)
            assert_logits_close(lg[0], rec.logits, f"step {step}")
            sc = logp32(lg[0], lse[0])
            r_ids, _ = S.top_k_rows(sc, k)
            r_path, _ = S.viterbi_union(r_ids, sc, o.log_q)
            assert np.array_equal(path[0], r_path), f"step {step}"
            a = int(acc[0])
            assert toks[0, :a].tolist() == path[0, :a].tolist()
    finally:
        dec.close()
