"""GPU parity of the split-KV decode attention over the paged bf16 cache (Sec. III-A)."""
import numpy as np
import pytest

import synth
from oracle.model import causal_attention

from gpu_util import lib_module

pytestmark = pytest.mark.gpu

H, HD, LAYERS = 4, 64, 3


def _case(groups, rpg, ctx_list, page_size, inactive=(), max_keys=None, layer=1, seed=0):
    """groups slots; group g has rows at positions ctx_list[g]-rpg .. ctx_list[g]-1."""
    import torch
    mtp = lib_module()
    max_ctx = max(ctx_list)
    pages_per_seq = (max_ctx + page_size - 1) // page_size + 1
    n_pages = groups * pages_per_seq + 3
    pool = synth.round_bf16(synth.normal(seed, "pool", n_pages * LAYERS * 2 * H * page_size * HD)
                            .astype(np.float32)).reshape(n_pages, LAYERS, 2, H, page_size, HD)
    perm = np.argsort(synth.uniform(seed, "perm", n_pages))        # scattered physical pages
    table = np.full((groups, pages_per_seq), -1, np.int32)
    for g in range(groups):
        table[g] = perm[g * pages_per_seq:(g + 1) * pages_per_seq]
    rows = groups * rpg
    q = synth.normal(seed, "q", rows * H * HD).astype(np.float32).reshape(rows, H, HD)
    row_seq = np.repeat(np.arange(groups, dtype=np.int32), rpg)
    row_pos = np.concatenate([np.arange(c - rpg, c) for c in ctx_list]).astype(np.int32)
    for r in inactive:
        row_seq[r] = -1
    dev = torch.device("cuda")
    bits = (pool.view(np.uint32) >> 16).astype(np.uint16)
    t_pool = torch.from_numpy(bits.view(np.int16)).to(dev)
    t_q = torch.from_numpy(q.reshape(rows, H * HD)).to(dev)
    t_tab = torch.from_numpy(table).to(dev)
    t_seq = torch.from_numpy(row_seq).to(dev)
    t_pos = torch.from_numpy(row_pos).to(dev)
    out = torch.full((rows, H * HD), -7.0, dtype=torch.float32, device=dev)
    args = mtp.attention_args(rows=rows, rows_per_group=rpg, n_heads=H, page_size=page_size, layers=LAYERS,
                              layer=layer, bt_stride=pages_per_seq, max_keys=max_keys or max_ctx,
                              q=t_q, kv_pool=t_pool, block_table=t_tab, row_seq=t_seq, row_pos=t_pos, out=out)
    nbytes = mtp.mtp_attention_workspace_bytes(args)
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=dev)
    for _ in range(2):        # the counters must come back to zero: a second call agrees
        mtp.mtp_attention(args, ws, nbytes, torch.cuda.current_stream())
        torch.cuda.synchronize()
        got = out.cpu().numpy().reshape(rows, H, HD)
        for g in range(groups):
            logical = np.concatenate([pool[table[g, p], layer] for p in range(pages_per_seq)], axis=2)
            k = logical[0].transpose(1, 0, 2).astype(np.float64)   # [T, H, HD]
            v = logical[1].transpose(1, 0, 2).astype(np.float64)
            rs = slice(g * rpg, (g + 1) * rpg)
            ref = causal_attention(q[rs].astype(np.float64), k, v, row_pos[rs], np.arange(k.shape[0]))
            for j in range(rpg):
                r = g * rpg + j
                if row_seq[r] < 0:
                    assert np.all(got[r] == -7.0), "inactive row was written"
                else:
                    assert np.abs(got[r] - ref[j]).max() < 1e-4, f"group {g} row {j}"


@pytest.mark.parametrize("groups,rpg,ctx,page", [
    (1, 4, [1039], 64),          # VALL-E-sized decode, 4 fed rows
    (1, 1, [1], 64),             # one key: output equals v
    (1, 8, [65], 64),            # ragged page tail
    (2, 4, [300, 77], 16),       # two slots, small pages
    (1, 2, [700], 128),
    (8, 1, [50, 60, 70, 80, 90, 100, 110, 2000], 64),
])
def test_attention_parity(groups, rpg, ctx, page):
    _case(groups, rpg, ctx, page)


def test_attention_inactive_rows_and_spare_splits():
    _case(2, 4, [130, 257], 64, inactive=(1, 6), max_keys=4000)
