"""The batched path's tensor-core GEMM (tcgen05 + TMA) against a plain
PyTorch fp32 product of the same operands: out = (a_hi + a_lo) @ w.T."""
import pytest

pytestmark = pytest.mark.gpu

CASES = [  # n_w, k, m, splits, accumulate
    (128, 64, 1, 1, 0),
    (256, 128, 5, 1, 0),
    (384, 1024, 100, 4, 1),
    (128, 4096, 128, 8, 1),
    (3072, 1024, 33, 2, 1),
    (1024, 1024, 200, 1, 0),
]


def _split(a):
    import torch
    hi = a.to(torch.bfloat16)
    lo = (a - hi.float()).to(torch.bfloat16)
    return hi, lo


@pytest.mark.parametrize("n_w,k,m,splits,accumulate", CASES)
def test_tc_gemm_matches_fp32_product(n_w, k, m, splits, accumulate):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from gpu_util import lib_module
    mtp = lib_module()
    g = torch.Generator(device="cuda").manual_seed(1000 * n_w + k + m)
    w = (torch.randn(n_w, k, device="cuda", generator=g) * 0.02).to(torch.bfloat16)
    a = torch.randn(m, k, device="cuda", generator=g)
    hi, lo = _split(a)
    base = torch.randn(m, n_w, device="cuda", generator=g) if accumulate else None
    out = base.clone() if accumulate else torch.full((m, n_w), float("nan"), device="cuda")
    mtp.mtp_gemm_bf16x2(w, hi, lo, out, n_w, k, m, splits, accumulate, torch.cuda.current_stream())
    ref = (hi.double() + lo.double()) @ w.double().T
    if accumulate:
        ref = ref + base.double()
    err = (out.double() - ref).abs().max().item()
    scale = ref.abs().max().item()
    assert err <= 1e-5 * max(1.0, scale) + 2e-6 * k ** 0.5, f"max abs err {err:.3e} (scale {scale:.3e})"


def test_tc_gemm_rejects_bad_shapes():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from gpu_util import lib_module
    mtp = lib_module()
    w = torch.zeros(100, 64, device="cuda", dtype=torch.bfloat16)
    a = torch.zeros(4, 64, device="cuda", dtype=torch.bfloat16)
    out = torch.zeros(4, 100, device="cuda")
    with pytest.raises(mtp.MTPError):
        mtp.mtp_gemm_bf16x2(w, a, a, out, 100, 64, 4, 1, 0)   # n_w not a multiple of 128
    w = torch.zeros(128, 64, device="cuda", dtype=torch.bfloat16)
    with pytest.raises(mtp.MTPError):
        mtp.mtp_gemm_bf16x2(w, a, a, out, 128, 64, 4, 2, 1)   # one k-chunk cannot split in two
