"""Tensor-core building blocks on the GPU: one 128x128x128 tcgen05 tile
product (shared-memory descriptors, instruction descriptor, TMEM loads, TMA
swizzle) against a float64 product of the same bf16 values."""
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ism():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2408_00539_gb300 import ism as m
    m.load(build_if_missing=True)
    if not m.has_tensor_cores():
        pytest.skip("tensor-core kernels need sm_103")
    return m


@pytest.mark.parametrize("mode", list(range(16)))
def test_mma_tile(ism, mode):
    """Each operand layout, with the k-steps issued one by one (modes 0-7) and
    through the batched eight-step form (modes 8-15)."""
    g = torch.Generator().manual_seed(100 + mode % 8)
    a = torch.randn(128, 128, generator=g).to(torch.bfloat16)
    b = torch.randn(128, 128, generator=g).to(torch.bfloat16)
    c = ism.debug_mma_tile(a.cuda(), b.cuda(), mode)
    ism.check_status()
    if mode % 8 in (6, 7):
        ref = a.double().T @ b.double()
    else:
        ref = a.double() @ (b.double().T if mode % 2 == 0 else b.double())
    err = (c.double().cpu() - ref).abs().max().item()
    assert err < 1e-3, f"mode {mode}: max abs err {err}"


@pytest.mark.parametrize("mode", [0, 1, 2])
def test_mma_tile_e4m3(ism, mode):
    """The e4m3 operand layouts (kind::f8f6f4): K-major A and B, MN-major B, A in
    tensor memory; e4m3 products are exact in the fp32 accumulator."""
    g = torch.Generator().manual_seed(200 + mode)
    a = (torch.randn(128, 128, generator=g) * 2).to(torch.float8_e4m3fn)
    b = (torch.randn(128, 128, generator=g) * 2).to(torch.float8_e4m3fn)
    c = ism.debug_mma_tile_e4m3(a.cuda(), b.cuda(), mode)
    ism.check_status()
    ref = a.double() @ (b.double().T if mode == 0 else b.double())
    err = (c.double().cpu() - ref).abs().max().item()
    assert err < 1e-4 * ref.abs().max().item(), f"mode {mode}: max abs err {err}"
