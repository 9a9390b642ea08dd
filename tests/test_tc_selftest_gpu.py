"""The tensor-core building blocks (TMA with 128-byte swizzle, tcgen05.mma
from shared-memory descriptors, tensor-memory loads) against torch: one
128x128x128 bf16 GEMM per operand layout the attention kernel uses."""

import pytest
import torch

from paper_2603_01639_gb300 import ltd

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2603_01639_gb300 import build
    build.build()


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("pattern", ["random", "identity", "ramp"])
def test_umma_gemm(mode, pattern):
    g = torch.Generator(device="cuda").manual_seed(mode * 10 + len(pattern))
    if pattern == "random":
        a = torch.randn(128, 128, generator=g, device="cuda").to(torch.bfloat16)
        b = torch.randn(128, 128, generator=g, device="cuda").to(torch.bfloat16)
    elif pattern == "identity":
        a = torch.randn(128, 128, generator=g, device="cuda").to(torch.bfloat16)
        b = torch.eye(128, device="cuda").to(torch.bfloat16)
    else:  # distinct small integers: any misplaced element changes the result
        idx = torch.arange(128 * 128, device="cuda").view(128, 128)
        a = ((idx % 7) - 3).to(torch.bfloat16)
        b = ((idx % 11) - 5).to(torch.bfloat16)
    c = ltd.ltd_selftest_umma(mode, a, b)
    assert ltd.ltd_check() == 0
    ref = a.double() @ (b.double().T if mode == 0 else b.double())
    err = (c.double() - ref).abs().max().item()
    assert err <= 1e-3 * max(1.0, ref.abs().max().item()), err
