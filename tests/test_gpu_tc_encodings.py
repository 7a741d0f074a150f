"""The tcgen05 encodings (swizzled K-major / MN-major shared-memory operands, instruction
descriptor, TMEM load layout) against torch's matmul on the same bf16 inputs."""
import pytest
import torch

from paper_2608_06146_gb300 import build as pbuild
from paper_2608_06146_gb300 import padoc_attn as pa

pytestmark = pytest.mark.gpu


def test_tcgen05_selftest_matches_matmul():
    pbuild.build()
    pa.load_library()
    g = torch.Generator().manual_seed(3)
    a, bk, v = (torch.randn(128, 128, generator=g).to(torch.bfloat16).cuda() for _ in range(3))
    c1 = torch.full((128, 128), float("nan"), device="cuda")
    c2 = torch.full((128, 128), float("nan"), device="cuda")
    c3 = torch.full((128, 128), float("nan"), device="cuda")
    pa.padoc_selftest_tcgen05(a, bk, v, c1, c2, c3)
    pa.padoc_check_device_errors()
    ref1 = a.double() @ bk.double().T
    ref2 = a.double() @ v.double()
    assert (c1.double() - ref1).abs().max().item() < 1e-3, "K-major x K-major product mismatch"
    assert (c2.double() - ref2).abs().max().item() < 1e-3, "K-major x MN-major product mismatch"
    assert (c3.double() - ref2).abs().max().item() < 1e-3, "TMEM A operand x MN-major product mismatch"
