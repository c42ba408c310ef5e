"""The tensor-core building blocks through the C ABI (GPU): shared-memory
descriptors, tcgen05.mma and the tensor-memory read-back, against a plain
PyTorch fp32 matmul of the same fp16 operands."""
import os

import numpy as np
import pytest
import torch

from gpu_common import api

pytestmark = pytest.mark.gpu

OUT = os.environ.get("SOMA_TEST_DUMP", "")


@pytest.mark.parametrize("a_in_tmem", [False, True])
@pytest.mark.parametrize("n", [16, 32, 64, 128, 256])
@pytest.mark.parametrize("k", [16, 32, 64, 256])
def test_tc_gemm_small_integers_exact(n, k, a_in_tmem):
    # entries in -2..2: every product and partial sum is exact in fp32
    g = torch.Generator().manual_seed(n * 1000 + k)
    a = torch.randint(-2, 3, (128, k), generator=g).to(torch.float16)
    b = torch.randint(-2, 3, (n, k), generator=g).to(torch.float16)
    d = api().debug_tc_gemm(a.cuda(), b.cuda(), a_in_tmem=a_in_tmem).cpu()
    assert api().get_status() == 0
    ref = a.float() @ b.float().T
    if OUT and not torch.equal(d, ref):
        np.save(os.path.join(OUT, f"tc_gemm_{n}_{k}_d.npy"), d.numpy())
        np.save(os.path.join(OUT, f"tc_gemm_{n}_{k}_ref.npy"), ref.numpy())
        np.save(os.path.join(OUT, f"tc_gemm_{n}_{k}_a.npy"), a.float().numpy())
        np.save(os.path.join(OUT, f"tc_gemm_{n}_{k}_b.npy"), b.float().numpy())
    assert torch.equal(d, ref)


def test_tc_gemm_random_normal():
    g = torch.Generator().manual_seed(5)
    a = (torch.randn(128, 256, generator=g) * 0.5).to(torch.float16)
    b = (torch.randn(256, 256, generator=g) * 0.5).to(torch.float16)
    d = api().debug_tc_gemm(a.cuda(), b.cuda()).cpu()
    ref = a.double() @ b.double().T
    err = (d.double() - ref).abs().max().item()
    assert err <= 1e-4 * ref.abs().max().item(), err
