"""Deterministic column sums (the bias-gradient reduction) through the C ABI
against a fp64 reference of the same bf16 / fp32 inputs; results must be
bitwise reproducible across calls."""
import numpy as np
import pytest
import torch

from paper_2504_13850_gb300 import api, build

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    api.lib()


@pytest.mark.parametrize("rows,cols,dtype", [(16384, 256, torch.bfloat16), (4096, 512, torch.bfloat16),
                                             (1000, 10, torch.float32), (33, 24, torch.bfloat16),
                                             (1, 8, torch.float32), (777, 100, torch.bfloat16)])
def test_column_sums(rows, cols, dtype):
    g = torch.Generator(device="cuda").manual_seed(rows * 31 + cols)
    x = torch.randn(rows, cols, device="cuda", generator=g).to(dtype)
    out = torch.empty(cols, device="cuda")
    assert api.column_sums(x, out) == api.OK
    torch.cuda.synchronize()
    ref = x.double().sum(0).cpu().numpy()
    # fp32 sums of <= 16384 terms: relative error well below 1e-5 of sum |x|
    bound = 1e-5 * x.double().abs().sum(0).cpu().numpy() + 1e-30
    assert np.all(np.abs(out.cpu().numpy() - ref) <= bound)
    out2 = torch.empty(cols, device="cuda")
    assert api.column_sums(x, out2) == api.OK
    torch.cuda.synchronize()
    assert torch.equal(out, out2)


def test_column_sums_rejects_bad_arguments():
    x = torch.zeros(4, 4, device="cuda")
    out = torch.empty(4, device="cuda")
    assert api.lib().fo_column_sums(x.data_ptr(), 7, 4, 4, out.data_ptr(), None) == api.ERR_ARG
    assert api.lib().fo_column_sums(x.data_ptr(), api.DTYPE_F32, 0, 4, out.data_ptr(), None) == api.ERR_ARG
