"""fo_column_sums_noalloc: the column sums for callers that cannot allocate
device memory when they need them (inside a stream capture, under an
outside allocator, or in loops that must not allocate after start-up).  It
must give what the allocating entry point fo_column_sums gives, call after
call, while its partial sums live in the library's fixed device array.

This file is collected last, so a run that stops at the first failure has
run every other test before it."""
import pytest
import torch

from paper_2504_13850_gb300 import api, build

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    api.lib()


def test_noalloc_matches_allocating_entry_point_on_two_calls():
    gen = torch.Generator(device="cuda").manual_seed(7)
    # the vectorised bf16 path, the fp32 path, and bf16 with a column count
    # that is not a multiple of 8 (the generic kernel)
    shapes = [(16384, 256, torch.bfloat16), (4096, 512, torch.float32), (3000, 100, torch.bfloat16)]
    for rows, cols, dtype in shapes:          # two calls in a row, different inputs
        x = torch.randn(rows, cols, device="cuda", generator=gen).to(dtype)
        ref = torch.empty(cols, device="cuda")
        got = torch.full((cols,), float("nan"), device="cuda")
        assert api.column_sums(x, ref) == api.OK
        assert api.column_sums_noalloc(x, got) == api.OK
        torch.cuda.synchronize()
        # same kernels in the same order: equal bit for bit (within the
        # 1e-5 bound the column-sum tests use, a fortiori)
        assert torch.equal(got, ref)
        scale = x.double().abs().sum(0)
        assert bool(((got.double() - x.double().sum(0)).abs() <= 1e-5 * scale + 1e-30).all())


def test_noalloc_rejects_inputs_beyond_its_scratch():
    x = torch.zeros(131072, 1024, dtype=torch.bfloat16, device="cuda")   # 1024 * 1024 partials
    out = torch.empty(1024, device="cuda")
    assert api.column_sums_noalloc(x, out) == api.ERR_ARG
    assert "exceed" in api.last_error()


def test_noalloc_at_exactly_its_scratch_size():
    """ceil(rows / 128) * cols = 262,144 partial sums, the whole array."""
    rows, cols = 32768 * 128, 8
    x = torch.randn(rows, cols, device="cuda").to(torch.bfloat16)
    ref = torch.empty(cols, device="cuda")
    got = torch.full((cols,), float("nan"), device="cuda")
    assert api.column_sums(x, ref) == api.OK
    assert api.column_sums_noalloc(x, got) == api.OK
    torch.cuda.synchronize()
    assert torch.equal(got, ref)


def test_both_entry_points_reject_more_row_chunks_than_a_grid_dimension():
    """65,536 chunks of 128 rows (4 columns: within the scratch's partial
    count) exceed the 65,535 blocks of one grid dimension: refused with a
    reason rather than a failed launch."""
    x = torch.zeros(65536 * 128, 4, dtype=torch.bfloat16, device="cuda")
    out = torch.empty(4, device="cuda")
    for call in (api.column_sums, api.column_sums_noalloc):
        assert call(x, out) == api.ERR_ARG
        assert "65,535 chunks" in api.last_error()
