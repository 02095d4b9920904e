"""featfix_op_verify_noalloc: the paid-check kernel for callers that cannot
allocate device memory (a host framework that owns all GPU memory, a
memory-budgeted service, a latency-critical loop).  Its partial sums live in a
fixed 16 KiB array inside the library instead of a caller workspace.

Checked through the C ABI against featfix_op_verify (which uses a caller
workspace) on two calls in a row with different sizes, so a stale partial
left in the shared array by the first call would show up in the second.
This file is collected last on purpose."""

import pytest
import torch

from paper_2607_27842_gb300 import featfix as ff

pytestmark = pytest.mark.gpu

TD = {"f32": torch.float32, "bf16": torch.bfloat16}


def inputs(dtype, n, seed):
    g = torch.Generator().manual_seed(seed)
    hist = [(torch.randn(n, generator=g) * 0.05).to(TD[dtype]).cuda() for _ in range(3)]
    u = torch.randn(n, generator=g).to(TD[dtype]).cuda()
    hf = (u.float().cpu() + torch.randn(n, generator=g) * 0.05).to(TD[dtype]).cuda()
    return hist, u, hf


def reference(dtype, hist, w, u, hf, write_draft):
    """The existing entry point, with a caller-allocated workspace."""
    n = u.numel()
    ws = torch.empty(ff.featfix_op_verify_workspace(n), dtype=torch.uint8, device="cuda")
    sums = torch.zeros(4, dtype=torch.float64, device="cuda")
    uu = u.clone()
    ff.featfix_op_verify(dtype, uu, hist, w, hf, sums, ws, write_draft=write_draft)
    torch.cuda.synchronize()
    return sums.cpu(), uu


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_noalloc_verify_matches_allocating_entry_point_twice(cuda, dtype):
    w = [1.5, -0.75, 0.25]
    for call, (n, write_draft) in enumerate([(4718592 + 8, False), (50000 + 3, True)]):
        hist, u, hf = inputs(dtype, n, seed=100 + call)
        want_sums, want_u = reference(dtype, hist, w, u, hf, write_draft)
        sums = torch.full((4,), -1.0, dtype=torch.float64, device=cuda)
        uu = u.clone()
        ff.featfix_op_verify_noalloc(dtype, uu, hist, w, hf, sums, write_draft=write_draft)
        torch.cuda.synchronize()
        # same kernel and reduction order: the tolerance of the verify tests
        # (2e-5 relative) holds, and in practice the sums agree exactly
        torch.testing.assert_close(sums.cpu(), want_sums, rtol=2e-5, atol=0.0)
        assert torch.equal(uu, want_u if write_draft else u)


def test_noalloc_verify_rejects_bad_arguments(cuda):
    x = torch.zeros(1024, device=cuda)
    sums = torch.zeros(4, dtype=torch.float64, device=cuda)
    with pytest.raises(ff.FeatFixError) as e:
        ff.featfix_op_verify_noalloc("f32", x, [x] * 5, [1.0] * 5, x, sums)
    assert e.value.status == ff.ERR_INVALID_ARG
    with pytest.raises(ff.FeatFixError) as e:
        ff.featfix_op_verify_noalloc("f32", x[1:], [x[1:]], [1.0], x[1:], sums)   # misaligned
    assert e.value.status == ff.ERR_INVALID_ARG
