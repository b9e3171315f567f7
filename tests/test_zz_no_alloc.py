"""libraspec_confidence_noalloc: the confidence step on the library's static
scratch (no workspace, no allocation) against libraspec_confidence.

The file name sorts last so that these tests also run after every other test
in one process; each test starts from whatever state the scratch was left in.
"""
import ctypes

import numpy as np
import pytest
import torch

from helpers import PROB_ATOL, cuda
from paper_2608_08721_gb300 import binding as lr
from paper_2608_08721_gb300 import workloads


def test_rejects_too_many_rows_before_any_cuda_call():
    # B*K above the scratch limit: EUNSUPPORTED with no pointer touched
    lib = lr.load()
    rc = lib.libraspec_confidence_noalloc(None, None, None, lr.NOALLOC_MAX_ROWS // 16 + 1, 16, 100, None, None,
                                          None, None)
    assert rc == lr.EUNSUPPORTED
    assert lib.libraspec_confidence_noalloc(None, None, None, 1, 4, 0, None, None, None, None) == lr.EINVAL


def _compare(conf, dstat, conf_ref, dstat_ref):
    a, r = conf.cpu().numpy(), conf_ref.cpu().numpy()
    assert np.max(np.abs(a - r)) <= PROB_ATOL
    np.testing.assert_array_equal(dstat[..., 0].cpu().numpy(), dstat_ref[..., 0].cpu().numpy())
    np.testing.assert_allclose(dstat[..., 1].cpu().numpy(), dstat_ref[..., 1].cpu().numpy(), rtol=2e-6)


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["tiny", "8b", "sampling", "ragged"])
def test_noalloc_matches_workspace_entry_point_twice(name):
    w = workloads.WORKLOADS[name]
    inp = workloads.logits(w, device=cuda())
    x, tok, temp = inp["draft_logits"], inp["draft_tokens"], inp["temperature"]
    assert w.B * w.K <= lr.NOALLOC_MAX_ROWS
    ws = lr.Workspace(w.B, w.K, w.V, device=cuda())
    conf_ref, dstat_ref = lr.libraspec_confidence(x, tok, temp, ws)
    for _ in range(2):  # two calls in a row: the tickets must be clear again
        conf = torch.full((w.B, w.K), -1.0, device=cuda())
        dstat = torch.full((w.B, w.K, 2), -1.0, device=cuda())
        status = torch.full((1,), -1, dtype=torch.int32, device=cuda())
        lr.libraspec_confidence_noalloc(x, tok, temp, conf, dstat, status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        _compare(conf, dstat, conf_ref, dstat_ref)


@pytest.mark.gpu
def test_noalloc_at_the_row_limit_and_after_a_violation():
    # a call that raises a status bit, then the largest allowed call: the
    # status word of the second call starts clear again
    g = torch.Generator(device="cuda").manual_seed(17)
    B, K, V = 64, 64, 777
    assert B * K == lr.NOALLOC_MAX_ROWS
    x = torch.randn((B, K, V), generator=g, device=cuda()) * 2
    tok = torch.randint(0, V, (B, K), generator=g, device=cuda(), dtype=torch.int32)
    temp = torch.rand((B,), generator=g, device=cuda()) * (torch.arange(B, device=cuda()) % 2)
    status = torch.zeros((1,), dtype=torch.int32, device=cuda())
    bad = tok.clone()
    bad[3, 5] = V
    conf = torch.empty((B, K), device=cuda())
    lr.libraspec_confidence_noalloc(x, bad, temp, conf, None, status)
    torch.cuda.synchronize()
    assert int(status.item()) & lr.ST_BAD_TOKEN
    dstat = torch.empty((B, K, 2), device=cuda())
    lr.libraspec_confidence_noalloc(x, tok, temp, conf, dstat, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    conf_ref, dstat_ref = lr.libraspec_confidence(x, tok, temp, lr.Workspace(B, K, V, device=cuda()))
    _compare(conf, dstat, conf_ref, dstat_ref)
    with pytest.raises(ValueError, match="static scratch limit"):
        lr.libraspec_confidence_noalloc(torch.zeros((B + 1, K, V), device=cuda()),
                                        torch.zeros((B + 1, K), dtype=torch.int32, device=cuda()),
                                        torch.zeros(B + 1, device=cuda()), torch.empty((B + 1, K), device=cuda()))


@pytest.mark.gpu
def test_noalloc_calls_no_allocator():
    # the entry point itself allocates nothing: torch's allocator is not
    # called and free device memory is unchanged across the call
    w = workloads.WORKLOADS["tiny"]
    inp = workloads.logits(w, device=cuda())
    conf = torch.empty((w.B, w.K), device=cuda())
    lr.libraspec_confidence_noalloc(inp["draft_logits"], inp["draft_tokens"], inp["temperature"], conf)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    n0 = torch.cuda.memory_stats().get("allocation.all.allocated", 0)
    lr.load().libraspec_confidence_noalloc(
        ctypes.c_void_p(inp["draft_logits"].data_ptr()), ctypes.c_void_p(inp["draft_tokens"].data_ptr()),
        ctypes.c_void_p(inp["temperature"].data_ptr()), w.B, w.K, w.V, ctypes.c_void_p(conf.data_ptr()), None,
        None, ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    torch.cuda.synchronize()
    assert torch.cuda.memory_stats().get("allocation.all.allocated", 0) == n0
    # device-wide free memory can move for reasons outside the call (the driver, other processes);
    # an allocation of the call's scratch (4.2 MB, in 2 MB pages) would take more than this
    assert free0 - torch.cuda.mem_get_info()[0] < (1 << 20)
