"""Failure detection on the GPU without a fault: a bounded wait that runs out.

The kernels' waits (the draws waiting for their sequence's decision, the
attention's grid barriers and pipeline barriers) give up after a time limit,
set LIBRASPEC_ST_TIMEOUT and return instead of hanging. Here the draws' wait
is pointed at a flag that nothing sets, with a short limit: the status must
report the timeout, the launch must return, and the same context and a
re-initialised workspace must then run a verify round that matches the
oracle."""
import time

import numpy as np
import pytest
import torch

from helpers import check_attn, cuda
from paper_2608_08721_gb300 import binding as lr
from paper_2608_08721_gb300 import workloads

pytestmark = pytest.mark.gpu


def test_bounded_wait_runs_out_and_the_context_stays_usable(orc):
    w = workloads.WORKLOADS["tiny"]
    kv = workloads.kv_lengths(w)
    lay = workloads.layer(w, 0, kv, device=cuda())
    ws = lr.Workspace(w.B, w.K, w.V, w.Hq, w.Hkv, w.d, lay["Kc"].shape[2], device=cuda())

    # a flag that nothing sets: the wait gives up after 5 ms
    flag = torch.zeros((1,), dtype=torch.int32, device=cuda())
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    seen = lr.libraspec_selftest_wait(flag, 5_000_000, ws)
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    assert int(seen.item()) == 0
    assert dt >= 0.005 and dt < 1.5, "the wait took %.3f s" % dt
    assert lr.libraspec_get_status(ws) & lr.ST_TIMEOUT

    # a set flag is seen at once and raises nothing
    flag.fill_(1)
    seen = lr.libraspec_selftest_wait(flag, 5_000_000, ws)
    torch.cuda.synchronize()
    assert int(seen.item()) == 1
    assert lr.libraspec_get_status(ws) == 0

    # the same context, a re-initialised workspace: a verify round matches the oracle
    ws = lr.Workspace(w.B, w.K, w.V, w.Hq, w.Hkv, w.d, lay["Kc"].shape[2], device=cuda())
    inp = workloads.logits(w, device=cuda())
    cost = workloads.cost_table(w)
    out = lr.libraspec_verify_round(inp["draft_logits"], inp["draft_tokens"], inp["temperature"],
                                    torch.tensor(cost, device=cuda()), inp["target_logits"], [lay],
                                    torch.tensor(kv, device=cuda()), w.philox_seed, ws)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    q, _ = orc.confidence(inp["draft_logits"].cpu().numpy(), inp["draft_tokens"].cpu().numpy(),
                          inp["temperature"].cpu().numpy())
    L, sflag = orc.select_lengths(q, cost.astype(np.float64))
    assert not sflag.any()
    np.testing.assert_array_equal(out.L.cpu().numpy(), L)
    n, bonus, aflag = orc.accept(inp["target_logits"].cpu().numpy(), inp["draft_logits"].cpu().numpy(),
                                 inp["draft_tokens"].cpu().numpy(), L, inp["temperature"].cpu().numpy(),
                                 w.philox_seed)
    assert not aflag.any()
    np.testing.assert_array_equal(out.n_accepted.cpu().numpy(), n)
    np.testing.assert_array_equal(out.bonus_token.cpu().numpy(), bonus)
    O_ref, lse_ref = orc.verify_attn(lay["Q"], lay["Kc"], lay["Vc"], kv, L)
    check_attn(out.O[0], None, O_ref, lse_ref, L)


def test_selftest_wait_rejects_bad_arguments():
    ws = lr.Workspace(1, 1, 8, device=cuda())
    flag = torch.zeros((1,), dtype=torch.int32, device=cuda())
    for limit in (0, 3_000_000_000):
        with pytest.raises(lr.LibraspecError):
            lr.libraspec_selftest_wait(flag, limit, ws)
