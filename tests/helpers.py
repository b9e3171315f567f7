"""Shared helpers of the parity tests (GPU path vs. CPU oracle)."""
import numpy as np
import torch

# Tolerances of the contract: probabilities within 1e-5 absolute; attention
# within max-abs 2e-2 and rel 1e-2 (bf16 in, fp32 accumulate). Because
# N(0,1) keys make the softmax nearly flat (|O| ~ 1/sqrt(kv_len)), attention
# is also held to a relative Frobenius error per (sequence, head) and to lse.
PROB_ATOL = 1e-5
ATTN_ATOL, ATTN_RTOL = 2e-2, 1e-2
ATTN_FRO_REL = 1e-2
LSE_ATOL = 1e-3


def cuda():
    return torch.device("cuda", 0)


def check_attn(O_gpu, lse_gpu, O_ref, lse_ref, L, rows=None, fro=True):
    """Compare verified rows t <= L_b (all, or the listed (b, h, t))."""
    O = O_gpu.float().cpu().numpy()
    lse = None if lse_gpu is None else lse_gpu.cpu().numpy()
    worst = 0.0
    if rows is None:
        B = O.shape[0]
        for b in range(B):
            n = int(L[b]) + 1
            a, r = O[b, :n], O_ref[b, :n]
            err = np.abs(a - r)
            bound = ATTN_ATOL + ATTN_RTOL * np.abs(r)
            assert np.all(err <= bound), "b=%d max err %.3e" % (b, err.max())
            worst = max(worst, float(err.max()))
            if fro:
                for h in range(a.shape[1]):
                    num = np.linalg.norm(a[:, h] - r[:, h])
                    den = np.linalg.norm(r[:, h]) + 1e-30
                    assert num / den <= ATTN_FRO_REL, "b=%d h=%d fro %.3e" % (b, h, num / den)
            if lse is not None:
                assert np.all(np.abs(lse[b, :n] - lse_ref[b, :n]) <= LSE_ATOL)
    else:
        for b, h, t in rows:
            a, r = O[b, t, h], O_ref[b, t, h]
            err = np.abs(a - r)
            assert np.all(err <= ATTN_ATOL + ATTN_RTOL * np.abs(r)), (b, h, t, err.max())
            if fro:
                assert np.linalg.norm(a - r) <= ATTN_FRO_REL * (np.linalg.norm(r) + 1e-30), (b, h, t)
            if lse is not None:
                assert abs(lse[b, t, h] - lse_ref[b, t, h]) <= LSE_ATOL
            worst = max(worst, float(err.max()))
    return worst


def assert_exact_unless_flagged(gpu, ref, flag, what):
    gpu, ref, flag = (np.asarray(x) for x in (gpu, ref, flag))
    bad = (gpu != ref) & (flag == 0)
    assert not bad.any(), "%s differs on unflagged sequences %s: gpu %s oracle %s" % (
        what, np.nonzero(bad)[0].tolist(), gpu[bad].tolist(), ref[bad].tolist())
    return int((flag != 0).sum())


def assert_flag_budget(n_flagged, B, what, per=16):
    """Flagged sequences are left out of the exact comparison; keep them few
    (at most max(1, B / per)) so that a flag rule too wide to test anything
    shows up. The count is printed for the record."""
    budget = max(1, B // per)
    print("%s: %d of %d sequences flagged (budget %d)" % (what, n_flagged, B, budget))
    assert n_flagged <= budget, "%s: %d of %d sequences flagged, budget %d" % (what, n_flagged, B, budget)
