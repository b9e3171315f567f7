"""Measure a workload's verification cost table on the GPU and freeze it to JSON.

T_verify(L) for L = 0..K is the latency of one verify-attention launch
(``libraspec_verify_attn_layers``, one layer) over the workload's batch with
every sequence at length L: the median of CUDA-event timings of a replayed
CUDA graph, with the L2 cache flushed before each replay. The table is
normalised to T(0) = 1 and made non-decreasing by a running maximum (a
latency that dips at a larger L is taken as the smaller L's), the reading of
the non-constant marginal cost that the selector's Thm. 4 criterion uses.

The frozen table is an input of the length selection, given to the CUDA path
and to the CPU oracle alike; it is a timing of the kernel, not an output of
its arithmetic.

    python -m paper_2608_08721_gb300.measure_cost_table [--workload ragged] [--reps 30]
"""
from __future__ import annotations

import argparse
import datetime
import json
import os
import statistics
import subprocess

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
DATA = os.path.join(HERE, "data")


def table_path(workload: str) -> str:
    return os.path.join(DATA, "%s_verify_attn_cost.json" % workload)


def measure(workload: str, reps: int) -> dict:
    import torch

    from paper_2608_08721_gb300 import binding as lr
    from paper_2608_08721_gb300 import build as cuda_build
    from paper_2608_08721_gb300 import workloads

    cuda_build.build()
    dev = torch.device("cuda", 0)
    w = workloads.WORKLOADS[workload]
    kv = workloads.kv_lengths(w)
    lay = workloads.layer(w, 0, kv, device=dev)
    S = lay["Kc"].shape[2]
    ws = lr.Workspace(w.B, w.K, w.V, w.Hq, w.Hkv, w.d, S, device=dev)
    kv_t = torch.tensor(kv, device=dev)
    O = torch.empty_like(lay["Q"])
    layers = [dict(lay, O=O)]
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    side = torch.cuda.Stream(device=dev)
    us = []
    for L in range(w.K + 1):
        Lt = torch.full((w.B,), L, dtype=torch.int32, device=dev)
        for _ in range(3):
            lr.libraspec_verify_attn_layers(layers, kv_t, Lt, ws)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=side):
            lr.libraspec_verify_attn_layers(layers, kv_t, Lt, ws)
        times = []
        for _ in range(reps):
            flush.fill_(1.0)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            g.replay()
            b.record()
            torch.cuda.synchronize()
            times.append(a.elapsed_time(b) * 1000.0)
        us.append(statistics.median(times))
        if lr.libraspec_get_status(ws) != 0:
            raise RuntimeError("device status set while timing L = %d" % L)
    t = np.maximum.accumulate(np.asarray(us) / us[0])
    try:
        clocks = subprocess.run(["nvidia-smi", "--query-gpu=clocks.sm,clocks.max.sm", "--format=csv,noheader"],
                                capture_output=True, text=True).stdout.strip()
    except OSError:
        clocks = ""
    return {
        "workload": workload,
        "kernel": "libraspec_verify_attn_layers, one layer, every sequence at length L",
        "B": w.B, "K": w.K, "gqa": "%d/%d" % (w.Hq, w.Hkv), "head_dim": w.d,
        "kv_len": [int(kv.min()), int(kv.max())],
        "L": list(range(w.K + 1)),
        "latency_us": [round(x, 3) for x in us],
        "T": [float(np.float32(x)) for x in t],
        "method": "median of %d CUDA-graph replays per L, L2 flushed before each; T = latency / latency[0], "
                  "then a running maximum" % reps,
        "gpu": torch.cuda.get_device_name(0), "clocks_sm_and_max": clocks,
        "measured": datetime.datetime.now(datetime.timezone.utc).strftime("%Y-%m-%dT%H:%M:%SZ"),
    }


def main():
    p = argparse.ArgumentParser()
    p.add_argument("--workload", default="ragged")
    p.add_argument("--reps", type=int, default=30)
    p.add_argument("--out", default="")
    args = p.parse_args()
    rec = measure(args.workload, args.reps)
    out = args.out or table_path(args.workload)
    os.makedirs(os.path.dirname(out), exist_ok=True)
    with open(out, "w") as f:
        json.dump(rec, f, indent=1)
    print(json.dumps({"out": out, "latency_us": rec["latency_us"], "T": rec["T"]}))


if __name__ == "__main__":
    main()
