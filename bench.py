"""Benchmark of the LibraSpec verify round on GB300.

One step = one verify round over one batch: drafter confidence + length
selection, every verify-attention layer, acceptance. Default workload: the
ragged heavy batch (B=64 sequences, K=32, V=128256, GQA 32/8 attention over
KV lengths log-uniform in [512, 32768], greedy and T=0.8 sequences
alternating); the sampling batch (B=16) and the 8B-class greedy round (B=1,
32 layers) are measured in the same run under "also".

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config NAME] [--also A,B] [--impl ours|reference]

Variants of the round (the default is the chain draft on dense caches):
  --selector alpha   Algorithm 1's alpha-mode length search instead of Thm. 4's scan;
  --logits bf16      bf16 drafter and target logits;
  --page-size P      KV caches in pages of P keys behind block tables;
  --lm-head          the confidence from the drafter's hidden states and the LM head
                     (the statistics in the GEMM's epilogue, no drafter logits);
  --tree N           a DDTree-shaped draft tree of N nodes: tree-masked attention and the
                     tree walk (greedy or drawing, per the workload's temperatures) replace
                     the chain's attention and acceptance.

N > 1 runs under torchrun, one process per GPU; every rank verifies its own
batch (weak scaling, no data-path collective) and rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "verify-round µs (select+attn+accept) and HBM TB/s vs ~8 TB/s, batch 1–64"
NOMINAL_HBM_GBS = 8000.0
ATTN_LAYERS_PER_LAUNCH = 64  # LIBRASPEC_ATTN_LAYERS_PER_LAUNCH
L2_BYTES = 129e6


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=0, help="timed steps (0: enough for ~2 s)")
    p.add_argument("--warmup", type=int, default=20)
    p.add_argument("--config", default="ragged")
    p.add_argument("--also", default="sampling,8b",
                   help="workloads also measured in the same run, each under its own key (empty: none)")
    p.add_argument("--also-steps", type=int, default=20, help="timed rounds of each 'also' workload")
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--e2e-steps", type=int, default=50)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-seconds", type=float, default=12.0, help="CPU work budget of the oracle sample")
    p.add_argument("--logits", default="f32", choices=["f32", "bf16"],
                   help="dtype of the drafter and target logits (bf16: libraspec_*_bf16, half the bytes)")
    p.add_argument("--selector", default="gain", choices=["gain", "alpha"],
                   help="gain: the Thm. 4 marginal-gain scan; alpha: Algorithm 1's alpha-mode search")
    p.add_argument("--alpha", type=float, default=2.2, help="alpha of the alpha-mode search (Sec. 4: 2.2)")
    p.add_argument("--tree", type=int, default=0,
                   help="verify a DDTree-shaped draft tree of this many nodes (depth <= K) instead of the chain")
    p.add_argument("--page-size", type=int, default=0,
                   help="keep the KV cache in pages of this many keys behind block tables (0: dense)")
    p.add_argument("--lm-head", action="store_true",
                   help="compute the confidence from the drafter's hidden states and the LM head (fused GEMM "
                        "epilogue, logits never stored) instead of from drafter logits")
    p.add_argument("--block-size", type=int, default=0,
                   help="first drafted block of the alpha-mode search (0: 2/3 of K, as 16 of d_max 24)")
    return p.parse_args()


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}, "fallback"


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------
_REASONS = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]


class ClockSampler:
    def __init__(self, gpu_index: int):
        self.path = tempfile.mktemp(suffix=".csv")
        self.proc = None
        self.gpu = gpu_index

    def __enter__(self):
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + q,
                                          "--format=csv,noheader,nounits", "-lms", "100"], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.f.close()

    def summary(self):
        out = {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        try:
            rows = [l.strip().split(",") for l in open(self.path) if l.strip()]
        except OSError:
            return out
        sm, mx, reasons = [], [], set()
        for r in rows:
            r = [x.strip() for x in r]
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                mx.append(float(r[2]))
            except ValueError:
                continue
            for name, val in zip(_REASONS, r[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        if sm:
            out.update(sm_mhz=statistics.median(sm), sm_max_mhz=max(mx), samples=len(sm))
        out["reasons"] = sorted(reasons)
        return out


def physical_gpu(local_rank):
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        ids = [x.strip() for x in vis.split(",") if x.strip()]
        if local_rank < len(ids):
            return ids[local_rank]
    return str(local_rank)


# ---------------------------------------------------------------------------
# algorithmic bytes (what the method must move)
# ---------------------------------------------------------------------------
def round_bytes(w, kv, L, temperature, n_acc, logit_bytes=4, L_tree=None):
    """Algorithmic bytes of one round. L_tree: node counts of draft trees
    (their attention and acceptance read every node's rows)."""
    conf = w.B * w.K * w.V * logit_bytes
    select = w.B * w.K * 4 + (w.K + 1) * 4
    Lv = L if L_tree is None else L_tree
    accept = float(np.sum((Lv + 1).astype(np.int64) * w.V * logit_bytes))
    if L_tree is None:
        rejected_sampling = np.sum((n_acc < L) & (temperature > 0))
        accept += float(rejected_sampling) * 2 * w.V * logit_bytes
    from paper_2608_08721_gb300 import workloads

    attn_launch = workloads.attn_bytes(w, kv, Lv)
    return {"conf": conf, "select": select, "attn_per_launch": attn_launch, "attn": attn_launch * w.n_layers,
            "accept": accept, "total": conf + select + accept + attn_launch * w.n_layers}


# ---------------------------------------------------------------------------
# the oracle on the host cores (CPU baseline / reference arm)
# ---------------------------------------------------------------------------
def _subset(w, inp_host, layers_host, kv, seqs):
    """The first ``seqs`` sequences of the batch (host inputs and one layer each)."""
    sub = {k: (v[:seqs] if k != "cost_table" else v) for k, v in inp_host.items()}
    lays = [{k: v[:seqs] for k, v in lay.items()} for lay in layers_host]
    return w.scaled(B=seqs), sub, lays, kv[:seqs]


def oracle_round_time(w, inp_host, layers_host, kv, budget_s, conf_fn=None, attn_fn=None, variant="",
                      threads=None, seqs=None):
    """Time the oracle's round on a bounded sample: the full logits steps and
    one attention layer (scaled to all layers). Repeats the sample until the
    budget is spent; returns (us per round, threads, sample text).
    conf_fn() -> q replaces the confidence from drafter logits (the LM-head
    variant); attn_fn(layer, L) replaces the dense attention (paged caches).
    threads: OpenMP threads (default: all cores). seqs: time the first seqs
    sequences only and scale the time by B / seqs."""
    import oracle

    oracle.build()
    threads = threads or (os.cpu_count() or 1)
    oracle.set_threads(threads)
    B = w.B
    if seqs and seqs < B:
        w, inp_host, layers_host, kv = _subset(w, inp_host, layers_host, kv, seqs)
    scale = B / w.B
    cost = np.asarray(inp_host["cost_table"], np.float64)
    times_logits, times_attn = [], []
    t_end = time.perf_counter() + budget_s
    while True:
        t0 = time.perf_counter()
        if conf_fn is not None:
            q = conf_fn()
        else:
            q, _ = oracle.confidence(inp_host["draft_logits"], inp_host["draft_tokens"], inp_host["temperature"])
        L, _ = oracle.select_lengths(q, cost)
        oracle.accept(inp_host["target_logits"], inp_host["draft_logits"], inp_host["draft_tokens"], L,
                      inp_host["temperature"], w.philox_seed)
        t1 = time.perf_counter()
        lay = layers_host[len(times_attn) % len(layers_host)]
        if attn_fn is not None:
            attn_fn(lay, L)
        else:
            oracle.verify_attn(lay["Q"], lay["Kc"], lay["Vc"], kv, L)
        t2 = time.perf_counter()
        times_logits.append(t1 - t0)
        times_attn.append(t2 - t1)
        if time.perf_counter() > t_end or len(times_attn) >= 50:
            break
    per_round = (statistics.median(times_logits) + statistics.median(times_attn) * w.n_layers) * scale
    sample = ("%d repetition(s) of: confidence, selection and acceptance on %s plus ONE of the %d "
              "attention layers (fp64 C oracle, %d thread%s); attention time scaled by %d layers%s%s" %
              (len(times_attn), "the full batch" if scale == 1 else "%d of the %d sequences" % (w.B, B),
               w.n_layers, threads, "" if threads == 1 else "s", w.n_layers,
               "" if scale == 1 else ", the round's time scaled by %d/%d sequences" % (B, w.B), variant))
    return per_round * 1e6, threads, sample


def oracle_flags(w, host, L_gpu, n_gpu, bonus_gpu):
    """Oracle flags of the chain round (near-threshold selections and draws)
    and the GPU's disagreements with the oracle outside them. The acceptance
    is compared given the GPU's lengths."""
    import oracle

    oracle.build()
    oracle.set_threads(os.cpu_count() or 1)
    q, _ = oracle.confidence(host["draft_logits"], host["draft_tokens"], host["temperature"])
    L, sflag = oracle.select_lengths(q, np.asarray(host["cost_table"], np.float64))
    n, bonus, aflag = oracle.accept(host["target_logits"], host["draft_logits"], host["draft_tokens"],
                                    L_gpu.astype(np.int32), host["temperature"], w.philox_seed)
    sel_bad = (L != L_gpu) & (sflag == 0)
    acc_bad = ((n != n_gpu) | (bonus != bonus_gpu)) & (aflag == 0)
    return {"sequences": int(w.B), "select_flagged": int(sflag.sum()), "accept_flagged": int(aflag.sum()),
            "select_mismatch_unflagged": int(sel_bad.sum()), "accept_mismatch_unflagged": int(acc_bad.sum())}


def oracle_tree_round_time(w, host, tree_host, layer_host, kv, budget_s):
    """The oracle's tree round on a bounded sample: confidence and selection
    on the batch, the greedy tree walk, and ONE attention layer scaled to all."""
    import oracle

    oracle.build()
    threads = os.cpu_count() or 1
    oracle.set_threads(threads)
    cost = np.asarray(host["cost_table"], np.float64)
    t_logits, t_attn = [], []
    t_end = time.perf_counter() + budget_s
    while True:
        t0 = time.perf_counter()
        q, _ = oracle.confidence(host["draft_logits"], host["draft_tokens"], host["temperature"])
        oracle.select_lengths(q, cost)
        oracle.accept_tree(tree_host["target_logits"], tree_host["draft_tokens"], tree_host["parent"],
                           tree_host["L"], host["temperature"], w.philox_seed)
        t1 = time.perf_counter()
        oracle.verify_attn_tree(layer_host["Q"], layer_host["Kc"], layer_host["Vc"], kv, tree_host["L"],
                                tree_host["parent"])
        t2 = time.perf_counter()
        t_logits.append(t1 - t0)
        t_attn.append(t2 - t1)
        if time.perf_counter() > t_end or len(t_attn) >= 50:
            break
    per_round = statistics.median(t_logits) + statistics.median(t_attn) * w.n_layers
    sample = ("%d repetition(s) of: confidence, selection and the tree walk on the full batch plus ONE of "
              "the %d tree-attention layers (fp64 C oracle, %d threads); attention time scaled by %d layers" %
              (len(t_attn), w.n_layers, threads, w.n_layers))
    return per_round * 1e6, threads, sample


def tree_flops(parent, kv, L, Hq, d):
    """Attention flops of one tree layer counting visible keys only:
    Σ_b Σ_t Hq · 4d · (kv_b + depth_t + 1)."""
    tot = 0.0
    for b in range(parent.shape[0]):
        n = int(L[b])
        dep = np.zeros(n + 1, np.int64)
        for t in range(1, n + 1):
            dep[t] = dep[parent[b, t]] + 1
        tot += float(Hq) * 4.0 * d * float(np.sum(int(kv[b]) + dep + 1))
    return tot


def host_inputs(w, kv, n_layer_samples=1):
    from paper_2608_08721_gb300 import workloads

    inp = workloads.logits(w)
    host = {k: v.numpy() for k, v in inp.items()}
    host["cost_table"] = workloads.cost_table(w, kv)
    layers = [workloads.layer(w, l, kv) for l in range(n_layer_samples)]
    return host, layers


def workload_config(args, w, kv, Lh, world, block_size):
    """The workload a line measures (shapes, the lengths selected, the
    variant); the same dict in both arms for the same arguments."""
    return {"workload": w.name, "B": w.B, "K": w.K, "V": w.V, "layers": w.n_layers,
            "resident_kv_layers": w.resident_layers if w.resident_layers else w.n_layers,
            "gqa": "%d/%d" % (w.Hq, w.Hkv), "head_dim": w.d,
            "kv_len": [int(kv.min()), int(kv.max())], "selected_L": [int(Lh.min()), int(Lh.max())],
            "selected_L_mean": round(float(Lh.mean()), 3),
            "cost_table": w.cost[0] if w.cost[0] != "measured" else "measured (%s)" % w.cost[1],
            "selector": ("alpha (Algorithm 1, alpha %g, first block %d)" % (args.alpha, block_size)
                         if args.selector == "alpha" else "marginal gain (Thm. 4)"),
            "logits": args.logits,
            "draft": ("DDTree-shaped tree of %d nodes (best-first, depth <= %d), tree walk" %
                      (args.tree, w.K) if args.tree else "chain"),
            "kv_cache": "paged, %d keys per page" % args.page_size if args.page_size else "dense",
            "confidence": ("from hidden states [%d, %d] and a %d x %d LM head (fused epilogue)" %
                           (w.B * w.K, w.hidden, w.V, w.hidden) if args.lm_head else "from drafter logits"),
            "parallelism": "dp%d (independent sequences)" % world,
            "l2": l2_note(w, kv)}


def l2_note(w, kv):
    """Whether a step's distinct inputs (both logit blocks and the resident
    KV caches) exceed the 129 MB L2; timed steps are not separated by a flush."""
    n_res = w.resident_layers if w.resident_layers else w.n_layers
    mb = (w.B * w.K * w.V * 4 + w.B * (w.K + 1) * w.V * 4 +
          n_res * float(np.sum(kv.astype(np.float64))) * w.Hkv * w.d * 2 * 2) / 1e6
    if mb > 129:
        return "no flush: about %d MB of distinct inputs per step exceed the 129 MB L2" % (int(mb) // 10 * 10)
    return "no flush: about %d MB of inputs per step fit the 129 MB L2 (timed warm)" % max(1, int(mb))


def run_reference(args, rank, world):
    """The reference arm: the oracle as it stands, on this host's cores."""
    from paper_2608_08721_gb300 import workloads

    if rank != 0:
        return
    w = workloads.WORKLOADS[args.config]
    kv = workloads.kv_lengths(w)
    host, layers = host_inputs(w, kv)
    steps = max(1, args.steps if args.steps > 0 else 3)
    budget = max(10.0, args.cpu_seconds)
    per = []
    cores, sample = 0, ""
    for _ in range(max(0, min(args.warmup, 1))):
        oracle_round_time(w, host, layers, kv, 0.0)
    for _ in range(steps):
        us, cores, sample = oracle_round_time(w, host, layers, kv, budget / steps)
        per.append(us)
    value = statistics.median(per)
    # the lengths the round selects (the oracle's; the GPU selects the same unless a sequence is flagged)
    import oracle

    q, _ = oracle.confidence(host["draft_logits"], host["draft_tokens"], host["temperature"])
    Lh, _ = oracle.select_lengths(q, np.asarray(host["cost_table"], np.float64))
    block_size = args.block_size if args.block_size > 0 else max(1, (2 * w.K) // 3)
    line = {"metric": METRIC, "value": round(value, 3), "unit": "us", "n_gpus": args.gpus, "steps": steps,
            "warmup": args.warmup, "ms_per_step": round(value / 1000, 6), "higher_is_better": False,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "impl": "reference",
            "config": workload_config(args, w, kv, np.asarray(Lh), world, block_size),
            "timing": "the fp64 C oracle's round on the host cores, a bounded sample per step (cpu_baseline)",
            "cpu_baseline": {"value": round(value, 3), "unit": "us", "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": round(value, 3), "unit": "us", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------
def attn_profile_record(kernel_file, workload):
    """ncu figures of the attention kernel on ``workload`` from the committed
    record (DRAM traffic per launch, tensor-pipe share), if they were taken on
    the current kernel source."""
    path = os.path.join(ROOT, "profiles", "verify_attn_traffic.json")
    try:
        rec = json.load(open(path))
    except (OSError, ValueError):
        return None
    sha = hashlib.sha256(open(kernel_file, "rb").read()).hexdigest()
    if rec.get("kernel_source_sha256") != sha:
        return None
    return rec.get("workloads", {}).get(workload)


def host_link(nbytes, dev):
    """Pinned host -> device copy rate: one copy of nbytes, and the same bytes
    as three copies on three streams (the staged round's parts). Median of 5."""
    import torch

    nbytes = int(nbytes) // 16 * 16
    src = torch.empty(nbytes, dtype=torch.uint8, pin_memory=True)
    dst = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    streams = [torch.cuda.Stream(device=dev) for _ in range(3)]
    third = nbytes // 3 // 16 * 16
    cuts = [0, third, 2 * third, nbytes]

    def one():
        dst.copy_(src, non_blocking=True)

    def three():
        cur = torch.cuda.current_stream()
        for i, st in enumerate(streams):
            st.wait_stream(cur)
            with torch.cuda.stream(st):
                dst[cuts[i]:cuts[i + 1]].copy_(src[cuts[i]:cuts[i + 1]], non_blocking=True)
        for st in streams:
            cur.wait_stream(st)

    out = {"bytes": nbytes}
    for name, fn in (("single_copy", one), ("three_streams", three)):
        fn()
        torch.cuda.synchronize()
        ts = []
        for _ in range(5):
            t0 = time.perf_counter()
            fn()
            torch.cuda.synchronize()
            ts.append(time.perf_counter() - t0)
        out[name + "_GBps"] = round(nbytes / statistics.median(ts) / 1e9, 1)
    return out


def measure_workload(args, w, dev, rank, world, local_rank, steps, primary):
    """One workload: the timed rounds (one CUDA graph each), a second pass of
    the same rounds as three graphs for the segments, the attention roofline,
    the logits segments, the end-to-end round through the host API, the
    oracle's flags and (primary, rank 0, one process) the CPU baseline."""
    import torch

    from paper_2608_08721_gb300 import binding as lr
    from paper_2608_08721_gb300 import dist as pdist
    from paper_2608_08721_gb300 import workloads

    kv = workloads.kv_lengths(w)
    seq_offset = rank * w.B  # weak scaling: each rank verifies its own B sequences
    inp = workloads.logits(w, device=dev)
    if args.logits == "bf16":  # as an engine's LM head emits them
        inp["draft_logits"] = inp["draft_logits"].to(torch.bfloat16)
        inp["target_logits"] = inp["target_logits"].to(torch.bfloat16)
    n_res = w.resident_layers if w.resident_layers else w.n_layers
    N = args.tree  # draft-tree node budget (0: the chain draft)
    if N and not 1 <= N <= lr.MAX_TREE_NODES:
        raise SystemExit("--tree must be in [1, %d]" % lr.MAX_TREE_NODES)
    K1 = N + 1 if N else w.K + 1   # verified positions per sequence
    S = workloads.s_cap(w, kv) if not N else (int(kv.max()) + N + 1 + 63) // 64 * 64
    P = args.page_size
    if P:
        if P % 64:
            raise SystemExit("--page-size must be a multiple of 64")
        S = -(-S // P) * P
    caches = [workloads.layer(w, l, kv, device=dev, scap=S) for l in range(n_res)]
    table = None
    if P:  # the same caches, moved into randomly permuted pages behind block tables
        max_pages = S // P
        perm = np.random.default_rng([w.data_seed, 55]).permutation(w.B * max_pages).astype(np.int32)
        table = torch.from_numpy(perm.reshape(w.B, max_pages)).to(dev)
        idx = torch.from_numpy(perm).long().to(dev)
        for c in caches:
            for key, pk in (("Kc", "Kp"), ("Vc", "Vp")):
                pages = c.pop(key).view(w.B, w.Hkv, max_pages, P, w.d).permute(0, 2, 1, 3, 4)
                pool = torch.empty((w.B * max_pages, w.Hkv, P, w.d), dtype=torch.bfloat16, device=dev)
                pool[idx] = pages.reshape(w.B * max_pages, w.Hkv, P, w.d)
                c[pk] = pool
    g = torch.Generator(device=dev).manual_seed(w.data_seed * 31 + 5)
    Qs = [torch.randn((w.B, K1, w.Hq, w.d), generator=g, device=dev).to(torch.bfloat16)
          for _ in range(w.n_layers)]
    Os = [torch.empty_like(q) for q in Qs]
    layers = [dict(caches[l % n_res], Q=Qs[l], O=Os[l]) for l in range(w.n_layers)]
    cost = torch.tensor(workloads.cost_table(w, kv), device=dev)
    kv_t = torch.tensor(kv, device=dev)
    ws = lr.Workspace(w.B, w.K, w.V, w.Hq, w.Hkv, w.d, S, device=dev)
    tree = None
    if N:
        parent = workloads.draft_tree(w.B, N, N, seed=w.data_seed, shape="ddtree", depth=w.K)
        tl = workloads.tree_logits(w, parent, N, device=dev)
        if args.logits == "bf16":
            tl["target_logits"] = tl["target_logits"].to(torch.bfloat16)
        tree = {"parent_np": parent, "parent": torch.from_numpy(parent).to(dev), "tokens": tl["draft_tokens"],
                "target": tl["target_logits"], "L": torch.full((w.B,), N, dtype=torch.int32, device=dev),
                "last": torch.empty((w.B,), dtype=torch.int32, device=dev),
                "ws": lr.Workspace(w.B, N, w.V, w.Hq, w.Hkv, w.d, S, device=dev)}
    conf = torch.empty((w.B, w.K), device=dev)
    dstat = torch.empty((w.B, w.K, 2), device=dev)
    L = torch.empty((w.B,), dtype=torch.int32, device=dev)
    n_acc = torch.empty((w.B,), dtype=torch.int32, device=dev)
    bonus = torch.empty((w.B,), dtype=torch.int32, device=dev)

    block_size = args.block_size if args.block_size > 0 else max(1, (2 * w.K) // 3)
    n_blocks = torch.empty((w.B,), dtype=torch.int32, device=dev)

    head = None
    if args.lm_head:
        head = workloads.lm_head(w, w.B * w.K, device=dev)
        head["ws"] = lr.LmHeadWorkspace(w.B * w.K, w.V, device=dev)
        head["tokens"] = inp["draft_tokens"].reshape(-1).contiguous()
        head["argmax"] = torch.empty((w.B * w.K,), dtype=torch.int32, device=dev)

    def seg_select():
        if head is not None:
            lr.libraspec_lm_head_stats(head["H"], head["W"], head["ws"], temperature=inp["temperature"],
                                       rows_per_seq=w.K, tokens=head["tokens"], row_stat=dstat.view(-1, 2),
                                       row_argmax=head["argmax"], token_prob=conf.view(-1))
        elif args.selector == "gain":  # confidence and Thm. 4's selection in one launch
            lr.libraspec_confidence_select(inp["draft_logits"], inp["draft_tokens"], inp["temperature"], cost, ws,
                                           conf=conf, dstat=dstat, L=L)
            return
        else:
            lr.libraspec_confidence(inp["draft_logits"], inp["draft_tokens"], inp["temperature"], ws, conf=conf,
                                    dstat=dstat)
        if args.selector == "alpha":
            lr.libraspec_select_alpha(conf, block_size, args.alpha, L=L, n_blocks=n_blocks)
        else:
            lr.libraspec_select_lengths(conf, cost, ws, L=L)

    def seg_attn():
        if N and P:
            lr.libraspec_verify_attn_tree_paged_layers(layers, tree["parent"], table, kv_t, tree["L"], tree["ws"])
        elif N:
            lr.libraspec_verify_attn_tree_layers(layers, tree["parent"], kv_t, tree["L"], tree["ws"])
        elif P:
            lr.libraspec_verify_attn_paged_layers(layers, table, kv_t, L, ws)
        else:
            lr.libraspec_verify_attn_layers(layers, kv_t, L, ws)

    def seg_accept():
        if N:
            lr.libraspec_accept_tree(tree["target"], tree["tokens"], tree["parent"], tree["L"], inp["temperature"],
                                     w.philox_seed, tree["ws"], seq_offset=seq_offset, n_accepted=n_acc,
                                     last_node=tree["last"], bonus_token=bonus)
            return
        lr.libraspec_accept(inp["target_logits"], inp["draft_logits"], inp["draft_tokens"], conf, dstat, L,
                            inp["temperature"], w.philox_seed, ws, seq_offset=seq_offset, n_accepted=n_acc,
                            bonus_token=bonus)

    # the plain chain round is the library's one-call round (the acceptance plan runs before the
    # attention layers); the variants chain their step calls
    one_call = not (N or P or head is not None or args.selector != "gain")
    outs = lr.RoundOutputs(conf, dstat, L, n_acc, bonus, Os, None) if one_call else None

    def seg_round():
        if one_call:
            lr.libraspec_verify_round(inp["draft_logits"], inp["draft_tokens"], inp["temperature"], cost,
                                      inp["target_logits"], layers, kv_t, w.philox_seed, ws, seq_offset=seq_offset,
                                      outputs=outs)
        else:
            seg_select()
            seg_attn()
            seg_accept()

    def device_status():
        st = lr.libraspec_get_status(ws) | (lr.libraspec_get_status(head["ws"]) if head is not None else 0)
        return st | (lr.libraspec_get_status(tree["ws"]) if N else 0)

    # eager warm-up (also configures kernels), then capture the graphs
    for _ in range(3):
        seg_round()
        seg_select(); seg_attn(); seg_accept()
    torch.cuda.synchronize()
    if device_status() != 0:
        raise RuntimeError("device status set during warm-up")
    side = torch.cuda.Stream(device=dev)
    round_graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(round_graph, stream=side):
        seg_round()
    graphs = []
    for seg in (seg_select, seg_attn, seg_accept):
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr, stream=side):
            seg()
        graphs.append(gr)
    stream = torch.cuda.current_stream()

    def step_split(ev_a, ev_b, ev_0, ev_c):
        ev_0.record(stream)
        graphs[0].replay()
        ev_a.record(stream)
        graphs[1].replay()
        ev_b.record(stream)
        graphs[2].replay()
        ev_c.record(stream)

    for _ in range(max(3, args.warmup)):
        round_graph.replay()
        for gr in graphs:
            gr.replay()
    torch.cuda.synchronize()
    if steps <= 0:  # enough for ~2 s of timed work
        t0 = time.perf_counter()
        for _ in range(20):
            round_graph.replay()
        torch.cuda.synchronize()
        per = (time.perf_counter() - t0) / 20
        steps = int(min(20000, max(50, 2.0 / max(per, 1e-6))))
    ev_0 = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ev_a = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ev_b = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ev_c = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    pdist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(physical_gpu(local_rank)) as clocks:
        start.record(stream)
        for _ in range(steps):
            round_graph.replay()
        end.record(stream)
        torch.cuda.synchronize()
        pdist.barrier()
        # second pass: the same rounds as three graphs, for the kernels' launch durations
        for i in range(steps):
            step_split(ev_a[i], ev_b[i], ev_0[i], ev_c[i])
        torch.cuda.synchronize()
    pdist.barrier()
    elapsed_ms = start.elapsed_time(end)
    attn_ms = sum(a.elapsed_time(b) for a, b in zip(ev_a, ev_b))
    select_ms = sum(a.elapsed_time(b) for a, b in zip(ev_0, ev_a))
    accept_ms = sum(a.elapsed_time(b) for a, b in zip(ev_b, ev_c))
    elapsed_max = pdist.max_over_ranks(elapsed_ms, device=dev)
    if device_status() != 0:
        raise RuntimeError("device status set during the timed steps")

    Lh = L.cpu().numpy()
    nh = n_acc.cpu().numpy()
    bh = bonus.cpu().numpy()
    temp = inp["temperature"].cpu().numpy()
    L_tree = np.full(w.B, N, np.int64) if N else None
    by = round_bytes(w, kv, Lh, temp, nh, logit_bytes=2 if args.logits == "bf16" else 4, L_tree=L_tree)
    us_per_round = elapsed_ms * 1000.0 / steps
    # one persistent attention launch runs up to ATTN_LAYERS_PER_LAUNCH layers
    attn_launches = -(-w.n_layers // ATTN_LAYERS_PER_LAUNCH)
    attn_launch_s = attn_ms / 1000.0 / (steps * attn_launches)
    attn_bytes_launch = by["attn_per_launch"] * w.n_layers / attn_launches
    peaks, peak_src = measured_peaks()
    hbm_peak = float(peaks["hbm_gbs"])
    tensor_peak = float(peaks.get("bf16_tflops_sustained") or peaks.get("bf16_tflops") or 1700.0)
    achieved = attn_bytes_launch / attn_launch_s / 1e9
    prof = None
    if not N and not P:
        prof = attn_profile_record(os.path.join(ROOT, "paper_2608_08721_gb300", "csrc", "attn.cu"), w.name)
    roof = {"kernel": "verify_attn", "bound": "hbm", "achieved": round(achieved, 1), "peak": hbm_peak,
            "unit": "GB/s", "frac": round(achieved / hbm_peak, 4),
            "traffic": None if prof is None else prof.get("traffic_bytes_per_launch"),
            "tensor_pipe_pct": None if prof is None else prof.get("tensor_pipe_pct"),
            "algorithmic_bytes_per_launch": attn_bytes_launch,
            "layers_per_launch": round(w.n_layers / attn_launches, 2),
            "launch_us": round(attn_launch_s * 1e6, 3),
            "peak_source": peak_src + " (MEASURED_PEAKS.json hbm_gbs)"}
    if N:
        # a tree's query rows share every key: bound by whichever roofline is slower
        fl = tree_flops(tree["parent_np"], kv, np.full(w.B, N), w.Hq, w.d) * w.n_layers / attn_launches
        roof["algorithmic_flops_per_launch"] = fl
        roof["kernel"] = "verify_attn (draft tree)"
        if fl / (tensor_peak * 1e12) > attn_bytes_launch / (hbm_peak * 1e9):
            tf = fl / attn_launch_s / 1e12
            roof.update({"bound": "tensor", "achieved": round(tf, 2), "peak": tensor_peak, "unit": "TFLOP/s",
                         "frac": round(tf / tensor_peak, 4),
                         "peak_source": peak_src + " (MEASURED_PEAKS.json bf16_tflops_sustained)"})

    # end to end through the public API with host buffers (the chain round on dense caches)
    e2e = None
    if args.e2e_steps > 0 and not N and not P:
        e2e = run_e2e(args, w, kv, inp, layers, cost, dev, seq_offset, steps=args.e2e_steps if primary else 5)
        if primary:
            e2e["host_link"] = host_link(e2e["h2d_bytes_per_step"], dev)
            best = max(e2e["host_link"]["single_copy_GBps"], e2e["host_link"]["three_streams_GBps"])
            e2e["host_link"]["copy_us_at_best_rate"] = round(e2e["h2d_bytes_per_step"] / best / 1e3, 1)

    host = None
    if rank == 0 and world == 1 and (not args.no_cpu_baseline or not (N or head is not None)):
        # bf16 logits widen exactly to f32 for the oracle
        host = {k: (v.float() if v.dtype == torch.bfloat16 else v).cpu().numpy() for k, v in inp.items()}
        host["cost_table"] = workloads.cost_table(w, kv)

    flags = None
    if host is not None and not N and head is None and args.selector == "gain":
        flags = oracle_flags(w, host, Lh, nh, bh)

    cpu = None
    if primary and host is not None and not args.no_cpu_baseline:
        import oracle

        conf_fn = attn_fn = None
        if P:
            table_np = table.cpu().numpy()
            lay_host = [{"Q": layers[0]["Q"].cpu(), "Kp": layers[0]["Kp"].cpu(), "Vp": layers[0]["Vp"].cpu()}]

            def attn_fn(lay, L):  # the oracle on the cache the pages describe (gather included)
                oracle.verify_attn_paged(lay["Q"], lay["Kp"], lay["Vp"], table_np, kv, L)
        else:
            lay_host = [{"Q": layers[0]["Q"].cpu(), "Kc": layers[0]["Kc"].cpu(), "Vc": layers[0]["Vc"].cpu()}]
        if head is not None:
            H_host, W_host = head["H"].cpu(), head["W"].cpu()
            tok_host = head["tokens"].cpu().numpy()

            def conf_fn():  # the head's statistics over the full vocabulary, in binary64
                return oracle.lm_head_stats(H_host, W_host, host["temperature"], w.K, tok_host)[3].reshape(w.B, w.K)
        if N:
            th = {"target_logits": tree["target"].float().cpu().numpy(), "draft_tokens": tree["tokens"].cpu().numpy(),
                  "parent": tree["parent_np"], "L": np.full(w.B, N, np.int32)}
            lay0 = lay_host[0]
            if P:
                S_all = int(table_np.shape[1] * P)
                lay0 = {"Q": lay0["Q"], "Kc": oracle.gather_pages(lay0["Kp"], table_np, S_all),
                        "Vc": oracle.gather_pages(lay0["Vp"], table_np, S_all)}
            us, cores, sample = oracle_tree_round_time(w, host, th, lay0, kv, args.cpu_seconds)
            cpu = {"value": round(us, 1), "unit": "us", "cores": cores, "kind": "oracle", "sample": sample}
        else:
            variant = "".join([
                "; the confidence from the hidden states and the LM head" if head is not None else "",
                "; attention on the cache gathered from its pages" if P else ""])
            us, cores, sample = oracle_round_time(w, host, lay_host, kv, args.cpu_seconds * 0.6, conf_fn=conf_fn,
                                                  attn_fn=attn_fn, variant=variant)
            cpu = {"value": round(us, 1), "unit": "us", "cores": cores, "kind": "oracle", "sample": sample}
            if conf_fn is None and attn_fn is None:
                # single-threaded, on a subset of the batch (about 1/16 of its sequences), scaled
                us1, _, sample1 = oracle_round_time(w, host, lay_host, kv, args.cpu_seconds * 0.4, threads=1,
                                                    seqs=max(1, w.B // 16))
                cpu["single_thread"] = {"value": round(us1, 1), "unit": "us", "cores": 1, "sample": sample1}

    lm = None
    if head is not None:
        # the conf+select graph is the head's GEMM plus a selection of a few microseconds
        head_bytes = (w.V + w.B * w.K) * w.hidden * 2
        lm_s = select_ms / 1000.0 / steps
        lm = {"kernel": "lm_head_stats (tcgen05 GEMM, statistics in the epilogue)", "us": round(lm_s * 1e6, 3),
              "bytes": head_bytes, "GBps": round(head_bytes / lm_s / 1e9, 1),
              "frac_of_measured_hbm": round(head_bytes / lm_s / 1e9 / hbm_peak, 4),
              "note": "time of the confidence+selection graph; the head's weights dominate its bytes"}
    # the logits-bound segments: confidence (+ selection) over B*K drafter rows, acceptance over the
    # verified target rows (+ residual rows); their graph times include the small launches beside them
    logits = None
    if head is None:
        logits = {}
        for name, nbytes, ms in (("conf_select", by["conf"] + by["select"], select_ms),
                                 ("accept", by["accept"], accept_ms)):
            sec = ms / 1000.0 / steps
            logits[name] = {"us": round(sec * 1e6, 3), "bytes": int(nbytes), "GBps": round(nbytes / sec / 1e9, 1),
                            "frac_of_measured_hbm": round(nbytes / sec / 1e9 / hbm_peak, 4)}
    # kernels launched per round: confidence + selection (one fused launch for the Thm. 4 selector, the LM
    # head's GEMM + merge + selection, or confidence + selection), the attention launches (+ the tree-mask
    # kernel per launch), and the acceptance: plan + rows + draws (the tree: statistics + walk)
    conf_launches = 3 if args.lm_head else (1 if args.selector == "gain" else 2)
    accept_launches = 2 if N else 3
    launches_per_round = attn_launches * (2 if N else 1) + conf_launches + accept_launches
    return {
        "w": w, "steps": steps, "elapsed_max_ms": elapsed_max, "us_per_round": us_per_round, "by": by,
        "Lh": Lh, "kv": kv, "n_res": n_res, "block_size": block_size, "hbm_peak": hbm_peak,
        "roofline": roof, "lm_head": lm, "logits_segments": logits,
        "segments_us": {"conf_select": round(select_ms * 1000.0 / steps, 3),
                        "attention": round(attn_ms * 1000.0 / steps, 3),
                        "accept": round(accept_ms * 1000.0 / steps, 3)},
        "clocks": clocks.summary(), "launches": launches_per_round * steps, "e2e": e2e, "cpu": cpu, "flags": flags,
        "one_call": one_call,
    }


def run_ours(args, rank, world, local_rank):
    import torch

    from paper_2608_08721_gb300 import binding as lr
    from paper_2608_08721_gb300 import build as cuda_build
    from paper_2608_08721_gb300 import dist as pdist
    from paper_2608_08721_gb300 import workloads

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    if rank == 0 or not os.path.exists(lr.LIB_PATH):
        cuda_build.build()
    pdist.barrier()
    w = workloads.WORKLOADS[args.config]
    m = measure_workload(args, w, dev, rank, world, local_rank, args.steps, primary=True)
    also = {}
    variant = args.tree or args.page_size or args.lm_head or args.selector != "gain" or args.logits != "f32"
    if not variant:
        for name in [x for x in args.also.split(",") if x and x != args.config]:
            torch.cuda.empty_cache()
            a = measure_workload(args, workloads.WORKLOADS[name], dev, rank, world, local_rank, args.also_steps,
                                 primary=False)
            also[name] = {
                "value_us": round(a["elapsed_max_ms"] * 1000.0 / (a["steps"] * world), 3), "steps": a["steps"],
                "config": {"B": a["w"].B, "K": a["w"].K, "V": a["w"].V, "layers": a["w"].n_layers,
                           "gqa": "%d/%d" % (a["w"].Hq, a["w"].Hkv), "kv_len": [int(a["kv"].min()), int(a["kv"].max())],
                           "selected_L": [int(a["Lh"].min()), int(a["Lh"].max())]},
                "hbm_tbs": round(a["by"]["total"] / (a["us_per_round"] * 1e-6) / 1e12, 3),
                "roofline": a["roofline"], "logits_segments": a["logits_segments"],
                "segments_us": a["segments_us"], "flags": a["flags"], "e2e": a["e2e"],
                "gpu_launches": a["launches"]}
    if rank != 0:
        return
    w, by, Lh, kv, K_steps = m["w"], m["by"], m["Lh"], m["kv"], m["steps"]
    clk = m["clocks"]
    us_per_round = m["us_per_round"]
    value = m["elapsed_max_ms"] * 1000.0 / (K_steps * world)
    line = {
        "metric": METRIC, "value": round(value, 3), "unit": "us", "n_gpus": world, "steps": K_steps,
        "warmup": max(3, args.warmup), "ms_per_step": round(m["elapsed_max_ms"] / K_steps, 6),
        "higher_is_better": False, "scaling": "weak", "vs_baseline": None, "dtype": "bf16+f32",
        "data": "synthetic (seeded; shapes of the paper's 8B-70B-class targets, random values)",
        "config": workload_config(args, w, kv, Lh, world, m["block_size"]),
        "timing": ("value: K rounds, each one CUDA graph replay of %s, events around the loop; "
                   "segments and roofline: a second pass of the same K rounds as three graphs "
                   "(conf+select | attention layers | accept, the acceptance plan included) with "
                   "events between" % ("libraspec_verify_round" if m["one_call"] else "the round's step calls")),
        "l2_bytes_per_step": int(by["total"]),
        "hbm_tbs": round(by["total"] / (us_per_round * 1e-6) / 1e12, 3),
        "hbm_frac_of_measured": round(by["total"] / (us_per_round * 1e-6) / 1e9 / m["hbm_peak"], 4),
        "hbm_frac_of_nominal_8tbs": round(by["total"] / (us_per_round * 1e-6) / 1e9 / NOMINAL_HBM_GBS, 4),
        "roofline": m["roofline"],
        "lm_head": m["lm_head"],
        "logits_segments": m["logits_segments"],
        "segments_us": m["segments_us"],
        "flags": m["flags"],
        "clocks": {"sm_mhz": clk["sm_mhz"], "sm_max_mhz": clk["sm_max_mhz"], "reasons": clk["reasons"],
                   "samples": clk["samples"]},
        "gpu_launches": m["launches"],
        "e2e": m["e2e"],
        "cpu_baseline": m["cpu"],
        "also": also or None,
    }
    print(json.dumps(line), flush=True)


def run_e2e(args, w, kv, inp, layers, cost, dev, seq_offset, steps):
    """Same metric through the public host-buffer API: per round, the round's
    inputs (one pinned buffer) are copied in, the block's keys and values
    appended to the caches, and the results read back."""
    import torch

    from paper_2608_08721_gb300.api import VerifyRound

    caches = [{"Kc": l["Kc"], "Vc": l["Vc"]} for l in layers]
    runner = VerifyRound(w.B, w.K, w.V, w.Hq, w.Hkv, w.d, layers[0]["Kc"].shape[2], caches, torch.tensor(kv),
                         device=dev, logits_dtype=inp["draft_logits"].dtype)
    K1 = w.K + 1
    h = runner.host_inputs()
    for name in ("draft_logits", "target_logits", "draft_tokens", "temperature"):
        h[name].copy_(inp[name].cpu())
    h["cost_table"].copy_(cost.cpu())
    for l, lay in enumerate(layers):
        h["Q"][l].copy_(lay["Q"].cpu())
        # the block rows the caches already hold, so that appending them changes nothing
        h["kv_new"][l, 0].copy_(torch.stack([lay["Kc"][b, :, int(kv[b]):int(kv[b]) + K1] for b in range(w.B)]).cpu())
        h["kv_new"][l, 1].copy_(torch.stack([lay["Vc"][b, :, int(kv[b]):int(kv[b]) + K1] for b in range(w.B)]).cpu())
    for _ in range(3):
        runner.run_staged(w.philox_seed, seq_offset=seq_offset)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(steps):
        n_acc, _ = runner.run_staged(w.philox_seed, seq_offset=seq_offset)
    dt = time.perf_counter() - t0
    L = runner.out.L.cpu().numpy()
    return {"value": round(dt * 1e6 / steps, 3), "unit": "us",
            "h2d_bytes_per_step": runner.h2d_bytes(L, n_acc, inp["temperature"].cpu().numpy()),
            "d2h_bytes_per_step": runner.d2h_bytes(), "steps": steps,
            "inputs": ("read in place from pinned host memory by the kernels (the queries copied); the bytes "
                       "counted are those the round reads over the host link" if runner.in_place else
                       "the pinned buffer copied to the device in three parts"),
            "pinned_input_buffer_bytes": runner._host_stage.numel(),
            "api": "paper_2608_08721_gb300.api.VerifyRound.run_staged (libraspec_verify_round_staged: the "
                   "block's keys and values appended, then the round; the results read back)"}


def main():
    args = parse()
    from paper_2608_08721_gb300 import dist as pdist

    rank, world, local_rank = pdist.env_world()
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    pdist.init("nccl" if world > 1 else "gloo")
    try:
        run_ours(args, rank, world, local_rank)
    finally:
        import torch.distributed as dist

        if dist.is_initialized():
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
