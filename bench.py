"""Benchmark of the UltraMem layer forward on GB300.

One step = one forward (S1-S9) of one decode batch of the named workload,
inputs already resident in HBM.  Default: the decode-shaped layer (1024x1024
physical grid, E=4, 2 heads, top-32, 64 tokens).  The L2 is flushed (256 MiB
write) between timed steps, outside the timed events.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME --batch B]
  python bench.py --impl reference ...      # the CPU oracle as the reference arm

Prints one JSON line on rank 0.  Under torchrun each rank runs its own
replica of the layer on its own token batches (no collective on the data
path); the step time is the max over ranks and ``value`` counts all ranks'
tokens.
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

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "UltraMem layer tokens/s at decode batch; gather HBM GB/s as % of GB300 peak"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=None)
    ap.add_argument("--batch", type=int, default=None)
    ap.add_argument("--cores", type=int, default=0,
                    help="component cores per head (Multi-Core Scoring); 0 = one core")
    ap.add_argument("--conv-k", type=int, default=0,
                    help="taps of the causal query convolution; each step continues B/L "
                         "sequences by L tokens, the conv state carried from step to step")
    ap.add_argument("--seq-len", type=int, default=1,
                    help="L, tokens per sequence per step with a query convolution")
    ap.add_argument("--query-ln", action="store_true", help="LayerNorm of each head's query")
    ap.add_argument("--pkm", action="store_true",
                    help="the layer as a product-key memory: rank 1, additive grid scores, "
                         "softmax weights")
    ap.add_argument("--backward", action="store_true",
                    help="also time the lookup-reduce backward (dV, dw, dW_p) on the "
                         "batch's slots")
    ap.add_argument("--recall", action="store_true",
                    help="also measure the two-phase search's recall@m against the "
                         "brute-force grid top-m, and the brute force's time")
    ap.add_argument("--no-graph", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--no-sweep", action="store_true",
                    help="skip the further workloads (mid_4m, large_20m, prefill_16k)")
    return ap.parse_args()


def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)),
            int(os.environ.get("LOCAL_RANK", 0)))


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def algorithmic_bytes(cfg, B, lists=False):
    """Bytes each stage must move at least (paper's Sec. 4 memory-access model
    with heads: the gather reads min(B*H*m, N) rows of D_v).  The selection
    reads, per (token, head), the rank-1 score keys of both axes (2 K x 4 B),
    the query (A D_k x 4 B) and the key rows of the 2k survivors
    (2 k D_k x es), and writes m slots (row, block and h weights: 8 + 4h B,
    h = 1 without Multi-Core Scoring).  With the scoring's candidate lists
    (`lists`) it reads, in place of the keys, each axis' group counts
    (ceil(K/16) x 4 B) and at least k list entries (8 B each)."""
    es = 4 if int(cfg["dtype"]) == 0 else 2
    H, dk, din = cfg["heads"], cfg["d_k"], cfg["d_in"]
    K = int(round(cfg["expand_e"] ** 0.5)) * cfg["n"]
    A = 1 if cfg["share_query"] else 2
    N = cfg["n"] ** 2
    k, m = cfg["topk"], cfg["topm"]
    rows = min(B * H * m, N)
    axis_in = 2 * ((K + 15) // 16 * 4 + k * 8) if lists else 2 * K * 4
    return {
        "query": A * H * dk * din * es + B * din * es,
        "score": 2 * H * K * dk * es,
        "select": B * H * (axis_in + A * dk * 4 + 2 * k * dk * es
                           + m * (8 + 4 * max(1, int(cfg.get("cores", 0))))),
        "gather": rows * cfg["d_v"] * es,
        "project": (cfg["expand_e"] * cfg["d_v"] * cfg["d_out"] * es if cfg["has_proj"] else 0)
        + B * cfg["d_out"] * es,
    }


def aggregate_step(ms, batch, dist=None, device="cpu"):
    """The slowest rank's step time and the whole-job tokens/s (every rank
    processes its own batch of `batch` tokens)."""
    world = 1
    if dist is not None and dist.is_available() and dist.is_initialized():
        import torch
        world = dist.get_world_size()
        t = torch.tensor([ms], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
    return ms, world * batch / (ms / 1e3)


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons during timing."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index, enabled=True):
        self.proc = None
        self.path = None
        self.gpu = gpu_index
        if not enabled:
            return
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(gpu_index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if not self.proc:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, fl in rows for i, f in enumerate(fl)
                          if f.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows),
                "sm_max_mhz": max(r[1] for r in rows), "reasons": reasons,
                "samples": len(rows)}


def source_sha(path):
    return hashlib.sha256(open(path, "rb").read()).hexdigest()[:16]


def ncu_traffic(kernel_stage, workload, batch):
    """DRAM bytes per launch of a stage's kernel from the committed ncu
    summary, or None if absent or taken on another version of the kernel."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    try:
        d = json.load(open(path))
        e = d[kernel_stage]
        src = os.path.join(ROOT, "paper_2411_12364_gb300", "csrc", e["source"])
        if e["workload"] != workload or int(e["batch"]) != batch:
            return None
        if e["source_sha"] != source_sha(src):
            return None
        return float(e["dram_bytes_per_launch"])
    except Exception:
        return None


def cpu_baseline(cfg, weights_np, B, budget_s=12.0):
    """The oracle, as it stands, on the host cores: whole batches of the
    workload until about budget_s seconds of wall time have passed."""
    import numpy as np
    import oracle
    from paper_2411_12364_gb300 import workloads
    cores = len(os.sched_getaffinity(0))
    done, t0, batches = 0, time.perf_counter(), 0
    while True:
        x = workloads.stored_numpy(workloads.make_tokens(cfg, B, 1000 + batches))
        t = dict(weights_np, x=x)
        oracle.forward(cfg, t, B, threads=cores)
        done += B
        batches += 1
        el = time.perf_counter() - t0
        if el >= budget_s:
            break
    return {"value": done / el, "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"{batches} batch(es) of {B} tokens of the same workload, "
                      f"{el:.1f} s wall, fp64, OpenMP over tokens"}


def numpy_weights(w):
    from paper_2411_12364_gb300 import workloads
    return {k: workloads.stored_numpy(v) for k, v in w.items()}


def run_reference(args, cfg, B, wl):
    """The reference arm: the CPU oracle timed on the host cores."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    import torch
    from paper_2411_12364_gb300 import workloads
    w = workloads.make_weights(cfg, device="cpu")
    wn = numpy_weights(w)
    import oracle
    cores = len(os.sched_getaffinity(0))
    sample = B              # tokens per step: the whole batch of the workload
    for i in range(args.warmup):
        x = workloads.stored_numpy(workloads.make_tokens(cfg, sample, 2000 + i))
        oracle.forward(cfg, dict(wn, x=x), sample, threads=cores)
    times = []
    for i in range(args.steps):
        x = workloads.stored_numpy(workloads.make_tokens(cfg, sample, 3000 + i))
        t0 = time.perf_counter()
        oracle.forward(cfg, dict(wn, x=x), sample, threads=cores)
        times.append(time.perf_counter() - t0)
        if sum(times) > 120:
            break
    k = len(times)
    ms = 1e3 * sum(times) / k
    value = sample / (ms / 1e3)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
            "n_gpus": args.gpus, "steps": k, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": dict(workload=wl, batch=B, **_cfg_brief(cfg)),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores,
                             "kind": "oracle",
                             "sample": f"the whole batch ({sample} tokens) of the workload "
                                       f"per step, fp64, OpenMP over tokens"},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def measure_backward(layer, x, cfg, stream, K, flush):
    """Device time of the lookup-reduce backward (dV accumulated, dw, dW_p)
    on one batch's slots, K timed calls with the L2 flushed between them,
    and the same without dW_p (whose forward re-gather and token-reduction
    contraction are the training-only extra)."""
    import torch
    B = x.shape[0]
    with torch.cuda.stream(stream):
        _, idx, w = layer.forward(x, with_slots=True)
        g = torch.randn((B, cfg["d_out"]), device="cuda").to(layer.dtype)
        dv, _, _ = layer.lookup_reduce_backward(idx, w, g)

        def timed(want_dwp):
            ts = []
            for i in range(K):
                flush.fill_(float(i))
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(stream)
                layer.lookup_reduce_backward(idx, w, g, dvalues=dv, want_dw_proj=want_dwp)
                b.record(stream)
                ts.append((a, b))
            torch.cuda.synchronize()
            return sum(a.elapsed_time(b) for a, b in ts) / K
        full = timed(True)
        rows_only = timed(False)
    es = 4 if int(cfg["dtype"]) == 0 else 2
    slots = B * cfg["heads"] * cfg["topm"]
    # the rows kernel: value rows read (D_v es), dV rows read and written (fp32)
    rows_bytes = slots * cfg["d_v"] * (es + 8)
    return {"ms": full, "ms_without_dw_proj": rows_only, "slots": slots,
            "rows_bytes": rows_bytes, "launches": layer.last_launches()}


def measure_recall(layer, x, cfg, stream):
    """recall@m of the forward's two-phase search (Eq. 6-10) against the
    brute-force top-m of each head's whole grid (Eq. 5), over one batch,
    and the device time of the brute force."""
    import torch
    with torch.cuda.stream(stream):
        _, a_idx, _ = layer.forward(x, with_slots=True)
        layer.retrieve_exact(x)   # warm-up
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
        ev[0].record(stream)
        e_idx, _ = layer.retrieve_exact(x)
        ev[1].record(stream)
    torch.cuda.synchronize()
    a, e = a_idx.cpu().numpy(), e_idx.cpu().numpy()
    B, H, m = a.shape
    hits = sum(len(set(a[b, h].tolist()) & set(e[b, h].tolist()))
               for b in range(B) for h in range(H))
    return {"recall_at_m": hits / (B * H * m), "heads": B * H, "m": m,
            "exact_ms": ev[0].elapsed_time(ev[1])}


def _cfg_brief(cfg):
    keys = ("d_in", "d_k", "heads", "rank", "n", "expand_e", "d_v", "d_out", "topk", "topm")
    d = {k: int(cfg[k]) for k in keys}
    d["storage"] = "f32" if int(cfg["dtype"]) == 0 else "bf16"
    if int(cfg.get("cores", 0)) > 1:
        d["mcs_cores"] = int(cfg["cores"])
    if int(cfg.get("conv_k", 0)) > 0:
        d["conv_k"] = int(cfg["conv_k"])
        d["seq_len_per_step"] = int(cfg.get("seq_len_per_step", 1))
    if int(cfg.get("query_ln", 0)):
        d["query_ln"] = 1
    if int(cfg.get("score_mode", 0)) == 1:
        d["score"] = "product keys (Eq. 2-3)"
    return d


def stage_profile(layer, fwd, stream, flush, K, use_graph, NB):
    """Device time of each stage (kernels of the stage: first CTA past its
    dependency wait to last warp done, from the kernels' own global-timer
    stamps) and the hand-off before it, averaged over K forwards replayed
    exactly as the timed ones (graphs, programmatic dependent launches, L2
    flushed between forwards)."""
    import torch
    layer.profile(True)
    graphs = []
    with torch.cuda.stream(stream):
        fwd(0)
        torch.cuda.synchronize()
        for i in range(NB if use_graph else 0):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                fwd(i)
            graphs.append(g)
    torch.cuda.synchronize()
    times, gaps = {}, {}
    with torch.cuda.stream(stream):
        for i in range(K):
            flush.fill_(float(i))
            if use_graph:
                graphs[i % NB].replay()
            else:
                fwd(i)
            torch.cuda.synchronize()
            t, g = layer.profile_read(gaps=True)
            for k, v in t.items():
                times.setdefault(k, []).append(v)
            for k, v in g.items():
                gaps.setdefault(k, []).append(v)
    torch.cuda.synchronize()
    layer.profile(False)
    del graphs
    avg = lambda d: {k: sum(v) / len(v) for k, v in d.items() if min(v) >= 0}
    return avg(times), avg(gaps)


def cold_gather(layer, x, stream, flush, K):
    """The gather kernel's device time with its value rows in HBM: the
    forward's slots, pooled through ultramem_lookup_reduce (no selection
    before it, so no row was prefetched into L2) after an L2 flush."""
    import torch
    with torch.cuda.stream(stream):
        idx, w = layer.retrieve(x)
        layer.lookup_reduce(idx, w)
        torch.cuda.synchronize()
        layer.profile(True)
        ts = []
        for i in range(K):
            flush.fill_(float(i))
            layer.lookup_reduce(idx, w)
            torch.cuda.synchronize()
            ts.append(layer.profile_read()["gather"])
        layer.profile(False)
    return sum(ts) / len(ts)


def roofline_of(stages, alg, peak, peak_kind):
    dominant = max(stages, key=stages.get)
    ach = alg[dominant] / (stages[dominant] * 1e6)
    return {"kernel": dominant, "bound": "hbm", "achieved": ach, "peak": peak, "unit": "GB/s",
            "frac": ach / peak, "peak_kind": peak_kind, "algorithmic_bytes": alg[dominant],
            "avg_ms": stages[dominant],
            "time_source": "kernel global-timer stamps in the replayed forward graph"}


def gather_entry(alg, gms, cold_ms, peak):
    """Gather GB/s: in the forward (its rows were prefetched into L2 by the
    selection) and cold (rows from HBM after an L2 flush)."""
    out = {"bytes": alg["gather"]}
    if gms:
        gbs = alg["gather"] / (gms * 1e6)
        out.update(ms=gms, achieved_gbs=gbs, frac_of_measured=gbs / peak,
                   frac_of_nominal_8tbs=gbs / NOMINAL_HBM_GBS)
    if cold_ms:
        cg = alg["gather"] / (cold_ms * 1e6)
        out.update(cold_ms=cold_ms, cold_gbs=cg, cold_frac_of_measured=cg / peak,
                   cold_frac_of_nominal_8tbs=cg / NOMINAL_HBM_GBS)
    return out


def time_steps(step, stream, flush, K, dist=None):
    """K timed steps (CUDA events on the stream, an L2 flush after each,
    outside the events); returns the mean ms per step."""
    import torch
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(K)]
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        for i in range(K):
            ev[i][0].record(stream)
            step(i)
            ev[i][1].record(stream)
            flush.fill_(float(i))
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    return sum(a.elapsed_time(b) for a, b in ev) / K


def build_layer(cfg, B, rank, NB):
    import torch
    from paper_2411_12364_gb300 import workloads
    from paper_2411_12364_gb300.binding import UltraMemLayer
    w = workloads.make_weights(cfg, device="cuda")
    layer = UltraMemLayer(cfg, w, B)
    xs = [workloads.make_tokens(cfg, B, 100 * rank + i, device="cuda") for i in range(NB)]
    return w, layer, xs


def capture(layer, fwd, stream, NB):
    import torch
    graphs = []
    with torch.cuda.stream(stream):
        for _ in range(3):
            fwd(0)
        torch.cuda.synchronize()
        for i in range(NB):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                fwd(i)
            graphs.append(g)
    torch.cuda.synchronize()
    return graphs


SWEEP = [("mid_4m", (128,)), ("large_20m", (64, 256)), ("prefill_16k", (16384,))]


def uses_lists(layer, fwd):
    """Whether the layer's default scoring form takes the candidate lists at
    this batch: two more launches than every key."""
    import torch
    layer.candidates(0)
    fwd(0)
    n0 = layer.last_launches()
    layer.candidates(2)
    fwd(0)
    torch.cuda.synchronize()
    return layer.last_launches() == n0 + 2


def sweep_workload(wl, batches, K, flush, stream, peak, peak_kind):
    """Further batches of one workload (one table): step time, tokens/s,
    per-stage device times, the gather's GB/s and the dominant kernel's
    roofline, measured like the headline line (graph replays, L2 flushed
    between steps)."""
    import torch
    from paper_2411_12364_gb300 import workloads
    cfg = workloads.layer_config(wl)
    NB = 2
    w, layer, xs_all = build_layer(cfg, max(batches), 0, NB)
    res = []
    for B in batches:
        xs = [x[:B].contiguous() for x in xs_all]
        out = torch.empty((B, cfg["d_out"]), dtype=layer.dtype, device="cuda")
        fwd = lambda i: layer.forward(xs[i % NB], out=out)
        lists = uses_lists(layer, fwd)
        graphs = capture(layer, fwd, stream, NB)
        big = B >= 4096
        steps, warm = (5, 2) if big else (max(5, min(K, 30)), 3)
        with torch.cuda.stream(stream):
            for i in range(warm):
                graphs[i % NB].replay()
                flush.fill_(float(i))
        ms = time_steps(lambda i: graphs[i % NB].replay(), stream, flush, steps)
        del graphs
        stages, gaps = stage_profile(layer, fwd, stream, flush, 3 if big else 20, True, NB)
        cold = cold_gather(layer, xs[0], stream, flush, 3 if big else 10)
        alg = algorithmic_bytes(cfg, B, lists)
        res.append({"workload": wl, "batch": B, "steps": steps, "ms_per_step": ms,
                    "scoring": "candidate_lists" if lists else "every_key",
                    "tokens_per_s": B / (ms / 1e3), "stages_ms": stages, "handoff_ms": gaps,
                    "roofline": roofline_of(stages, alg, peak, peak_kind),
                    "gather": gather_entry(alg, stages.get("gather"), cold, peak),
                    "step_hbm_gbs": sum(alg.values()) / (ms * 1e6)})
        del xs, out
    layer.close()
    del layer, w, xs_all
    torch.cuda.empty_cache()
    return res


def main():
    args = parse()
    from paper_2411_12364_gb300 import workloads
    wl = args.workload or workloads.HEADLINE[0]
    B = args.batch or (workloads.HEADLINE[1] if wl == workloads.HEADLINE[0]
                       else workloads.CONFIGS[wl]["batches"][-1])
    over = {"cores": args.cores} if args.cores > 1 else {}
    if args.conv_k > 0:
        over["conv_k"] = args.conv_k
    if args.query_ln:
        over.update(query_ln=1, ln_eps=1e-5)
    if args.conv_k > 0:
        over["seq_len_per_step"] = args.seq_len
    if args.pkm:
        over.update(rank=1, score_mode=1, act=1)
    cfg = workloads.layer_config(wl, **over)
    if args.impl == "reference":
        return run_reference(args, cfg, B, wl)

    import torch
    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")

    NB = 8     # distinct token batches cycled through (per rank)
    w, layer, xs = build_layer(cfg, B, rank, NB)
    out = torch.empty((B, cfg["d_out"]), dtype=layer.dtype, device="cuda")
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device="cuda")
    kc = int(cfg.get("conv_k", 0))
    # with a query convolution every step continues B/L sequences by L tokens
    # (L = 1: a decode step); batch i reads state i % 2 and writes the other
    n_seq = B // max(1, args.seq_len)
    states = [workloads.make_conv_state(cfg, n_seq, 0, device="cuda") for _ in range(2)] \
        if kc > 1 else None

    def fwd(i):
        if states is None:
            layer.forward(xs[i % NB], out=out)
        else:
            layer.forward_seq(xs[i % NB], n_seq, states[i % 2], states[(i + 1) % 2], out=out)

    stream = torch.cuda.Stream()
    use_graph = not args.no_graph
    with torch.cuda.stream(stream):
        for i in range(3):
            fwd(0)
        torch.cuda.synchronize()
    lists = uses_lists(layer, fwd)
    with torch.cuda.stream(stream):
        fwd(0)
        torch.cuda.synchronize()
    launches = layer.last_launches()   # kernels per forward (and per graph replay)
    graphs = capture(layer, fwd, stream, NB) if use_graph else []

    def step(i):
        if use_graph:
            graphs[i % NB].replay()
        else:
            fwd(i)

    with torch.cuda.stream(stream):
        for i in range(args.warmup):
            step(i)
            flush.fill_(float(i))
    torch.cuda.synchronize()

    # ---- timed region ----------------------------------------------------
    K = args.steps
    clocks = Clocks(local, enabled=not args.no_clocks)
    time.sleep(0.3)
    step_ms = time_steps(step, stream, flush, K, dist)
    clk = clocks.stop()
    ms, value = aggregate_step(step_ms, B, dist, device="cuda")
    del graphs

    # ---- per-stage device times from the kernels' own stamps -------------
    stages, gaps = stage_profile(layer, fwd, stream, flush, min(K, 50), use_graph, NB)
    cold = cold_gather(layer, xs[0], stream, flush, 10) if states is None else None
    alg = algorithmic_bytes(cfg, B, lists)
    peak, peak_kind = peaks()
    roof = roofline_of(stages, alg, peak, peak_kind)
    roof["traffic"] = None if int(cfg.get("cores", 0)) > 1 else \
        ncu_traffic(roof["kernel"], wl, B)
    gather = gather_entry(alg, stages.get("gather"), cold, peak)
    gather["traffic"] = ncu_traffic("gather", wl, B)

    # ---- end to end through the public API with host buffers -------------
    xh = [x.cpu().pin_memory() for x in xs]
    oh = torch.empty((B, cfg["d_out"]), dtype=layer.dtype).pin_memory()
    with torch.cuda.stream(stream):
        for i in range(3):
            layer.forward_host(xh[i % NB], oh)
        e2e_t = []
        for i in range(K):
            t0 = time.perf_counter()
            layer.forward_host(xh[i % NB], oh)
            e2e_t.append(time.perf_counter() - t0)
    e2e_ms, e2e_value = aggregate_step(1e3 * sum(e2e_t) / len(e2e_t), B, dist, device="cuda")
    es = 4 if int(cfg["dtype"]) == 0 else 2
    e2e = {"value": e2e_value, "unit": "tokens/s",
           "h2d_bytes_per_step": B * cfg["d_in"] * es, "d2h_bytes_per_step": B * cfg["d_out"] * es,
           "ms_per_step": e2e_ms}

    recall = None
    if args.recall and rank == 0:
        recall = measure_recall(layer, xs[0], cfg, stream)
    backward = None
    if args.backward and rank == 0:
        backward = measure_backward(layer, xs[0], cfg, stream, K, flush)

    wn = numpy_weights(w) if rank == 0 and world == 1 and not args.no_cpu_baseline else None
    sweep = None
    if world == 1 and not args.no_sweep and args.workload is None and not over:
        layer.close()
        del layer, w, xs, xh, out
        torch.cuda.empty_cache()
        sweep = [r for swl, bs in SWEEP
                 for r in sweep_workload(swl, bs, K, flush, stream, peak, peak_kind)]
    cpu = cpu_baseline(cfg, wn, B) if wn is not None else None

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
                "steps": K, "warmup": args.warmup, "ms_per_step": ms,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": "bf16" if int(cfg["dtype"]) else "f32", "data": "synthetic",
                "config": dict(workload=wl, batch=B, **_cfg_brief(cfg), accumulate="f32",
                               scoring="candidate_lists" if lists else "every_key",
                               l2="flushed between steps (256 MiB write, outside timing)",
                               cuda_graph=use_graph, parallelism=f"replicas x{world}"),
                "roofline": roof, "gather": gather, "stages_ms": stages, "handoff_ms": gaps,
                "step_hbm_gbs": sum(alg.values()) / (ms * 1e6),
                "gpu_launches": K * launches, "e2e": e2e,
                "cpu_baseline": cpu, "clocks": clk}
        if sweep is not None:
            line["sweep"] = sweep
        if recall is not None:
            line["recall"] = recall
        if backward is not None:
            line["backward"] = backward
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
