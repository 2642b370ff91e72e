#!/usr/bin/env python3
"""Throughput of SEED's draft/verify hot path on GB300.

One step = one decode round of Alg. 2 over one batch of the chosen synthetic
workload: k draft steps (each: draft-row append + draft attention in the 2
decoder layers), the verify pass (each of the 28 layers: append of the k+1 new
rows + verify attention), then greedy accept/commit.  Every call goes through
the C ABI (libseed.so); each phase of a round is replayed from a CUDA graph.

Metric: achieved HBM GB/s = algorithmic bytes of the round (every visible K/V
row read once per attention call, queries, outputs, appended rows) / device
time of the round.  Inputs are resident in HBM; a round's working set
(gigabytes of KV) is far larger than the 129 MB L2.

    python bench.py [--workload 3] [--steps 10] [--warmup 3] [--impl seed|reference]
"""

from __future__ import annotations

import argparse
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

from workloads import WORKLOADS, gen  # noqa: E402

METRIC = "draft+verify attention achieved HBM GB/s (% of GB300 peak); draft/verify step µs"
UNIT = "GB/s"


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


# ------------------------------------------------------------------ accounting
def round_bytes(wl, lens: np.ndarray, k_b: np.ndarray, n_layers: int) -> dict:
    """Algorithmic bytes of one round.  R = K+V bytes of one token in one layer.
    draft call (b, step i): (L_b + i) rows + q (bf16) + o (f32) + lse (f32)
    draft append (b):       one new row read + written
    verify call (b):        (L_b + n_b) rows + n_b*(q + o + lse), n_b = k_b + 1
    verify append (b):      n_b new rows read + written
    accept:                 ids, lengths and slots (int32)."""
    R = wl.row_bytes
    qo = wl.hq * wl.head_dim * (2 + 4) + wl.hq * 4
    nd = len(wl.dec_layers)
    draft = draft_attn = 0
    for L, kb in zip(lens.tolist(), k_b.tolist()):
        for i in range(1, kb + 1):
            draft_attn += nd * ((L + i) * R + qo)
            draft += nd * ((L + i) * R + qo + 2 * R)
    verify = verify_attn = 0
    for L, kb in zip(lens.tolist(), k_b.tolist()):
        n = kb + 1
        verify_attn += n_layers * ((L + n) * R + n * qo)
        verify += n_layers * ((L + n) * R + n * qo + 2 * n * R)
    W = wl.kmax + 1
    accept = wl.batch * 4 * ((wl.kmax + W + 2) + (2 * W + 2))
    return dict(draft=draft, draft_attn=draft_attn, verify=verify, verify_attn=verify_attn,
                accept=accept, total=draft + verify + accept)


# ------------------------------------------------------------------ clocks
class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "200", "-f", self.path],
                stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        smax = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i] == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None, "reasons": reasons,
                "samples": len(rows)}


# ------------------------------------------------------------------ oracle leg
def oracle_sample(wl, budget_s: float) -> dict:
    """The oracle timed on host cores over a bounded sample of one round: the
    draft attention of step 1 in both decoder layers and the verify attention
    of as many layers as fit in the budget, all sequences."""
    from oracle.workload import OracleRun

    orc = OracleRun(wl, rounds=1)
    lens = orc.lens.copy()
    k_b = gen.round_plan(wl, 0)[0]
    R = wl.row_bytes
    qo = wl.hq * wl.head_dim * 6 + wl.hq * 4
    done = 0
    t0 = time.perf_counter()
    for l in wl.dec_layers:
        orc.draft(0, 1, l)
        done += sum((int(L) + 1) * R + qo for L in lens)
    layers = 0
    while time.perf_counter() - t0 < budget_s and layers < wl.n_layers:
        orc.verify(0, layers)
        orc._ctx_cache.clear()
        done += sum((int(L) + int(k) + 1) * R + (int(k) + 1) * qo for L, k in zip(lens, k_b))
        layers += 1
    dt = time.perf_counter() - t0
    return {"value": done / dt / 1e9, "unit": UNIT, "cores": len(os.sched_getaffinity(0)),
            "kind": "oracle", "seconds": round(dt, 2),
            "sample": f"workload {wl.index}: draft step 1 in {len(wl.dec_layers)} decoder layers "
                      f"+ verify attention of {layers} of {wl.n_layers} layers, all "
                      f"{wl.batch} sequences, float64 NumPy"}


# ------------------------------------------------------------------ GPU leg
def run_seed(args, rank, world, device):
    import torch

    from paper_2609_36590_gb300 import build
    build.build()
    from workloads.device import DeviceWorkload

    wl = WORKLOADS[args.workload]
    W, K = args.warmup, args.steps
    torch.cuda.set_device(device)
    dw = DeviceWorkload(wl, device=device, rounds=W + K + 1)
    stream = torch.cuda.Stream(device=device)

    # host bookkeeping of lengths (the planned acceptance is what accept returns)
    lens = [dw.lens0.astype(np.int64)]
    for r in range(W + K):
        _, n_plan, _, _ = gen.round_plan(wl, r)
        lens.append(lens[-1] + n_plan + 1)
    for r in range(W + K):
        dw.round_inputs(r)

    # round 0 runs eagerly (sets launch attributes); later rounds replay graphs
    with torch.cuda.stream(stream):
        dw.run_round(0)
    stream.synchronize()
    assert int(dw.err.item()) == 0, "device error flag raised in warm-up"

    graphs = {}
    for r in range(1, W + K):
        ins = dw.round_inputs(r)
        gd, gv, ga = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
        with torch.cuda.graph(gd, stream=stream):
            for i in range(1, ins["steps"] + 1):
                dw.draft_step(ins, i)
        with torch.cuda.graph(gv, stream=stream):
            for l in dw.layers:
                dw.verify_layer(ins, l)
        with torch.cuda.graph(ga, stream=stream):
            dw.accept(ins)
        graphs[r] = (gd, gv, ga)

    for r in range(1, W):
        for g in graphs[r]:
            g.replay()
    torch.cuda.synchronize()

    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(K)]
    sampler = ClockSampler(torch.cuda.current_device()) if rank == 0 else None
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    if sampler:
        sampler.start()
    with torch.cuda.stream(stream):
        for t in range(K):
            gd, gv, ga = graphs[W + t]
            ev[t][0].record(stream)
            gd.replay()
            ev[t][1].record(stream)
            gv.replay()
            ev[t][2].record(stream)
            ga.replay()
            ev[t][3].record(stream)
    stream.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    clocks = sampler.stop() if sampler else None
    assert int(dw.err.item()) == 0, "device error flag raised in timed rounds"
    got_lens = dw.ctx_lens.cpu().numpy()
    assert (got_lens == lens[W + K]).all(), "accepted lengths diverged from the plan"

    t_round = [ev[t][0].elapsed_time(ev[t][3]) for t in range(K)]
    t_draft = [ev[t][0].elapsed_time(ev[t][1]) for t in range(K)]
    t_verify = [ev[t][1].elapsed_time(ev[t][2]) for t in range(K)]
    byt = [round_bytes(wl, lens[W + t], gen.round_plan(wl, W + t)[0], len(dw.layers))
           for t in range(K)]
    total_ms = sum(t_round)
    total_bytes = sum(b["total"] for b in byt)
    steps_per_round = [int(gen.round_plan(wl, W + t)[0].max()) for t in range(K)]

    # dominant kernel: verify attention alone, all layers back to back
    ins = dw.round_inputs(W + K - 1)
    gk = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gk, stream=stream):
        for l in dw.layers:
            q, _, _ = ins["verify"][l]
            import paper_2609_36590_gb300 as seed
            seed.seed_verify_attn(dw.cfg, q, ins["n_q"], dw.kv[l], dw.ctx_lens, dw.out_v,
                                  dw.lse_v, dw.ws, dw.err)
    for _ in range(2):
        gk.replay()
    k0, k1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = max(3, K)
    with torch.cuda.stream(stream):
        k0.record(stream)
        for _ in range(reps):
            gk.replay()
        k1.record(stream)
    stream.synchronize()
    cur = got_lens.astype(np.int64)
    kbytes = round_bytes(wl, cur, ins["k_b_np"], len(dw.layers))["verify_attn"]
    per_launch_s = k0.elapsed_time(k1) / 1e3 / (reps * len(dw.layers))
    k_gbs = kbytes / len(dw.layers) / per_launch_s / 1e9

    res = dict(total_ms=total_ms, total_bytes=total_bytes, t_round=t_round, t_draft=t_draft,
               t_verify=t_verify, steps_per_round=steps_per_round, clocks=clocks,
               kernel_gbs=k_gbs, kernel_us=per_launch_s * 1e6,
               kernel_bytes=kbytes / len(dw.layers), n_launches=count_launches(wl, steps_per_round,
                                                                               len(dw.layers)))
    if not args.no_e2e:
        res["e2e"] = run_e2e(dw, wl, stream, W, K, lens)
    return res


def count_launches(wl, steps_per_round, n_layers):
    nd = len(wl.dec_layers)
    return sum(2 * nd * s + 2 * n_layers + 1 for s in steps_per_round)


def run_e2e(dw, wl, stream, W, K, lens):
    """Same rounds end to end through the public API: every round copies its
    inputs from pinned host buffers, runs, and reads back the accept results."""
    import torch

    dev = dw.device
    B, Hq, Hkv, D, Km = wl.batch, wl.hq, wl.hkv, wl.head_dim, wl.kmax
    steps = Km
    dec = list(wl.dec_layers)
    # device staging for one round's inputs, filled by host->device copies
    st = dict(
        dq=torch.empty(steps, len(dec), B, Hq, D, dtype=torch.bfloat16, device=dev),
        dk=torch.empty(steps, len(dec), B, Hkv, D, dtype=torch.bfloat16, device=dev),
        dv=torch.empty(steps, len(dec), B, Hkv, D, dtype=torch.bfloat16, device=dev),
        vq=torch.empty(len(dw.layers), B, Km + 1, Hq, D, dtype=torch.bfloat16, device=dev),
        vk=torch.empty(len(dw.layers), B, Km + 1, Hkv, D, dtype=torch.bfloat16, device=dev),
        vv=torch.empty(len(dw.layers), B, Km + 1, Hkv, D, dtype=torch.bfloat16, device=dev),
        ints=torch.empty(steps + 2, B, dtype=torch.int32, device=dev))
    ints = st["ints"]
    ins = dict(steps=steps, draft_lens=[ints[i] for i in range(steps)], k_b=ints[steps],
               n_q=ints[steps + 1])
    ins["draft_ids"] = torch.empty(B, Km, dtype=torch.int32, device=dev)
    ins["target_ids"] = torch.empty(B, Km + 1, dtype=torch.int32, device=dev)
    ins["draft"] = {(i, l): (st["dq"][i - 1, j], st["dk"][i - 1, j], st["dv"][i - 1, j])
                    for i in range(1, steps + 1) for j, l in enumerate(dec)}
    ins["verify"] = {l: (st["vq"][j], st["vk"][j], st["vv"][j]) for j, l in enumerate(dw.layers)}

    def host_round(r):
        """Pinned host copies of round r's inputs (built outside the timing)."""
        d = dw.round_inputs(r)
        h = {}
        h["dq"] = torch.stack([torch.stack([d["draft"].get((i, l), d["draft"][(1, l)])[0]
                                            for l in dec]) for i in range(1, steps + 1)])
        h["dk"] = torch.stack([torch.stack([d["draft"].get((i, l), d["draft"][(1, l)])[1]
                                            for l in dec]) for i in range(1, steps + 1)])
        h["dv"] = torch.stack([torch.stack([d["draft"].get((i, l), d["draft"][(1, l)])[2]
                                            for l in dec]) for i in range(1, steps + 1)])
        h["vq"] = torch.stack([d["verify"][l][0] for l in dw.layers])
        h["vk"] = torch.stack([d["verify"][l][1] for l in dw.layers])
        h["vv"] = torch.stack([d["verify"][l][2] for l in dw.layers])
        kb = d["k_b_np"]
        rows = [np.where(kb >= i, i, 0) for i in range(1, steps + 1)] + [kb, kb + 1]
        h["ints"] = torch.from_numpy(np.stack(rows).astype(np.int32))
        h["draft_ids"] = d["draft_ids"]
        h["target_ids"] = d["target_ids"]
        return {k: v.cpu().pin_memory() for k, v in h.items()}

    # fresh state: rebuild lengths for rounds W..W+K-1 from round W's start
    rounds = list(range(W, W + K))
    hosts = {r: host_round(r) for r in rounds}
    dw.ctx_lens.copy_(torch.from_numpy(lens[W].astype(np.int32)))
    g = torch.cuda.CUDAGraph()
    # warm the staging path once eagerly, then capture
    for k, v in hosts[rounds[0]].items():
        (st.get(k) if k in st else ins[k]).copy_(v)
    with torch.cuda.graph(g, stream=stream):
        for i in range(1, steps + 1):
            dw.draft_step(ins, i)
        for l in dw.layers:
            dw.verify_layer(ins, l)
        dw.accept(ins)
    out_h = [torch.empty(B, dtype=torch.int32).pin_memory(),
             torch.empty(B, Km + 1, dtype=torch.int32).pin_memory(),
             torch.empty(B, Km + 1, dtype=torch.int32).pin_memory(),
             torch.empty(B, dtype=torch.int32).pin_memory()]
    h2d = sum(v.numel() * v.element_size() for v in hosts[rounds[0]].values())
    d2h = sum(v.numel() * v.element_size() for v in out_h)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        for r in rounds:
            for k, v in hosts[r].items():
                (st.get(k) if k in st else ins[k]).copy_(v, non_blocking=True)
            g.replay()
            for dst, src in zip(out_h, (dw.accepted, dw.tokens, dw.slots, dw.ctx_lens)):
                dst.copy_(src, non_blocking=True)
        e1.record(stream)
    stream.synchronize()
    assert (out_h[3].numpy() == lens[W + K]).all(), "e2e lengths diverged"
    ms = e0.elapsed_time(e1)
    tot = sum(round_bytes(wl, lens[r], gen.round_plan(wl, r)[0], len(dw.layers))["total"]
              for r in rounds)
    return {"value": tot / (ms / 1e3) / 1e9, "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": ms / K}


# ------------------------------------------------------------------ main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", type=int, default=3, choices=[1, 2, 3, 4, 5])
    ap.add_argument("--impl", default="seed", choices=["seed", "reference"])
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=12.0)
    args = ap.parse_args()
    if args.warmup < 1:
        ap.error("--warmup must be >= 1")

    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    local = int(os.environ.get("LOCAL_RANK", 0))
    wl = WORKLOADS[args.workload]
    peak, peak_kind = load_peaks()
    config = {"workload": wl.name, "batch": wl.batch, "layers": wl.n_layers,
              "decoder_layers": len(wl.dec_layers), "hq": wl.hq, "hkv": wl.hkv,
              "head_dim": wl.head_dim, "kmax": wl.kmax, "page_size": 16,
              "l2": "inputs larger than L2: each round streams the KV of every layer",
              "parallelism": f"replicas x{world}" if world > 1 else "single GPU"}

    if args.impl == "reference":
        if rank != 0:
            return
        vals = []
        for _ in range(args.warmup):
            oracle_sample(wl, min(args.cpu_budget, 3.0))
        t0 = time.perf_counter()
        for _ in range(args.steps):
            vals.append(oracle_sample(wl, args.cpu_budget / max(1, args.steps)))
        dt = time.perf_counter() - t0
        v = statistics.mean(x["value"] for x in vals)
        line = {"metric": METRIC, "value": v, "unit": UNIT, "impl": "reference", "n_gpus": 1,
                "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": dt * 1e3 / args.steps, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": config,
                "cpu_baseline": dict(vals[-1], value=v),
                "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return

    import torch
    if world > 1:
        torch.distributed.init_process_group("nccl", device_id=torch.device(f"cuda:{local}"))
    device = f"cuda:{local}"
    res = run_seed(args, rank, world, device)

    total_s = res["total_ms"] / 1e3
    if world > 1:
        t = torch.tensor([total_s], device=device)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        total_s = float(t.item())
    value = world * res["total_bytes"] / total_s / 1e9
    if rank == 0:
        cpu = oracle_sample(wl, args.cpu_budget) if world == 1 else None
        K = args.steps
        line = {
            "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
            "steps": K, "warmup": args.warmup, "ms_per_step": total_s * 1e3 / K,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic", "config": config,
            "pct_of_peak": round(100 * value / world / peak, 1), "peak_gbs": peak,
            "peak_kind": peak_kind, "pct_of_8000": round(100 * value / world / 8000, 1),
            "draft_step_us": 1e3 * sum(res["t_draft"]) / sum(res["steps_per_round"]),
            "verify_step_us": 1e3 * statistics.mean(res["t_verify"]),
            "round_us": 1e3 * statistics.mean(res["t_round"]),
            "roofline": {"bound": "hbm", "kernel": "seed_verify_attn (decode_attn_kernel)",
                         "achieved": round(res["kernel_gbs"], 1), "peak": peak,
                         "unit": "GB/s", "frac": round(res["kernel_gbs"] / peak, 3),
                         "peak_kind": peak_kind, "traffic": None,
                         "bytes_per_launch": res["kernel_bytes"],
                         "us_per_launch": round(res["kernel_us"], 2)},
            "gpu_launches": res["n_launches"],
            "clocks": res["clocks"],
            "cpu_baseline": cpu,
        }
        if "e2e" in res:
            line["e2e"] = res["e2e"]
        print(json.dumps(line))
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
