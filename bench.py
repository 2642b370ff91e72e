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

    python bench.py [--workload 4] [--steps 10] [--warmup 3] [--impl seed|reference]
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


def load_bf16_peak():
    """Dense bf16 tensor-core peak (TFLOP/s, burst) from the measured file, else
    the fallback figure."""
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            return float(json.load(f)["bf16_tflops"])
    return 1900.0


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


# ------------------------------------------------------------------ ncu traffic
# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) of one attention
# launch from an ncu capture of `bench.py --profile <kind> --workload <n>`
# (one launch on the workload's two decoder layers), with the algorithmic bytes
# of that launch and a hash of the kernel's sources at capture time.  The
# reported traffic is scaled to the timed launches by their algorithmic bytes,
# and is null once the kernel's sources differ from the captured ones.
NCU_TRAFFIC = {
    (4, "verify"): {"kernel": "attn_tc_kernel", "sources": "a9f183f7f0271aeb",
                    "dram_bytes": 537557760 + 3322112, "alg_bytes": 537907712},
    (4, "draft"): {"kernel": "attn_tc_kernel", "sources": "a9f183f7f0271aeb",
                   "dram_bytes": 537235712 + 3060480, "alg_bytes": 536986112},
}

KERNEL_SOURCES = {
    "attn_tc_kernel": ["attn_tc.cu", "attn_sched.cuh", "tc.cuh", "common.cuh", "kernels.h"],
    "attn_kt_kernel": ["attn_kt.cu", "attn_sched.cuh", "tc.cuh", "common.cuh", "kernels.h"],
    "decode_attn_kernel": ["decode_attn.cu", "common.cuh", "kernels.h"],
    "attn_cl_kernel": ["attn_cluster.cu", "attn_sched.cuh", "tc.cuh", "common.cuh", "kernels.h"],
}


def kernel_source_hash(name: str) -> str:
    import hashlib
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[name]:
        with open(os.path.join(ROOT, "paper_2609_36590_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def ncu_traffic(wl, kind: str, alg_bytes: float):
    rec = NCU_TRAFFIC.get((wl.index, kind))
    name = attn_kernel_name(wl, kind)
    if rec is None or rec["kernel"] != name or rec["sources"] != kernel_source_hash(name):
        return None
    return round(rec["dram_bytes"] * alg_bytes / rec["alg_bytes"])


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
def blas_threads():
    """Threads of the BLAS that NumPy calls (the oracle's matrix products)."""
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads") for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return int(max(n))
    except Exception:
        pass
    for k in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
        if os.environ.get(k, "").isdigit():
            return int(os.environ[k])
    return None


class OracleSlice:
    """A fixed slice of round 0 of the workload, run by the oracle on host
    cores: draft step 1 in both decoder layers, then the verify attention of
    layer 0, all sequences.  The same slice serves the reference arm (one
    slice per step) and the cpu_baseline of the GPU arm (median of 3)."""

    def __init__(self, wl):
        from oracle.workload import OracleRun
        self.wl = wl
        self.orc = OracleRun(wl, rounds=1)
        lens = self.orc.lens.copy()
        k_b = gen.round_plan(wl, 0)[0]
        R = wl.row_bytes
        qo = wl.hq * wl.head_dim * 6 + wl.hq * 4
        self.draft_bytes = len(wl.dec_layers) * sum((int(L) + 1) * R + qo for L in lens)
        self.verify_bytes = sum((int(L) + int(k) + 1) * R + (int(k) + 1) * qo
                                for L, k in zip(lens, k_b))
        self.bytes = self.draft_bytes + self.verify_bytes
        self.steps = int(k_b.max())

    def run_draft(self) -> float:
        t0 = time.perf_counter()
        for l in self.wl.dec_layers:
            self.orc.draft(0, 1, l)
        return time.perf_counter() - t0

    def run_verify(self) -> float:
        t0 = time.perf_counter()
        self.orc.verify(0, 0)
        self.orc._ctx_cache.clear()
        return time.perf_counter() - t0

    def run(self) -> tuple[float, float]:
        return self.run_draft(), self.run_verify()

    def describe(self, td: float, tv: float, reps: int) -> dict:
        wl = self.wl
        t = td + tv
        threads = blas_threads()
        return {"value": self.bytes / t / 1e9, "unit": UNIT,
                "cores": threads if threads else len(os.sched_getaffinity(0)),
                "host_cores": len(os.sched_getaffinity(0)), "blas_threads": threads,
                "kind": "oracle",
                "sample": f"workload {wl.index}: draft step 1 in {len(wl.dec_layers)} decoder "
                          f"layers + verify attention of 1 of {wl.n_layers} verify layers "
                          f"(layer 0), all {wl.batch} sequences, float64 NumPy; "
                          f"median of {reps}",
                "slice_us": round(t * 1e6, 1),
                "draft_layer_us": round(td * 1e6 / len(wl.dec_layers), 1),
                "verify_layer_us": round(tv * 1e6, 1),
                "round_us_extrapolated": round(
                    1e6 * (td * self.steps + tv * wl.n_layers), 1),
                "extrapolation": f"round = draft part x {self.steps} steps + verify layer x "
                                 f"{wl.n_layers} layers (extrapolated, not timed)"}


def oracle_sample(wl, reps: int = 3) -> dict:
    """cpu_baseline: the fixed slice, timed reps times; the median slice."""
    sl = OracleSlice(wl)
    runs = sorted((sl.run() for _ in range(reps)), key=lambda x: x[0] + x[1])
    td, tv = runs[len(runs) // 2]
    return sl.describe(td, tv, reps)


# ------------------------------------------------------------------ GPU leg
def run_seed(args, rank, world, device):
    import torch

    from paper_2609_36590_gb300 import build
    build.build()
    from workloads.device import DeviceWorkload

    wl = WORKLOADS[args.workload]
    W, K = args.warmup, args.steps
    torch.cuda.set_device(device)
    # rounds [W, W+K) are the timed steps; rounds [W+K, W+2K) repeat the same
    # kind of step with timing events around every attention launch (those
    # events serialise the stream, so they stay out of the timed steps)
    n_rounds = W + 2 * K
    dw = DeviceWorkload(wl, device=device, rounds=n_rounds + 1)
    stream = torch.cuda.Stream(device=device)

    # host bookkeeping of lengths (the planned acceptance is what accept returns)
    lens = [dw.lens0.astype(np.int64)]
    for r in range(n_rounds):
        _, n_plan, _, _ = gen.round_plan(wl, r)
        lens.append(lens[-1] + n_plan + 1)
    for r in range(n_rounds):
        dw.round_inputs(r)

    # round 0 runs eagerly (sets launch attributes); later rounds replay graphs
    with torch.cuda.stream(stream):
        dw.run_round(0)
    stream.synchronize()
    assert int(dw.err.item()) == 0, f"device error flag {int(dw.err.item())} raised in warm-up"

    graphs, timers, b2b = {}, {}, {}
    for r in range(1, n_rounds):
        ins = dw.round_inputs(r)
        marks = None
        if r >= W + K:
            timers[r] = AttnTimer()
            marks = timers[r].marks()
        gd, gv, ga = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
        with torch.cuda.graph(gd, stream=stream):
            for i in range(1, ins["steps"] + 1):
                dw.draft_step(ins, i, marks=marks)
        with torch.cuda.graph(gv, stream=stream):
            for l in dw.layers:
                dw.verify_layer(ins, l, marks=marks)
        with torch.cuda.graph(ga, stream=stream):
            dw.accept(ins)
        graphs[r] = (gd, gv, ga)
        if r >= W + K:
            # the same round's attention calls alone, back to back as in the
            # round (one graph each), replayed after its draft and verify
            # phases, before accept: same caches, lengths and draft rows
            gda, gva = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
            with torch.cuda.graph(gda, stream=stream):
                for i in range(1, ins["steps"] + 1):
                    for l in wl.dec_layers:
                        dw.draft_attn(ins, i, l)
            with torch.cuda.graph(gva, stream=stream):
                for l in dw.layers:
                    dw.verify_attn(ins, l)
            b2b[r] = (gda, gva)

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
    # the kernel-timing rounds: every attention launch between events, then
    # the same calls back to back between one pair of events
    bev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(K)]
    with torch.cuda.stream(stream):
        for t in range(K):
            gd, gv, ga = graphs[W + K + t]
            gda, gva = b2b[W + K + t]
            gd.replay()
            gv.replay()
            bev[t][0].record(stream)
            gda.replay()
            bev[t][1].record(stream)
            gva.replay()
            bev[t][2].record(stream)
            ga.replay()
    stream.synchronize()
    clocks = sampler.stop() if sampler else None
    assert int(dw.err.item()) == 0, f"device error flag {int(dw.err.item())} raised in timed rounds"
    got_lens = dw.ctx_lens.cpu().numpy()
    assert (got_lens == lens[n_rounds]).all(), "accepted lengths diverged from the plan"

    t_round = [ev[t][0].elapsed_time(ev[t][3]) for t in range(K)]
    t_draft = [ev[t][0].elapsed_time(ev[t][1]) for t in range(K)]
    t_verify = [ev[t][1].elapsed_time(ev[t][2]) for t in range(K)]
    t_accept = [ev[t][2].elapsed_time(ev[t][3]) for t in range(K)]
    byt = [round_bytes(wl, lens[W + t], gen.round_plan(wl, W + t)[0], len(dw.layers))
           for t in range(K)]
    total_ms = sum(t_round)
    total_bytes = sum(b["total"] for b in byt)
    steps_per_round = [int(gen.round_plan(wl, W + t)[0].max()) for t in range(K)]

    # attention kernels: every launch of the kernel-timing rounds, timed by
    # the events recorded around it inside the round graphs
    kern = {}
    for kind in ("verify", "draft"):
        nbytes = secs = launches = 0
        for r in range(W + K, n_rounds):
            k_b = gen.round_plan(wl, r)[0]
            for key, ms in timers[r].durations(kind):
                nbytes += attn_call_bytes(wl, kind, key, lens[r], k_b)
                secs += ms / 1e3
                launches += 1
        # back to back: the kind's calls of each kernel-timing round between
        # one pair of events
        bsecs = 0.0
        for t in range(K):
            a, b = (0, 1) if kind == "draft" else (1, 2)
            bsecs += bev[t][a].elapsed_time(bev[t][b]) / 1e3
        kern[kind] = dict(gbs=nbytes / bsecs / 1e9, us=bsecs / launches * 1e6,
                          gbs_isolated=nbytes / secs / 1e9, us_isolated=secs / launches * 1e6,
                          bytes=nbytes / launches, launches=launches)

    res = dict(total_ms=total_ms, total_bytes=total_bytes, t_round=t_round, t_draft=t_draft,
               t_verify=t_verify, t_accept=t_accept, steps_per_round=steps_per_round,
               clocks=clocks, kern=kern,
               n_launches=count_launches(wl, steps_per_round, len(dw.layers)))
    if not args.no_e2e:
        res["e2e"] = run_e2e(dw, wl, stream, W, K, lens)
    return res


class AttnTimer:
    """CUDA events recorded around each attention call while a round graph is
    captured.  They are external events, so the graph holds real event-record
    nodes and every replay stamps them on the launching stream."""

    def __init__(self):
        self.calls = []

    def marks(self):
        import torch

        def before(kind, key):
            e = torch.cuda.Event(enable_timing=True, external=True)
            e.record()
            self.calls.append([kind, key, e, None])

        def after(kind, key):
            e = torch.cuda.Event(enable_timing=True, external=True)
            e.record()
            self.calls[-1][3] = e

        return before, after

    def durations(self, kind):
        return [(key, a.elapsed_time(b)) for k, key, a, b in self.calls if k == kind]


def attn_call_bytes(wl, kind, key, lens, k_b) -> int:
    """Algorithmic bytes of one attention launch (one layer): every visible K/V
    row once, plus q in and o, lse out for each active query row."""
    R = wl.row_bytes
    qo = wl.hq * wl.head_dim * (2 + 4) + wl.hq * 4
    if kind == "draft":
        i = key[0]
        return sum((int(L) + i) * R + qo for L, kb in zip(lens, k_b) if kb >= i)
    return sum((int(L) + int(kb) + 1) * R + (int(kb) + 1) * qo for L, kb in zip(lens, k_b))


def attn_kernel_name(wl, kind: str = "verify") -> str:
    """The kernel behind seed_draft_attn / seed_verify_attn ("draft",
    "verify") or seed_tree_verify_attn ("tree") for this workload.  On a GPU
    the library says (seed_attn_route: few (sequence, KV head) pairs and short
    page tables take the cluster kernel); the shape rule below is the rest of
    the choice: head_dim 128 with the query rows of one KV head in one 128-row
    tile: the query-rows tensor-core kernel; head_dim 64 with at most 48 such
    rows: the keys-as-rows tensor-core kernel; else the CUDA-core split-KV
    kernel."""
    if kind != "tree":
        try:
            import torch
            if torch.cuda.is_available():
                import paper_2609_36590_gb300 as seed
                cfg = seed.SeedConfig(hq=wl.hq, hkv=wl.hkv, head_dim=wl.head_dim, kmax=wl.kmax)
                r = seed.seed_attn_route(cfg, wl.batch, kind == "draft", gen.max_pages(wl))
                return seed.ROUTE_KERNELS[r]
        except (ImportError, OSError, RuntimeError):
            pass
    G = wl.hq // wl.hkv
    w1 = 1 if kind == "draft" else wl.kmax + 1
    if wl.head_dim == 128 and G * w1 <= 128:
        return "attn_tc_kernel"
    if wl.head_dim == 64 and G * w1 <= 48:
        return "attn_kt_kernel"
    return "decode_attn_kernel"


def run_profile(args):
    """--profile draft|verify|tree: the appends of round 0 on the workload's two
    decoder layers, then `--reps` launches of one attention kind alternating
    between them (a few hundred MB of KV, above the L2 size).  `tree` verifies
    a full draft tree of kmax+1 nodes per sequence (binary, node i's parent is
    (i-1)/2) with the tree mask of Sec. D.1.  For ncu captures of one launch
    (`-k regex:<kernel> -s 2 -c 1`); prints the algorithmic bytes of each
    launch, no bench value."""
    import torch

    from paper_2609_36590_gb300 import build
    build.build()
    import paper_2609_36590_gb300 as seed
    from workloads.device import DeviceWorkload

    wl = WORKLOADS[args.workload]
    if args.prefix is not None or args.batch is not None:
        # the workload's heads and draft lengths with a fixed prefix length
        # and/or another batch (e.g. a head_dim 64 verify over a 32k prefix)
        import dataclasses
        L = args.prefix if args.prefix is not None else wl.ctx_lo
        B = args.batch if args.batch is not None else wl.batch
        fixed = args.prefix is not None
        wl = dataclasses.replace(wl, batch=B, ctx="fixed" if fixed else wl.ctx,
                                 ctx_lo=L if fixed else wl.ctx_lo,
                                 ctx_hi=L if fixed else wl.ctx_hi,
                                 name=f"{wl.name} (batch {B}, prefix {L if fixed else 'as is'})")
    torch.cuda.set_device(0)
    if args.profile == "head":
        run_profile_head(args, wl, args.head_batch)
        return
    if args.profile == "draftstep":
        run_profile_draftstep(args, wl)
        return
    if args.profile == "blockattn":
        run_profile_blockattn(args, wl)
        return
    dw = DeviceWorkload(wl, device="cuda:0", layers=list(wl.dec_layers), rounds=2)
    ins = dw.round_inputs(0)
    k_b = ins["k_b_np"]
    lens = dw.lens0
    dec = list(wl.dec_layers)
    W = wl.kmax + 1
    n_q = ins["n_q"]
    if args.profile == "tree":
        k_b = np.full(wl.batch, W - 1, dtype=np.int64)
        n_q = torch.full((wl.batch,), W, dtype=torch.int32, device="cuda:0")
        anc = np.zeros(W, dtype=np.int64)
        for i in range(W):
            a = i
            while True:
                anc[i] |= 1 << a
                if a == 0:
                    break
                a = (a - 1) // 2
        anc_dev = torch.from_numpy(np.tile(anc.astype(np.uint32).view(np.int32),
                                           (wl.batch, 1))).to("cuda:0")
    for l in dec:
        q, kn, vn = ins["draft"][(1, l)]
        seed.seed_draft_kv_append(dw.cfg, kn, vn, ins["draft_lens"][0], dw.draft_k[l],
                                  dw.draft_v[l], dw.err)
        _, kn, vn = ins["verify"][l]
        seed.seed_kv_append(dw.cfg, dw.kv[l], kn, vn, n_q, dw.ctx_lens, dw.err)
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.reps + 1)]
    ev[0].record()
    for r in range(args.reps):
        l = dec[r % len(dec)]
        if args.profile == "draft":
            dw.draft_attn(ins, 1, l)
        elif args.profile == "tree":
            seed.seed_tree_verify_attn(dw.cfg, ins["verify"][l][0], n_q, anc_dev, dw.kv[l],
                                       dw.ctx_lens, dw.out_v, dw.lse_v, dw.ws, dw.err)
        else:
            dw.verify_attn(ins, l)
        ev[r + 1].record()
    torch.cuda.synchronize()
    assert int(dw.err.item()) == 0, f"device error flag {int(dw.err.item())} raised"
    key = (1, dec[0]) if args.profile == "draft" else dec[0]
    nbytes = attn_call_bytes(wl, "draft" if args.profile == "draft" else "verify", key, lens, k_b)
    kname = attn_kernel_name(wl, args.profile)
    print(json.dumps({"profile": args.profile, "workload": wl.name,
                      "kernel": kname, "sources": kernel_source_hash(kname),
                      "alg_bytes_per_launch": nbytes,
                      "us": [round(ev[i].elapsed_time(ev[i + 1]) * 1e3, 1)
                             for i in range(args.reps)]}))


HEAD_D_MODEL, HEAD_VOCAB = 2560, 151936   # a 4B-scale (Qwen3-4B) LM head


def run_profile_head(args, wl, batch=None):
    """--profile head: the dynamic-drafting head (LM head + softmax + top-10,
    Sec. D.1) at 4B scale (d = 2560, V = 151936) for the workload's batch (or
    `batch`), `--reps` launches back to back after 3 warm-up launches.  The
    head's 778 MB of weights are far above the L2 size, so every launch
    streams them from HBM.  Algorithmic bytes: the weights once, h, and the
    outputs.  Times are CUDA events between consecutive launches (head kernel
    plus merge kernel)."""
    import torch

    import paper_2609_36590_gb300 as seed

    B, d, V = batch or wl.batch, HEAD_D_MODEL, HEAD_VOCAB
    g = torch.Generator(device="cuda:0").manual_seed(20260)
    h = torch.randn(B, d, device="cuda:0", generator=g).to(torch.bfloat16)
    w = (torch.randn(V, d, device="cuda:0", generator=g) / d ** 0.5).to(torch.bfloat16)
    ids = torch.empty(B, 10, dtype=torch.int32, device="cuda:0")
    probs = torch.empty(B, 10, device="cuda:0")
    n_sib = torch.empty(B, dtype=torch.int32, device="cuda:0")
    stop = torch.empty(B, dtype=torch.int32, device="cuda:0")
    lse = torch.empty(B, device="cuda:0")
    err = torch.zeros(1, dtype=torch.int32, device="cuda:0")
    ws = seed.new_draft_head_workspace(B)
    for _ in range(3):
        seed.seed_draft_head_topk(h, w, 0.7, ids, probs, n_sib, stop, lse, ws, err)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.reps + 1)]
    torch.cuda.synchronize()
    ev[0].record()
    for r in range(args.reps):
        seed.seed_draft_head_topk(h, w, 0.7, ids, probs, n_sib, stop, lse, ws, err)
        ev[r + 1].record()
    torch.cuda.synchronize()
    assert int(err.item()) == 0, f"device error flag {int(err.item())} raised"
    nbytes = V * d * 2 + B * d * 2 + B * (10 * 8 + 12)
    us = [ev[i].elapsed_time(ev[i + 1]) * 1e3 for i in range(args.reps)]
    med = float(np.median(us))
    peak, kind = load_peaks()
    gbs = nbytes / med / 1e3
    print(json.dumps({"profile": "head", "workload": wl.name, "batch": B, "d_model": d,
                      "vocab": V, "kernel": "head_tc_kernel + head_merge_kernel",
                      "alg_bytes_per_launch": nbytes, "us_median": round(med, 1),
                      "achieved_gbs": round(gbs, 1), "peak_gbs": peak, "peak_kind": kind,
                      "frac": round(gbs / peak, 3), "us": [round(u, 1) for u in us]}))


DRAFTER = dict(d_model=2560, d_ff=9728)   # Qwen3-4B decoder layers


def drafter_bytes(wl) -> int:
    """Weight bytes one draft step reads: per decoder layer W_qkv, W_o,
    W_gate, W_up, W_down and three norm gains, plus the tied head."""
    dm, F, D = DRAFTER["d_model"], DRAFTER["d_ff"], wl.head_dim
    per_layer = (wl.hq + 2 * wl.hkv) * D * dm + dm * wl.hq * D + 3 * F * dm + 2 * dm + 2 * D
    return 2 * (len(wl.dec_layers) * per_layer + HEAD_VOCAB * dm + dm)


def run_profile_draftstep(args, wl):
    """--profile draftstep: one whole draft step of the workload's batch on the
    device -- embedding, the two decoder layers (norms, QKV, q/k norm + RoPE,
    draft KV append, draft attention over the layer's cache, output product,
    SwiGLU MLP), final norm and the dynamic-drafting head -- with random
    bf16 weights of a Qwen3-4B drafter, replayed `--reps` times from one CUDA
    graph.  Algorithmic bytes: the drafter's weights once, plus each decoder
    layer's draft attention bytes (its visible K/V rows, q, o).  Weights and
    caches (GBs) are far above the L2 size."""
    import torch

    import paper_2609_36590_gb300 as seed
    from workloads.device import DeviceWorkload

    dev = "cuda:0"
    dw = DeviceWorkload(wl, device=dev, layers=list(wl.dec_layers), rounds=2)
    ins = dw.round_inputs(0)
    B, dm, F, D = wl.batch, DRAFTER["d_model"], DRAFTER["d_ff"], wl.head_dim
    g = torch.Generator(device=dev).manual_seed(20261)

    def w(*shape, s=1.0):
        return (torch.randn(*shape, device=dev, generator=g) * s).to(torch.bfloat16)

    def gain(n):
        return (1.0 + 0.1 * torch.randn(n, device=dev, generator=g)).to(torch.bfloat16)

    layers = {l: seed.DecoderLayer(
        g_attn=gain(dm), w_qkv=w((wl.hq + 2 * wl.hkv) * D, dm, s=dm ** -0.5), g_q=gain(D),
        g_k=gain(D), w_o=w(dm, wl.hq * D, s=(wl.hq * D) ** -0.5), g_mlp=gain(dm),
        w_gate=w(F, dm, s=dm ** -0.5), w_up=w(F, dm, s=dm ** -0.5), w_down=w(dm, F, s=F ** -0.5))
        for l in wl.dec_layers}
    w_emb = w(HEAD_VOCAB, dm, s=0.02)
    g_final = gain(dm)
    tokens = torch.randint(0, HEAD_VOCAB, (B,), device=dev, generator=g, dtype=torch.int32)
    draft_lens = ins["draft_lens"][0]          # step 1 of round 0 (ragged k: some skip)
    x = torch.empty(B, dm, device=dev)
    h = torch.empty(B, dm, dtype=torch.bfloat16, device=dev)
    ids = torch.empty(B, 10, dtype=torch.int32, device=dev)
    probs = torch.empty(B, 10, device=dev)
    n_sib = torch.empty(B, dtype=torch.int32, device=dev)
    stop = torch.empty(B, dtype=torch.int32, device=dev)
    lse = torch.empty(B, device=dev)
    ws = seed.new_draft_layer_workspace(dw.cfg, layers[wl.dec_layers[0]], B, dev)
    hws = seed.new_draft_head_workspace(B, dev)
    err = dw.err

    def step():
        seed.seed_embed(tokens, w_emb, x, err)
        for l in wl.dec_layers:
            seed.seed_draft_layer(dw.cfg, layers[l], x, dw.kv[l], dw.ctx_lens, dw.draft_k[l],
                                  dw.draft_v[l], draft_lens, ws, err)
        seed.seed_rmsnorm(x, g_final, 1e-6, h)
        seed.seed_draft_head_topk(h, w_emb, 0.7, ids, probs, n_sib, stop, lse, hws, err)

    s = torch.cuda.Stream(device=dev)
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        for _ in range(3):
            step()
    torch.cuda.current_stream().wait_stream(s)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step()
    for _ in range(3):
        graph.replay()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.reps + 1)]
    torch.cuda.synchronize()
    ev[0].record()
    for r in range(args.reps):
        graph.replay()
        ev[r + 1].record()
    torch.cuda.synchronize()
    assert int(err.item()) == 0, f"device error flag {int(err.item())} raised"
    k_b = ins["k_b_np"]
    attn = sum(attn_call_bytes(wl, "draft", (1, l), dw.lens0, k_b) for l in wl.dec_layers)
    nbytes = drafter_bytes(wl) + attn
    us = [ev[i].elapsed_time(ev[i + 1]) * 1e3 for i in range(args.reps)]
    med = float(np.median(us))
    peak, kind = load_peaks()
    gbs = nbytes / med / 1e3
    print(json.dumps({"profile": "draftstep", "workload": wl.name, "batch": B,
                      "active": int((draft_lens > 0).sum().item()), "d_model": dm, "d_ff": F,
                      "vocab": HEAD_VOCAB, "weight_bytes": drafter_bytes(wl),
                      "attn_bytes": attn, "alg_bytes_per_step": nbytes,
                      "us_median": round(med, 1), "achieved_gbs": round(gbs, 1),
                      "peak_gbs": peak, "peak_kind": kind, "frac": round(gbs / peak, 3),
                      "us": [round(u, 1) for u in us]}))


def run_profile_blockattn(args, wl, n=1000, block=10, batch=8):
    """--profile blockattn: the decoder's block-causal training attention
    (Sec. 4.2) for `batch` sequences of n tokens in blocks of 10 (the paper's
    training block size) at the workload's head shape, `--reps` calls back to
    back.  Reports the attention FLOPs (4 D per query head and visible key)
    against the bf16 peak and the bytes moved against the HBM peak: on the
    tensor-core route (head_dim 128, groups 1, 2, 4) every input read once and
    o and lse written once; on the virtual-sequence route each block's deep
    prefix and own rows, q in, o and lse out, plus the paged copy it builds."""
    import torch

    import paper_2609_36590_gb300 as seed

    dev = "cuda:0"
    hq, hkv, D = wl.hq, wl.hkv, wl.head_dim
    g = torch.Generator(device=dev).manual_seed(20262)
    q = torch.randn(batch, n, hq, D, device=dev, generator=g).to(torch.bfloat16)
    kv = [torch.randn(batch, n, hkv, D, device=dev, generator=g).to(torch.bfloat16)
          for _ in range(4)]
    out = torch.empty(batch, n, hq, D, device=dev)
    lse = torch.empty(batch, n, hq, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    cfg = seed.SeedConfig(hq=hq, hkv=hkv, head_dim=D, kmax=1)
    ws = seed.new_block_attn_workspace(cfg, batch, n, block, dev)
    for _ in range(3):
        seed.seed_block_attn(cfg, block, q, *kv, out, lse, ws, err)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.reps + 1)]
    torch.cuda.synchronize()
    ev[0].record()
    for r in range(args.reps):
        seed.seed_block_attn(cfg, block, q, *kv, out, lse, ws, err)
        ev[r + 1].record()
    torch.cuda.synchronize()
    assert int(err.item()) == 0, f"device error flag {int(err.item())} raised"
    R = 2 * hkv * D * 2                               # K + V bytes of one row
    nblk = n // block
    qo = n * hq * (D * (2 + 4) + 4)
    if D == 128 and hq // hkv in (1, 2, 4):
        # tensor-core route: every input read once, o and lse written once
        route = "tensor-core"
        nbytes = batch * (2 * n * R + qo)
    else:
        route = "virtual-sequence"
        rows_read = sum(s * block + block for s in range(nblk))  # deep prefix + own rows
        pages = -(-n // 16) + nblk * -(-(15 + block) // 16)
        copy = (n * 2 * R) + pages * 16 * R           # read 4 inputs, write the paged copy
        nbytes = batch * (rows_read * R + pages * 16 * R + copy + qo)
    vis = sum(s * block + (j + 1) for s in range(nblk) for j in range(block))
    flops = batch * hq * vis * D * 4
    us = [ev[i].elapsed_time(ev[i + 1]) * 1e3 for i in range(args.reps)]
    med = float(np.median(us))
    peak, kind = load_peaks()
    gbs = nbytes / med / 1e3
    print(json.dumps({"profile": "blockattn", "route": route, "batch": batch, "n": n,
                      "block": block, "hq": hq,
                      "hkv": hkv, "head_dim": D, "bytes_moved": nbytes, "flops": flops,
                      "us_median": round(med, 1), "achieved_gbs": round(gbs, 1),
                      "peak_gbs": peak, "peak_kind": kind, "frac": round(gbs / peak, 3),
                      "tflops": round(flops / med / 1e6, 2),
                      "bf16_peak_tflops": load_bf16_peak(),
                      "us": [round(u, 1) for u in us]}))


def aggregate(rank_bytes: float, rank_seconds: float, world: int, device="cpu"):
    """Whole-job throughput of N replicas: every rank processed `rank_bytes` in
    `rank_seconds`; the job takes as long as its slowest rank.  Returns
    (max seconds over ranks, GB/s of all ranks together).  With world > 1 the
    process group must be initialised (NCCL on GPUs, gloo on CPU)."""
    import torch

    total_s = float(rank_seconds)
    if world > 1:
        t = torch.tensor([total_s], dtype=torch.float64, device=device)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        total_s = float(t.item())
    return total_s, world * rank_bytes / total_s / 1e9


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


KERN_TIMING = ("us_per_launch and achieved: each round's attention calls of the kind replayed "
               "back to back (one CUDA graph, as in the round: programmatic dependent launch "
               "between calls), CUDA events around the graph, divided by the calls; "
               "*_isolated: CUDA events around every single call of the round graphs (the "
               "events serialise the calls). Both include the merge kernel.")


def kern_line(k: dict, kernel: str, peak: float) -> dict:
    return {"kernel": kernel, "us_per_launch": round(k["us"], 2),
            "achieved": round(k["gbs"], 1), "frac": round(k["gbs"] / peak, 3),
            "us_per_launch_isolated": round(k["us_isolated"], 2),
            "frac_isolated": round(k["gbs_isolated"] / peak, 3),
            "bytes_per_launch": round(k["bytes"]), "launches": k["launches"]}


def per_workload(args, rank, device, peak) -> dict:
    """Workloads 2, 3 and 5 (batch 1, a 16-sequence mix, the 64-sequence
    paged mix), each from a fresh device workload: 3 warm-up and 3 timed
    rounds, with the attention launches of 3 more rounds timed one by one."""
    import copy
    import torch
    out = {}
    for w in (2, 3, 5):
        a = copy.copy(args)
        a.workload, a.steps, a.warmup, a.no_e2e = w, 3, 3, True
        r = run_seed(a, rank, 1, device)
        wl = WORKLOADS[w]
        kv_, kd_ = r["kern"]["verify"], r["kern"]["draft"]
        out[str(w)] = {
            "workload": wl.name,
            "value": round(r["total_bytes"] / (r["total_ms"] / 1e3) / 1e9, 1), "unit": UNIT,
            "round_us": round(1e3 * statistics.mean(r["t_round"]), 1),
            "accept_us": round(1e3 * statistics.mean(r["t_accept"]), 2),
            "verify": kern_line(kv_, attn_kernel_name(wl), peak),
            "draft": kern_line(kd_, attn_kernel_name(wl, "draft"), peak),
            "timing": "3 warm-up + 3 timed rounds; then 3 kernel-timing rounds: "
                      + KERN_TIMING}
        del r
        torch.cuda.empty_cache()
    return out


# ------------------------------------------------------------------ main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", type=int, default=4, choices=[1, 2, 3, 4, 5])
    ap.add_argument("--impl", default="seed", choices=["seed", "reference"])
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--cpu-reps", type=int, default=3,
                    help="timed repetitions of the oracle slice for cpu_baseline (0: none)")
    ap.add_argument("--no-per-workload", action="store_true",
                    help="skip the per-workload lines of workloads 2, 3 and 5")
    ap.add_argument("--profile", choices=["draft", "verify", "tree", "head", "draftstep",
                                          "blockattn"],
                    default=None,
                    help="launch one attention kind a few times for an ncu capture")
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--prefix", type=int, default=None,
                    help="--profile draft|verify|tree: a fixed prefix length instead of the "
                         "workload's")
    ap.add_argument("--batch", type=int, default=None,
                    help="--profile draft|verify|tree: batch instead of the workload's")
    ap.add_argument("--head-batch", type=int, default=None,
                    help="--profile head: batch instead of the workload's")
    args = ap.parse_args()
    if args.profile:
        run_profile(args)
        return
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
        # one step = the oracle's fixed slice; a warm-up step runs its draft
        # part (the oracle has no caches to warm, so that bounds the run)
        sl = OracleSlice(wl)
        for _ in range(args.warmup):
            sl.run_draft()
        runs = [sl.run() for _ in range(args.steps)]
        runs.sort(key=lambda x: x[0] + x[1])
        td, tv = runs[len(runs) // 2]
        cpu = sl.describe(td, tv, args.steps)
        v = cpu["value"]
        line = {"metric": METRIC, "value": v, "unit": UNIT, "impl": "reference", "n_gpus": 1,
                "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": statistics.mean(a + b for a, b in runs) * 1e3,
                "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": config,
                "cpu_baseline": cpu,
                "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return

    import torch
    if world > 1:
        torch.distributed.init_process_group("nccl", device_id=torch.device(f"cuda:{local}"))
    device = f"cuda:{local}"
    res = run_seed(args, rank, world, device)

    total_s, value = aggregate(res["total_bytes"], res["total_ms"] / 1e3, world, device)
    if rank == 0:
        cpu = oracle_sample(wl, args.cpu_reps) if world == 1 and args.cpu_reps > 0 else None
        K = args.steps
        kv_, kd_ = res["kern"]["verify"], res["kern"]["draft"]
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
            "accept_us": round(1e3 * statistics.mean(res["t_accept"]), 2),
            "roofline": {"bound": "hbm",
                         "kernel": f"seed_verify_attn ({attn_kernel_name(wl)})",
                         "achieved": round(kv_["gbs"], 1), "peak": peak,
                         "unit": "GB/s", "frac": round(kv_["gbs"] / peak, 3),
                         "peak_kind": peak_kind,
                         "traffic": ncu_traffic(wl, "verify", kv_["bytes"]),
                         "bytes_per_launch": round(kv_["bytes"]),
                         "us_per_launch": round(kv_["us"], 2), "launches": kv_["launches"],
                         "us_per_launch_isolated": round(kv_["us_isolated"], 2),
                         "frac_isolated": round(kv_["gbs_isolated"] / peak, 3),
                         "timing": "K kernel-timing rounds: " + KERN_TIMING},
            "draft_attn": dict(kern_line(kd_, f"seed_draft_attn ({attn_kernel_name(wl, 'draft')})",
                                         peak),
                               traffic=ncu_traffic(wl, "draft", kd_["bytes"])),
            "gpu_launches": res["n_launches"],
            "clocks": res["clocks"],
            "cpu_baseline": cpu,
        }
        if "e2e" in res:
            line["e2e"] = res["e2e"]
        if world == 1 and not args.no_per_workload:
            line["per_workload"] = per_workload(args, rank, device, peak)
        print(json.dumps(line))
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
