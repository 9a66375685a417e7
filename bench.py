"""Benchmark of the E2S-Pruner pruning decision on GB300.

One step = the whole hot path for one batch of the LLaVA-1.5-7B workload
(35 system + 24x24 visual + 64 text tokens, 3 evidence layers, 32 heads x
128, batch 1, K = 64): e2s_score (tcgen05, causal-prefix probability),
e2s_fuse, e2s_select and e2s_compact of the hidden states and every evidence
layer's K and V.  Inputs are seeded synthetic bf16 tensors (no dataset or
checkpoint is available); L2 is flushed (256 MiB write) before every step.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line.  --impl reference times the float64 CPU oracle on the
same workload (a bounded sample of steps).  Under torchrun every rank runs an
independent replica (images are independent: no collective on the data path).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "pruning decisions/sec (images/s) at LLaVA-1.5 shape, K=64; % of HBM roofline"
UNIT = "images/s"
CFG_ID, KEEP = 1, 64
WORKLOAD = "llava-1.5-7b decision+compaction, batch 1, 35+576(24x24)+64 tokens, 3 layers, " \
           "32x128 MHA, K=64 (configs[1])"

# ncu dram__bytes_read.sum + dram__bytes_write.sum of one score-kernel launch on this
# workload, and the sha256 (first 16 hex) of csrc/score_tc.cu when it was captured.
NCU_TRAFFIC = {"score_tc_kernel": None}


def _src_hash(name: str) -> str:
    p = os.path.join(ROOT, "paper_2608_23253_gb300", "csrc", name)
    return hashlib.sha256(open(p, "rb").read()).hexdigest()[:16]


def measured_peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except OSError:
        return None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx = float(parts[1])
            except ValueError:
                continue
            for nm, val in zip(names, parts[4:8]):
                if val.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


def oracle_step(inp, params):
    from oracle import e2s_oracle as orc
    ref = orc.decide(inp.q_text, inp.k, inp.n_sys, inp.n_vis, inp.n_text, inp.grid_h, inp.grid_w,
                     inp.keep, H_kv=inp.spec.H_kv, params=params)
    orc.compact(inp.hidden, inp.n_sys, inp.n_vis, inp.n_text, ref["keep"])
    for l in range(inp.spec.L):
        orc.compact(inp.k[l], inp.n_sys, inp.n_vis, inp.n_text, ref["keep"])
        orc.compact(inp.v[l], inp.n_sys, inp.n_vis, inp.n_text, ref["keep"])
    return ref


def cpu_oracle_rate(seconds: float = 12.0, threads: int = 1):
    """Times the oracle (decision + compaction) on the host in a fresh process."""
    code = (
        "import sys,time,json;sys.path.insert(0,%r);import bench;"
        "from paper_2608_23253_gb300 import synth;"
        "from oracle import e2s_oracle as orc;"
        "inp=synth.make_inputs(synth.config_spec(%d,keep=%d));p=orc.Params();"
        "bench.oracle_step(inp,p);n=0;t=time.perf_counter()\n"
        "while True:\n bench.oracle_step(inp,p);n+=1\n"
        " if time.perf_counter()-t>%f: break\n"
        "print(json.dumps({'images':n,'seconds':time.perf_counter()-t}))"
    ) % (ROOT, CFG_ID, KEEP, seconds)
    env = dict(os.environ)
    for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        env[v] = str(threads)
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env,
                       timeout=600)
    if r.returncode != 0:
        raise RuntimeError("oracle timing failed: " + r.stderr[-2000:])
    out = json.loads(r.stdout.strip().splitlines()[-1])
    return out["images"] / out["seconds"], out


def dist_setup(n_gpus: int):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world != n_gpus:
        raise SystemExit(f"--gpus {n_gpus} but WORLD_SIZE={world}")
    return world, rank, local


def run_reference(args, world, rank):
    if rank != 0:
        return
    rate, info = cpu_oracle_rate(seconds=max(3.0, 3.0 * args.steps / 10.0 + 2.0))
    line = {
        "impl": "reference", "metric": METRIC, "value": rate, "unit": UNIT, "n_gpus": args.gpus,
        "steps": info["images"], "warmup": 1, "ms_per_step": 1e3 / rate,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": WORKLOAD},
        "cpu_baseline": {"value": rate, "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": f"{info['images']} decisions+compactions of one config-1 image "
                                   f"in {info['seconds']:.1f} s, 1 thread"},
        "e2e": {"value": rate, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_ours(args, world, rank, local):
    import torch

    from paper_2608_23253_gb300 import e2s, synth
    from paper_2608_23253_gb300.decision import Batch, Decision, bf16_tensor

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    inp = synth.make_inputs(synth.config_spec(CFG_ID, keep=KEEP), with_payload=True)
    s = inp.spec
    batch = Batch.from_inputs(inp, device=dev)
    dec = Decision(batch, inp.keep, e2s.params())
    q = bf16_tensor(inp.q_text, dev)
    k = bf16_tensor(inp.k, dev)
    v = bf16_tensor(inp.v, dev)
    hid = bf16_tensor(inp.hidden, dev)
    kv_rows = s.H_kv * s.d
    src = [hid] + [k[l].view(batch.sum_T, kv_rows) for l in range(s.L)] + \
          [v[l].view(batch.sum_T, kv_rows) for l in range(s.L)]
    R = dec.out_rows()
    dst = [torch.empty((R, t.shape[1]), dtype=t.dtype, device=dev) for t in src]
    pos = torch.empty(R, dtype=torch.int32, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)

    stream = torch.cuda.Stream(device=dev)
    graphs = {}
    with torch.cuda.stream(stream):
        # eager warm-up (also sets kernel attributes outside capture)
        dec.score(q, k, stream=stream)
        dec.fuse(stream=stream)
        dec.select(stream=stream)
        dec.compact(src, dst, pos, stream=stream)
        stream.synchronize()
        e2s.check(dec.status(stream), "device status after warm-up")
        for name, fn in (("score", lambda: dec.score(q, k, stream=stream)),
                         ("fuse_select", lambda: (dec.fuse(stream=stream),
                                                  dec.select(stream=stream))),
                         ("compact", lambda: dec.compact(src, dst, pos, stream=stream))):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                fn()
            graphs[name] = g
    launches_per_step = 1 + 2 + 1 + 1
    stages = list(graphs)

    def step(evs):
        flush.zero_()
        evs[0].record(stream)
        for i, name in enumerate(stages):
            graphs[name].replay()
            evs[i + 1].record(stream)

    def new_events():
        return [torch.cuda.Event(enable_timing=True) for _ in range(len(stages) + 1)]

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step(new_events())
        stream.synchronize()
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()
        records = []
        with ClockSampler(local) as clocks:
            t_wall = time.perf_counter()
            for _ in range(args.steps):
                evs = new_events()
                step(evs)
                records.append(evs)
            stream.synchronize()
            torch.cuda.synchronize()
            t_wall = time.perf_counter() - t_wall
        if world > 1:
            torch.distributed.barrier()
        e2s.check(dec.status(stream), "device status after timing")
        stage_ms = {name: [ev[i].elapsed_time(ev[i + 1]) for ev in records]
                    for i, name in enumerate(stages)}
        step_ms = [ev[0].elapsed_time(ev[-1]) for ev in records]

        # end to end through the public API, host buffers in pinned memory
        host_in = [torch.from_numpy(x.view(np.int16)).pin_memory()
                   for x in (inp.q_text, inp.k, inp.v, inp.hidden)]
        dev_in = [q, k, v, hid]
        h2d = sum(t.numel() * t.element_size() for t in host_in)
        out_keep = torch.empty(dec.keep_idx.numel(), dtype=torch.int32).pin_memory()
        out_pos = torch.empty(R, dtype=torch.int32).pin_memory()
        d2h = out_keep.numel() * 4 + out_pos.numel() * 4
        e2e_ms = []
        for it in range(args.warmup + args.steps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for hsrc, ddst in zip(host_in, dev_in):
                ddst.view(torch.int16).view(-1).copy_(hsrc.view(-1), non_blocking=True)
            for name in stages:
                graphs[name].replay()
            out_keep.copy_(dec.keep_idx, non_blocking=True)
            out_pos.copy_(pos, non_blocking=True)
            e1.record(stream)
            e1.synchronize()
            if it >= args.warmup:
                e2e_ms.append(e0.elapsed_time(e1))

    total_ms = sum(step_ms)
    if world > 1:
        t = torch.tensor([total_ms, sum(e2e_ms)], device=dev)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        total_ms, e2e_total = float(t[0]), float(t[1])
    else:
        e2e_total = sum(e2e_ms)
    images = batch.B * args.steps * world
    value = images / (total_ms * 1e-3)

    # roofline of the dominant kernel
    L, H, Hkv, d = s.L, s.H, s.H_kv, s.d
    bytes_stage = {
        "score": L * batch.sum_T * Hkv * d * 2 + L * batch.sum_text * H * d * 2
                 + L * H * batch.sum_vis * 4,
        "fuse_select": L * H * batch.sum_vis * 4 * 3 + L * batch.sum_vis * 16
                       + batch.sum_vis * (16 + 4 + 4) + dec.sum_keep * 4,
        "compact": 2 * R * sum(t.stride(0) * t.element_size() for t in src) + R * 4,
    }
    mean_ms = {n: statistics.mean(v_) for n, v_ in stage_ms.items()}
    dom = max(mean_ms, key=mean_ms.get)
    peaks = measured_peaks()
    peak, peak_src = (peaks["hbm_gbs"], "measured") if peaks else (6800.0, "fallback")
    achieved = bytes_stage[dom] / (mean_ms[dom] * 1e-3) / 1e9
    traffic = None
    key = "score_tc_kernel" if dom == "score" else None
    if key and NCU_TRAFFIC.get(key) and NCU_TRAFFIC[key]["src"] == _src_hash("score_tc.cu"):
        traffic = NCU_TRAFFIC[key]["bytes"]
    clk = clocks.summary()
    if rank != 0:
        return
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": statistics.mean(step_ms),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": WORKLOAD, "global_batch": batch.B * world, "seq_len": batch.sum_T,
                   "n_vis": int(inp.n_vis[0]), "n_text": int(inp.n_text[0]), "layers": L,
                   "keep": KEEP, "score_mode": "causal_prob", "norm": "renorm",
                   "parallelism": f"replicas{world}",
                   "l2": "flushed before every step (256 MiB write)"},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic, "kernel": dom,
                     "peak_source": f"{peak_src} hbm_gbs",
                     "algorithmic_bytes": bytes_stage[dom]},
        "stages": {n: {"us": mean_ms[n] * 1e3, "algorithmic_bytes": bytes_stage[n],
                       "GB/s": bytes_stage[n] / (mean_ms[n] * 1e-3) / 1e9,
                       "frac_hbm": bytes_stage[n] / (mean_ms[n] * 1e-3) / 1e9 / peak}
                   for n in stages},
        "gpu_launches": launches_per_step * args.steps,
        "e2e": {"value": images / (e2e_total * 1e-3), "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "clocks": clk,
        "wall_s_timed_region": t_wall,
    }
    if world == 1 and not args.no_cpu_baseline:
        rate, info = cpu_oracle_rate()
        line["cpu_baseline"] = {"value": rate, "unit": UNIT, "cores": 1, "kind": "oracle",
                                "sample": f"{info['images']} decisions+compactions of one "
                                          f"config-1 image in {info['seconds']:.1f} s, 1 thread"}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    if args.warmup < 3:
        raise SystemExit("--warmup must be >= 3")
    world, rank, local = dist_setup(args.gpus)
    if args.impl == "reference":
        run_reference(args, world, rank)
    else:
        run_ours(args, world, rank, local)


if __name__ == "__main__":
    main()
