"""Throughput of the ChronoStitch composition hot path on GB300.

One step = one composition query: re-base all layers' stored keys, score the
candidates, select the top rho, repair-attend the selected rows over the
composed cache (four kernel launches).  The metric is composed visual tokens
per second: T_vis / step time.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

Prints one JSON line (rank 0).  --impl reference times the CPU oracle on the
host cores instead (a bounded sample of each step, scaled to the full step).
With N > 1 (torchrun) every rank runs an independent replica of the query.
"""
from __future__ import annotations

import os

# the CPU oracle is timed single-threaded: fix BLAS / OpenMP threads before numpy loads
for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, "1")

import argparse
import json
import statistics
import subprocess
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import cs_workloads as W  # noqa: E402

METRIC = "composed visual tokens/sec (rebase+score+select+repair attn); % HBM / tensor peak"
UNIT = "tokens/s"


def _dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(x: float, device) -> float:
    """The largest value of x over all ranks (x itself with a single process)."""
    if not (torch.distributed.is_available() and torch.distributed.is_initialized()):
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def replica_throughput(units_per_replica: float, ms_slowest: float, world: int) -> float:
    """Whole-job throughput of `world` independent replicas timed by the slowest one."""
    return world * units_per_replica / (ms_slowest / 1e3)


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": p["hbm_gbs"], "bf16_tflops": p["bf16_tflops"],
                "bf16_tflops_sustained": p.get("bf16_tflops_sustained"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


def profiled_traffic(kernel_file: str):
    """dram bytes per launch recorded in a committed ncu summary (profiles/<file>), else None."""
    path = os.path.join(ROOT, "profiles", kernel_file)
    if not os.path.exists(path):
        return None
    for line in open(path):
        if line.startswith("dram_bytes_per_launch_full_workload:"):
            try:
                return float(line.split(":", 1)[1].split()[0])
            except ValueError:
                return None
    return None


class ClockSampler:
    """nvidia-smi clock / throttle samples taken while the timed steps run."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None
        self.out = None

    def start(self):
        try:
            self.out = open(os.path.join("/tmp", f"cs_clocks_{os.getpid()}.csv"), "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(self.dev)], stdout=self.out, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.out.close()
        sm, smax, reasons = [], [], set()
        names = ["active", "hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                 "sw_power_cap"]
        with open(self.out.name) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax.append(float(parts[2]))
                except ValueError:
                    continue
                for n, v in zip(names[1:], parts[5:9]):
                    if v.lower().startswith("active"):
                        reasons.add(n)
        os.unlink(self.out.name)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ----------------------------------------------------------------------------- GPU arm

def run_gpu(args, w, ws, rank, local):
    import paper_2607_19547_gb300 as cs
    from paper_2607_19547_gb300.pipeline import (ComposedQuery, GraphedQuery, PipelinedQuery,
                                                 QueryShape, compose_from_host)

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    x = W.make_inputs(w, seed=args.seed, device=dev)
    loc, glo = W.coordinates(w)
    pl = torch.from_numpy(loc).to(dev)
    pg = torch.from_numpy(glo).to(dev)
    cand = slice(w.cand0, w.cand0 + w.n_cand)
    # fresh keys at global coordinates: what the shallow recompute would hand over (setup)
    fresh = torch.empty_like(x["k_fresh_local"])
    cs.cs_rebase_keys(x["k_fresh_local"][None], pl[cand].contiguous(), pg[cand].contiguous(),
                      k_out=fresh[None])
    pristine = x["k"].clone()
    shape = QueryShape(n_layers=w.n_layers, T=w.T, hq=w.hq, hkv=w.hkv, cand0=w.cand0,
                       n_cand=w.n_cand, k=w.k, suffix=w.suffix, score_layer=w.score_layer)
    q = ComposedQuery(shape, w.torch_dtype, device=dev)
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)   # > 129 MB L2
    stream = torch.cuda.current_stream(dev)

    def restore_and_flush():
        # untimed: restore the stored cache (the step re-bases it in place) and flush L2
        x["k"].copy_(pristine)
        flush.zero_()

    def rebase_and_score():
        if args.no_fuse:
            cs.cs_rebase_keys(x["k"], pl, pg, theta=w.theta, sections=w.sections)
            cs.cs_score_deviation(fresh, x["k"][w.score_layer, cand], out=q.score)
        else:
            cs.cs_rebase_and_score(x["k"], pl, pg, fresh, w.score_layer, w.cand0,
                                   score_out=q.score, theta=w.theta, sections=w.sections)

    def one_step(ev):
        """One timed step.  ev: step start, attention start, step end.  No event sits
        between re-base and selection: a timing event drains the stream (about 3 us at
        4x1024), so the first two calls' own durations come from sequential_step."""
        restore_and_flush()
        ev[0].record(stream)
        rebase_and_score()
        cs.cs_select_topk(q.score, w.k, w.cand0, out=q.qpos[:w.k])
        ev[1].record(stream)
        cs.cs_repair_attention(x["q"], x["k"], x["v"], q.qpos, out=q.out)
        ev[2].record(stream)

    def sequential_step(ev):
        """The first two calls with an event around each (for their durations)."""
        restore_and_flush()
        ev[0].record(stream)
        rebase_and_score()
        ev[1].record(stream)
        cs.cs_select_topk(q.score, w.k, w.cand0, out=q.qpos[:w.k])
        ev[2].record(stream)

    # the library fuses re-base and score into one launch for these shapes
    fused = w.dtype == "bf16" and w.hkv in (1, 2, 4) and not args.no_fuse
    launches_per_step = 3 if fused else 4
    for _ in range(args.warmup):
        one_step([torch.cuda.Event(enable_timing=True) for _ in range(3)])
    cs.cs_sync_status()
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    events = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    if ws > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    wall0 = time.perf_counter()
    for i in range(args.steps):
        one_step(events[i])
    torch.cuda.synchronize()
    wall = time.perf_counter() - wall0
    if ws > 1:
        torch.distributed.barrier()
    cs.cs_sync_status()
    time.sleep(0.2)
    clk = clocks.stop()
    per = np.array([[events[i][0].elapsed_time(events[i][1]),
                     events[i][1].elapsed_time(events[i][2])] for i in range(args.steps)])
    step_ms = per.sum(axis=1)          # ms: step start to the end of the attention
    ms_per_step = max_over_ranks(float(step_ms.mean()), dev)
    value = replica_throughput(w.t_vis, ms_per_step, ws)
    # the first two calls' own durations, from steps after the timed loop
    seq_steps = max(3, min(args.steps, 20))
    seq_ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(seq_steps)]
    for i in range(seq_steps):
        sequential_step(seq_ev[i])
    torch.cuda.synchronize()
    seq = np.array([[e[0].elapsed_time(e[1]), e[1].elapsed_time(e[2])] for e in seq_ev]).mean(axis=0)

    qpos = q.qpos.cpu().numpy()
    pk = peaks()
    attn_flop = W.attention_flops(w, qpos)
    mean = per.mean(axis=0)            # ms: re-base + score + select, attention
    rb_bytes, sc_bytes = W.rebase_bytes(w), W.score_bytes(w)
    sel_bytes = 4.0 * w.n_cand + 4.0 * w.k
    attn_tflops = attn_flop / (mean[1] / 1e3) / 1e12
    traffic = profiled_traffic(f"attn_tc_{w.name}.md")
    roofline = {"bound": "tensor", "achieved": round(attn_tflops, 2), "peak": pk["bf16_tflops"],
                "unit": "TFLOP/s", "frac": round(attn_tflops / pk["bf16_tflops"], 4),
                "traffic": traffic, "kernel": "attn_tc_kernel",
                "peak_source": pk["source"] + " (burst)"}
    if w.dtype == "f32":
        roofline.update({"bound": "alu", "kernel": "attn_f32_kernel", "peak": None, "frac": None})
    rs_bytes = rb_bytes + sc_bytes
    kernels = {
        "rebase_score": {"us": round(seq[0] * 1e3, 2), "bytes": rs_bytes,
                         "gbs": round(rs_bytes / (seq[0] / 1e3) / 1e9, 1),
                         "frac_hbm": round(rs_bytes / (seq[0] / 1e3) / 1e9 / pk["hbm_gbs"], 4),
                         "launches": 1 if fused else 2,
                         "timed": f"event around the call, {seq_steps} steps after the timed loop"},
        "select": {"us": round(seq[1] * 1e3, 2), "bytes": sel_bytes,
                   "gbs": round(sel_bytes / (seq[1] / 1e3) / 1e9, 1),
                   "timed": f"event around the call, {seq_steps} steps after the timed loop"},
        "rebase_score_select": {"us": round(mean[0] * 1e3, 2),
                                "timed": "in the timed loop, no event between the two calls"},
        "attention": {"us": round(mean[1] * 1e3, 2), "flop": attn_flop,
                      "tflops": round(attn_tflops, 2),
                      "frac_tensor": round(attn_tflops / pk["bf16_tflops"], 4),
                      "timed": "in the timed loop, events on its stream around the call"},
    }

    # ---- end to end through the public API: host buffers, copies inside the timed region
    host = {"k": pristine.cpu().pin_memory(), "v": x["v"].cpu().pin_memory(),
            "q": x["q"].cpu().pin_memory(), "k_fresh": fresh.cpu().pin_memory()}
    devb = {"k": x["k"], "v": x["v"], "q": x["q"], "k_fresh": fresh, "pos_local": pl,
            "pos_global": pg}
    out_host = {"o": torch.empty(q.out.shape, dtype=q.out.dtype).pin_memory(),
                "qpos": torch.empty(w.M, dtype=torch.int32).pin_memory()}
    e2e_steps = max(3, min(args.steps, 20))

    spread = {}

    def time_e2e(run):
        ms = []
        for _ in range(e2e_steps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            run()
            e1.record(stream)
            torch.cuda.synchronize()
            ms.append(e0.elapsed_time(e1))
        spread[run] = [round(float(v), 4) for v in (np.min(ms), np.median(ms), np.max(ms))]
        return float(np.mean(ms))

    # eager: the calls one by one from Python
    for _ in range(2):
        h2d, d2h = compose_from_host(q, host, devb, out_host)
    torch.cuda.synchronize()
    eager_mean = time_e2e(lambda: compose_from_host(q, host, devb, out_host))
    # graphed: the same query captured once (copies in, launches, copies out), one launch per query
    graphed = GraphedQuery(q, host, devb, out_host)
    graphed.replay()
    torch.cuda.synchronize()
    graph_mean = time_e2e(graphed.replay)
    # pipelined: uploads, kernels and downloads overlapped layer group by layer group, one graph
    pipelined = PipelinedQuery(q, host, devb, out_host)
    pipelined.replay()
    torch.cuda.synchronize()
    pipe_mean = time_e2e(pipelined.replay)
    pipe_spread = spread[pipelined.replay]
    cs.cs_sync_status()
    e2e_mean = max_over_ranks(pipe_mean, dev)
    graph_mean = max_over_ranks(graph_mean, dev)
    eager_mean = max_over_ranks(eager_mean, dev)
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": w.dtype,
        "data": "synthetic: seeded N(0,1) stored keys/values/queries, lognormal fresh-key "
                "deviation, Qwen2.5-VL-shaped",
        "config": {"workload": w.name, "layers": w.n_layers, "chunks": w.n_chunks,
                   "tokens_per_chunk": w.chunk_tokens, "T": w.T, "T_vis": w.t_vis,
                   "q_heads": w.hq, "kv_heads": w.hkv, "rho": w.rho_bp / 1e4, "k": w.k,
                   "suffix_rows": w.suffix,
                   "l2": "flushed between steps (256 MB write) and stored keys restored, untimed",
                   "parallelism": f"{ws} independent replica(s)"},
        "roofline": roofline,
        "kernels": kernels,
        "e2e": {"value": round(replica_throughput(w.t_vis, e2e_mean, ws), 1), "unit": UNIT,
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "ms_per_step": round(e2e_mean, 4),
                "ms_min_median_max": pipe_spread,
                "steps": e2e_steps,
                "path": "PipelinedQuery.replay (copies and kernels overlapped by layer group, "
                        "one CUDA graph)",
                "graph_value": round(replica_throughput(w.t_vis, graph_mean, ws), 1),
                "eager_value": round(replica_throughput(w.t_vis, eager_mean, ws), 1)},
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clk,
        "wall_s_timed_loop": round(wall, 4),
    }
    return line


# ----------------------------------------------------------------------------- oracle

def oracle_step(w, st, layers):
    """The oracle's composition query restricted to `layers` for re-base and attention
    (score and select always full).  Returns seconds per phase."""
    import oracle as O
    t = {}
    loc, glo = st["loc"], st["glo"]
    cand = slice(w.cand0, w.cand0 + w.n_cand)
    t0 = time.perf_counter()
    k_r = {l: O.rebase(st["k"][l][None], loc, glo, w.dtype)[0][0] for l in layers}
    t["rebase"] = time.perf_counter() - t0
    t0 = time.perf_counter()
    kc = O.rebase(st["k_score"][None], loc[cand], glo[cand], w.dtype)[0][0]
    score = O.score_f32_canonical(st["fresh"].astype(np.float32), kc.astype(np.float32))
    t["score"] = time.perf_counter() - t0
    t0 = time.perf_counter()
    sel = O.select_topk(score, w.k, w.cand0)
    qpos = np.concatenate([sel, np.arange(w.T - w.suffix, w.T)]).astype(np.int32)
    t["select"] = time.perf_counter() - t0
    t0 = time.perf_counter()
    for l in layers:
        O.repair_attention(st["q"][l][None], k_r[l][None], st["v"][l][None], qpos)
    t["attention"] = time.perf_counter() - t0
    return t


def oracle_state(w, seed, layers):
    import oracle as O
    x = W.make_inputs(w, seed=seed, device="cpu")
    loc, glo = W.coordinates(w)
    cand = slice(w.cand0, w.cand0 + w.n_cand)
    f = lambda t: t.float().numpy().astype(np.float64)   # noqa: E731
    st = {"loc": loc, "glo": glo, "k": {l: f(x["k"][l]) for l in layers},
          "v": {l: f(x["v"][l]) for l in layers}, "q": {l: f(x["q"][l]) for l in layers},
          "k_score": f(x["k"][w.score_layer, cand])}
    st["fresh"] = O.rebase(f(x["k_fresh_local"])[None], loc[cand], glo[cand], w.dtype)[0][0]
    return st


def oracle_rate(w, seed, layers, steps):
    """Composed visual tokens/s of the oracle, scaling the per-layer phases to all layers."""
    st = oracle_state(w, seed, layers)
    times = []
    for _ in range(steps):
        t = oracle_step(w, st, layers)
        scale = w.n_layers / len(layers)
        times.append(t["score"] + t["select"] + scale * (t["rebase"] + t["attention"]))
    return w.t_vis / float(np.mean(times)), times


def cpu_baseline(w, seed, layers, steps):
    rate, times = oracle_rate(w, seed, layers, steps)
    return {"value": round(rate, 2), "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"{steps} step(s); re-base and attention timed on layers {list(layers)} of "
                      f"{w.n_layers} and scaled by {w.n_layers}/{len(layers)}; score and select "
                      f"over all {w.n_cand} candidates; numpy, 1 thread",
            "seconds_per_full_step_est": round(float(np.mean(times)), 3)}


def run_reference(args, w):
    layers = [w.score_layer]
    st = oracle_state(w, args.seed, layers)
    for _ in range(args.warmup):
        oracle_step(w, st, layers)
    times = []
    for _ in range(max(1, args.steps)):
        t = oracle_step(w, st, layers)
        times.append(t["score"] + t["select"] + w.n_layers / len(layers) * (t["rebase"] + t["attention"]))
    rate = w.t_vis / float(np.mean(times))
    ms = float(np.mean(times)) * 1e3
    cb = {"value": round(rate, 2), "unit": UNIT, "cores": 1, "kind": "oracle",
          "sample": f"each step: re-base and attention of layer {layers} scaled by "
                    f"{w.n_layers}, score and select over all candidates; numpy, 1 thread"}
    return {"impl": "reference", "metric": METRIC, "value": round(rate, 2), "unit": UNIT,
            "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic, same workload as the GPU arm",
            "config": {"workload": w.name, "T": w.T, "T_vis": w.t_vis, "k": w.k},
            "cpu_baseline": cb,
            "e2e": {"value": round(rate, 2), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--workload", default=W.BENCH_WORKLOAD, choices=sorted(W.CONFIGS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-fuse", action="store_true",
                    help="run re-base and score as two calls (the standalone score kernel), "
                         "not the fused cs_rebase_and_score launch")
    ap.add_argument("--cpu-layers", type=int, default=2)
    args = ap.parse_args()
    w = W.CONFIGS[args.workload]
    ws, rank, local = _dist_env()

    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args, w)), flush=True)
        return

    if ws > 1:
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local))
    line = run_gpu(args, w, ws, rank, local)
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        layers = list(range(min(args.cpu_layers, w.n_layers)))
        line["cpu_baseline"] = cpu_baseline(w, args.seed, layers, steps=1)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
