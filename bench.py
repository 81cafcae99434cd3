"""Throughput of the ChronoStitch composition hot path on GB300.

One step = one composition query: re-base all layers' stored keys, score the
candidates, select the top rho, repair-attend the selected rows over the
composed cache (three kernel launches: re-base and score are one).  The metric
is composed visual tokens per second: T_vis / step time.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

Prints one JSON line (rank 0).  The default workload is the largest single-GPU
configuration, qwen3b_64x1024_r15 (3B shape, 64 chunks x 1024 tokens, rho 0.15).
--impl reference times the CPU oracle on the host cores instead: each step is a
bounded sample of the workload (one layer of re-base, score and select over all
candidates, attention of a seeded sample of rows), scaled to the full step by the
work it stands for.  With N > 1 (torchrun) every rank runs an independent replica
of the query; the reference arm runs on rank 0 only.
"""
from __future__ import annotations

import os

# the oracle is timed on explicit worker processes: one BLAS / OpenMP thread each
for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, "1")

import argparse
import json
import platform
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
DATA = ("synthetic: seeded N(0,1) stored keys/values/queries, lognormal fresh-key deviation, "
        "Qwen2.5-VL-shaped")


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
    """(dram bytes per launch, source note) from a committed ncu summary, or (None, why)."""
    path = os.path.join(ROOT, "profiles", kernel_file)
    if not os.path.exists(path):
        return None, f"no committed ncu summary profiles/{kernel_file}"
    for line in open(path):
        if line.startswith("dram_bytes_per_launch_full_workload:"):
            try:
                v = float(line.split(":", 1)[1].split()[0])
            except ValueError:
                break
            return v, (f"profiles/{kernel_file}: dram__bytes_read.sum + dram__bytes_write.sum "
                       "of an ncu capture (not measured by this run)")
    return None, f"profiles/{kernel_file} holds no per-launch DRAM figure"


def cpu_model() -> str:
    """The host CPU's model name (lscpu), else what the platform module knows."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    return platform.processor() or platform.machine()


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


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


def numa_nodes() -> int:
    """NUMA nodes the host exposes (1 if unknown)."""
    try:
        return max(1, len([d for d in os.listdir("/sys/devices/system/node")
                           if d.startswith("node") and d[4:].isdigit()]))
    except OSError:
        return 1


def host_link_rates(h_in, d_in, h_out, d_out, stream) -> dict:
    """Host<->device copy rates of the e2e buffers on their own (pinned host memory):
    one host-to-device copy of the stored keys and one device-to-host copy of the output,
    each timed with CUDA events, best of 3."""
    def rate(dst, src):
        best = None
        for _ in range(3):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            dst.copy_(src, non_blocking=True)
            e1.record(stream)
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1)
            best = ms if best is None else min(best, ms)
        return round(src.numel() * src.element_size() / (best / 1e3) / 1e9, 1)
    return {"h2d_gbs": rate(d_in, h_in), "d2h_gbs": rate(h_out, d_out),
            "h2d_bytes": h_in.numel() * h_in.element_size(),
            "d2h_bytes": d_out.numel() * d_out.element_size(),
            "pinned": bool(h_in.is_pinned()), "host_numa_nodes": numa_nodes(),
            "placement": "pinned with cudaHostAlloc through torch on the process's NUMA node "
                         "(the host exposes the node count given)"}


def config_of(w, ws: int) -> dict:
    """The workload description both arms print (the same dict for the same run)."""
    return {"workload": w.name, "layers": w.n_layers, "chunks": w.n_chunks,
            "tokens_per_chunk": w.chunk_tokens, "T": w.T, "T_vis": w.t_vis,
            "q_heads": w.hq, "kv_heads": w.hkv, "rho": w.rho_bp / 1e4, "k": w.k,
            "suffix_rows": w.suffix,
            "l2": "inputs larger than L2; also flushed between steps (256 MB written, then "
                  "another 256 MB read, so L2 holds no dirty lines) with the stored keys "
                  "restored, untimed",
            "parallelism": f"{ws} independent replica(s)"}


# ----------------------------------------------------------------------------- GPU arm

def _event_mean_ms(run, flush_l2, stream, reps: int) -> float:
    """Mean device time of run() over reps calls, L2 flushed (untimed) before each."""
    ms = []
    for _ in range(reps):
        flush_l2()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        run()
        e1.record(stream)
        torch.cuda.synchronize()
        ms.append(e0.elapsed_time(e1))
    return float(np.mean(ms))


def measure_next_rows(w, x, q, flush_l2, stream, pk, reps: int = 5) -> dict:
    """The two next-step kernels of the query outside the timed step, on the same workload:

    * scatter-back (Sec. 2): fresh K and V rows of the k repaired tokens, all layers, written
      into the cache at the step's selected positions (two cs_scatter_rows calls); bytes =
      the fresh rows read + the cache rows written, for K and V;
    * shallow recompute (Eq. 6, 2 c_a |C| T): every candidate as a query row over the first
      two layers (cs_repair_attention through ComposedQuery.shallow_recompute); FLOP as for
      the repair attention over the candidates' positions.

    Inputs are seeded random draws of the right shapes; V's overwritten rows are restored
    afterwards (K is restored by every step)."""
    import paper_2607_19547_gb300 as cs

    dev = x["k"].device
    g = torch.Generator(device=dev).manual_seed(20260)
    L, k, b = w.n_layers, w.k, w.elem_bytes
    idx = q.qpos[:k]
    rows = lambda: torch.randn((L, k, w.hkv, w.head_dim), generator=g, device=dev).to(w.torch_dtype)  # noqa: E731
    k_rows, v_rows = rows(), rows()
    v_saved = x["v"][:, idx.long()].clone()

    def scatter():
        cs.cs_scatter_rows(x["k"], k_rows, idx)
        cs.cs_scatter_rows(x["v"], v_rows, idx)

    scatter()
    torch.cuda.synchronize()
    sc_ms = _event_mean_ms(scatter, flush_l2, stream, reps)
    x["v"][:, idx.long()] = v_saved
    sc_bytes = 2.0 * 2.0 * L * k * w.hkv * w.head_dim * b + 2.0 * 4.0 * k
    sc_gbs = sc_bytes / (sc_ms / 1e3) / 1e9
    out = {"scatter_back": {"us": round(sc_ms * 1e3, 2), "bytes": sc_bytes,
                            "gbs": round(sc_gbs, 1), "frac_hbm": round(sc_gbs / pk["hbm_gbs"], 4),
                            "launches": 2, "rows": f"{L} layers x {k} rows, K and V",
                            "timed": f"event around the two calls, mean of {reps}, L2 flushed"}}
    nl = min(2, L)
    q_cand = torch.randn((nl, w.n_cand, w.hq, w.head_dim), generator=g, device=dev).to(w.torch_dtype)
    o_cand = torch.empty_like(q_cand)
    run = lambda: q.shallow_recompute(q_cand, x["k"], x["v"], out=o_cand)   # noqa: E731
    run()
    torch.cuda.synchronize()
    sr_reps = max(2, reps // 2)
    sr_ms = _event_mean_ms(run, flush_l2, stream, sr_reps)
    cs.cs_sync_status()
    pos = np.arange(w.cand0, w.cand0 + w.n_cand, dtype=np.int64)
    flop = 4.0 * w.head_dim * w.hq * nl * float(np.sum(pos + 1))
    tflops = flop / (sr_ms / 1e3) / 1e12
    out["shallow_recompute"] = {
        "us": round(sr_ms * 1e3, 2), "flop": flop, "tflops": round(tflops, 2),
        "frac_tensor": round(tflops / pk["bf16_tflops"], 4) if w.dtype == "bf16" else None,
        "rows": f"{w.n_cand} candidates x {nl} layers",
        "kernel": "attn_tc_kernel" if w.dtype == "bf16" else "attn_f32_kernel",
        "timed": f"event around the call, mean of {sr_reps}, L2 flushed"}
    return out


def run_gpu(args, w, ws, rank, local):
    import paper_2607_19547_gb300 as cs
    from paper_2607_19547_gb300.pipeline import (ComposedQuery, GraphedQuery, PipelinedQuery,
                                                 QueryShape, QueryStream, compose_from_host)

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
    # L2 flush (129 MB of L2): write 256 MB, then read another 256 MB, so the timed kernels
    # start from a cold L2 holding no dirty lines (writing back the flush's own dirty lines
    # would otherwise land inside the timed region)
    flush_w = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)
    flush_r = torch.zeros(64 * 1024 * 1024, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def flush_l2():
        flush_w.zero_()
        flush_r.amax()

    def restore_and_flush():
        # untimed: restore the stored cache (the step re-bases it in place) and flush L2
        x["k"].copy_(pristine)
        flush_l2()

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

    # the library fuses re-base and score into one launch (any head count, bf16 or fp32)
    fused = not args.no_fuse
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
    sel_bytes = 4.0 * w.n_cand + 4.0 * w.k
    attn_tflops = attn_flop / (mean[1] / 1e3) / 1e12
    traffic, traffic_src = profiled_traffic(f"attn_tc_{w.name}.md")
    if args.layers is not None:
        traffic, traffic_src = None, "profiling slice: no summary for this layer count"
    roofline = {"bound": "tensor", "achieved": round(attn_tflops, 2), "peak": pk["bf16_tflops"],
                "unit": "TFLOP/s", "frac": round(attn_tflops / pk["bf16_tflops"], 4),
                "traffic": traffic, "traffic_source": traffic_src, "kernel": "attn_tc_kernel",
                "peak_source": pk["source"] + " (burst)",
                "frac_of_sustained": (round(attn_tflops / pk["bf16_tflops_sustained"], 4)
                                      if pk.get("bf16_tflops_sustained") else None),
                "algorithmic": "FLOP = 4 * 128 * Hq * L * sum(qpos + 1) over the step's selection"}
    if w.dtype == "f32":
        roofline.update({"bound": "alu", "kernel": "attn_f32_kernel", "peak": None, "frac": None})
    rs_bytes = W.rebase_score_bytes(w, fused)
    kernels = {
        "rebase_score": {"us": round(seq[0] * 1e3, 2), "bytes": rs_bytes,
                         "gbs": round(rs_bytes / (seq[0] / 1e3) / 1e9, 1),
                         "frac_hbm": round(rs_bytes / (seq[0] / 1e3) / 1e9 / pk["hbm_gbs"], 4),
                         "launches": 1 if fused else 2,
                         "bytes_counted": ("re-base r+w of every moved key row; score: fresh rows "
                                           "read + fp32 written" + (" (the re-based rows are "
                                           "read back from L2 inside the launch)" if fused else
                                           " + re-based rows read again")),
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
    config = config_of(w, ws)
    if args.layers is not None:
        config["profiling_slice"] = f"first {w.n_layers} layers only (--layers)"
    next_rows = None if args.no_next_rows else measure_next_rows(w, x, q, flush_l2, stream, pk)

    line = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": w.dtype, "data": DATA, "config": config,
        "roofline": roofline, "kernels": kernels,
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clk,
        "wall_s_timed_loop": round(wall, 4),
    }
    if next_rows is not None:
        line["next_rows"] = next_rows
    if args.no_e2e:
        return line, x, pristine

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
            flush_l2()
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
    del pipelined, graphed
    # a stream of queries with up to four in flight (per slot: device buffers and captured
    # graphs of the uploads, the launches and the downloads of each layer part, on shared
    # upload, compute and download streams; four slots let the uploads run up to three queries
    # ahead, so a stall of the shared host link is absorbed): e2e_steps queries in one timed
    # region, every query copying its own inputs in and its result out
    n_slots = 4
    qstream = QueryStream(shape, w.torch_dtype, host, pl, pg, n_slots=n_slots)
    qstream.run(n_slots)
    torch.cuda.synchronize()
    flush_l2()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    s_h2d, s_d2h = qstream.run(e2e_steps)
    e1.record(stream)
    torch.cuda.synchronize()
    stream_mean = e0.elapsed_time(e1) / e2e_steps
    assert (s_h2d, s_d2h) == (h2d, d2h)
    del qstream
    torch.cuda.empty_cache()
    cs.cs_sync_status()
    link = host_link_rates(host["k"], x["k"], out_host["o"], q.out, stream)
    e2e_mean = max_over_ranks(stream_mean, dev)
    pipe_mean = max_over_ranks(pipe_mean, dev)
    graph_mean = max_over_ranks(graph_mean, dev)
    eager_mean = max_over_ranks(eager_mean, dev)
    line["e2e"] = {"value": round(replica_throughput(w.t_vis, e2e_mean, ws), 1), "unit": UNIT,
                   "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                   "ms_per_step": round(e2e_mean, 4),
                   "steps": e2e_steps,
                   "h2d_gbs_effective": round(h2d / (e2e_mean / 1e3) / 1e9, 1),
                   "path": f"QueryStream.run: the steps as a stream of queries, {n_slots} slots "
                           "(uploads, launches and downloads of each layer part of a query as "
                           "graphs on shared upload, compute and download streams), one timed "
                           "region",
                   "single_query": {
                       "value": round(replica_throughput(w.t_vis, pipe_mean, ws), 1),
                       "ms_per_step": round(pipe_mean, 4), "ms_min_median_max": pipe_spread,
                       "path": "PipelinedQuery.replay per step (copies and kernels overlapped "
                               "by layer group, one CUDA graph), events around each step"},
                   "graph_value": round(replica_throughput(w.t_vis, graph_mean, ws), 1),
                   "eager_value": round(replica_throughput(w.t_vis, eager_mean, ws), 1),
                   "host_link": link}
    # the CPU-baseline leg reads the GPU arm's own inputs (not its results)
    return line, x, pristine


# ----------------------------------------------------------------------------- oracle

# Oracle worker state: the sampled inputs as .npy files in a scratch directory, opened
# as memory maps by the parent and by every worker process of the pool.
_ORC = {}


def _oracle_init(workdir: str, meta: dict):
    """Opens the sample's arrays (in the parent for the 1-process run, in each worker)."""
    import oracle as O
    _ORC.clear()
    _ORC.update(meta)
    _ORC["O"] = O
    ld = lambda name, mode="r": np.load(os.path.join(workdir, name + ".npy"), mmap_mode=mode)  # noqa: E731
    for l in meta["layers"]:
        _ORC[("k", l)] = ld(f"k{l}")
        _ORC[("v", l)] = ld(f"v{l}")
        _ORC[("q", l)] = ld(f"q{l}")
    _ORC["fresh32"] = ld("fresh32")
    _ORC["loc"] = ld("loc")
    _ORC["glo"] = ld("glo")
    _ORC["dir"] = workdir


def _kr(l, sid):
    """Re-based keys of layer l for step sid: a new file every step (rewriting pages of a
    file under writeback would stall the writer)."""
    key = ("kr", l, sid)
    if key not in _ORC:
        for old in [k for k in _ORC if isinstance(k, tuple) and k[0] == "kr"]:
            del _ORC[old]
        _ORC[key] = np.load(os.path.join(_ORC["dir"], f"kr{l}_{sid}.npy"), mmap_mode="r+")
    return _ORC[key]


def _oracle_rebase(task):
    l, sid, a, b = task
    O = _ORC["O"]
    out = O.rebase(np.asarray(_ORC[("k", l)][a:b])[None], _ORC["loc"][a:b], _ORC["glo"][a:b],
                   _ORC["dtype"])[0][0]
    _kr(l, sid)[a:b] = out
    return b - a


def _oracle_score(task):
    sid, a, b = task
    c0, sl = _ORC["cand0"], _ORC["score_layer"]
    kc = np.asarray(_kr(sl, sid)[c0 + a:c0 + b]).astype(np.float32)
    return _ORC["O"].score_f32_canonical(np.asarray(_ORC["fresh32"][a:b]), kc)


def _oracle_attention(task):
    l, sid, rows, qpos = task
    _ORC["O"].repair_attention(_ORC[("q", l)][None], _kr(l, sid)[None], _ORC[("v", l)][None],
                               qpos, rows=rows)
    return len(rows)


class OracleSample:
    """The oracle's composition query on a bounded sample of one workload.

    One sampled step: re-base of the layers in `layers` (all tokens), score and
    selection over every candidate (on the re-based score layer), and repair
    attention of a seeded sample of query rows at those layers.  The full step is
    estimated by scaling the re-base by L / len(layers) and the attention by
    (L / len(layers)) * sum over all rows of (qpos + 1) / the same sum over the
    sampled rows (its work is linear in the visible keys).  With a process pool the
    work is split by token range, candidate range and row subset over worker
    processes (spawned, so none inherits a CUDA context); the oracle's functions
    run unchanged on each part.
    """

    def __init__(self, w, k, v, q, fresh_local, layers):
        import shutil
        import tempfile

        import oracle as O
        self.w = w
        self.layers = list(layers)
        if w.score_layer not in self.layers:
            raise ValueError("the sampled layers must include the score layer")
        # a memory-backed directory when it has room for the sample, else the temp directory
        need = 8 * (3 * k[self.layers[0]].size + q[self.layers[0]].size) * len(self.layers)
        base = None
        if os.path.isdir("/dev/shm"):
            try:
                if shutil.disk_usage("/dev/shm").free > 2 * need:
                    base = "/dev/shm"
            except OSError:
                pass
        self.dir = tempfile.mkdtemp(prefix="cs_oracle_", dir=base)
        self.sid = 0
        loc, glo = W.coordinates(w)
        cand = slice(w.cand0, w.cand0 + w.n_cand)
        # set-up, untimed: the fresh keys at global coordinates (the shallow recompute's output)
        fresh = O.rebase(fresh_local[None], loc[cand], glo[cand], w.dtype)[0][0]
        sv = lambda name, a: np.save(os.path.join(self.dir, name + ".npy"), a)  # noqa: E731
        for l in self.layers:
            sv(f"k{l}", k[l])
            sv(f"v{l}", v[l])
            sv(f"q{l}", q[l])
        self.kshape = k[self.layers[0]].shape
        sv("fresh32", fresh.astype(np.float32))
        sv("loc", loc)
        sv("glo", glo)
        self.meta = {"layers": self.layers, "dtype": w.dtype, "cand0": w.cand0,
                     "score_layer": w.score_layer}
        self.pool = None
        self.workers = 1

    @classmethod
    def from_tensors(cls, w, x, layers):
        """Inputs copied from the tensors of make_inputs (layer i of x = layers[i])."""
        f = lambda t: t.detach().float().cpu().numpy().astype(np.float64)   # noqa: E731
        return cls(w, {l: f(x["k"][i]) for i, l in enumerate(layers)},
                   {l: f(x["v"][i]) for i, l in enumerate(layers)},
                   {l: f(x["q"][i]) for i, l in enumerate(layers)}, f(x["k_fresh_local"]), layers)

    def start(self, workers: int):
        """Runs the next steps on `workers` processes (1: in this process)."""
        import multiprocessing as mp
        self.stop()
        self.workers = workers
        if workers > 1:
            self.pool = mp.get_context("spawn").Pool(workers, initializer=_oracle_init,
                                                     initargs=(self.dir, self.meta))
        _oracle_init(self.dir, self.meta)

    def stop(self):
        if self.pool is not None:
            self.pool.close()
            self.pool.join()
            self.pool = None

    def close(self):
        import shutil
        self.stop()
        _ORC.clear()
        shutil.rmtree(self.dir, ignore_errors=True)

    @staticmethod
    def _split(n, parts):
        edges = np.linspace(0, n, max(1, min(parts, n)) + 1).astype(int)
        return [(int(a), int(b)) for a, b in zip(edges[:-1], edges[1:]) if b > a]

    def _map(self, fn, items):
        if self.pool is None:
            return [fn(i) for i in items]
        return self.pool.map(fn, items, chunksize=1)

    def step(self, n_rows: int, row_seed: int):
        w, p = self.w, self.workers
        sid = self.sid = self.sid + 1
        for l in self.layers:   # untimed: this step's output files (the previous step's go)
            np.lib.format.open_memmap(os.path.join(self.dir, f"kr{l}_{sid}.npy"), mode="w+",
                                      dtype=np.float64, shape=self.kshape).flush()
            old = os.path.join(self.dir, f"kr{l}_{sid - 1}.npy")
            if os.path.exists(old):
                os.unlink(old)
        t = {}
        t0 = time.perf_counter()
        self._map(_oracle_rebase, [(l, sid, a, b) for l in self.layers
                                   for a, b in self._split(w.T, p)])
        t["rebase"] = time.perf_counter() - t0
        t0 = time.perf_counter()
        parts = self._map(_oracle_score, [(sid, a, b) for a, b in self._split(w.n_cand, p)])
        score = np.concatenate(parts) if parts else np.zeros(0, np.float32)
        t["score"] = time.perf_counter() - t0
        t0 = time.perf_counter()
        sel = _ORC["O"].select_topk(score, w.k, w.cand0)
        qpos = np.concatenate([sel, np.arange(w.T - w.suffix, w.T)]).astype(np.int32)
        t["select"] = time.perf_counter() - t0
        rows = W.sample_rows(w.M, n_rows, seed=row_seed)
        # interleaved row subsets: each worker gets early and late rows alike
        subsets = [rows[i::p] for i in range(min(p, len(rows)))]
        t0 = time.perf_counter()
        self._map(_oracle_attention, [(l, sid, r, qpos) for l in self.layers for r in subsets])
        t["attention"] = time.perf_counter() - t0
        lay = w.n_layers / len(self.layers)
        vis_all = float(np.sum(qpos.astype(np.float64) + 1.0))
        vis_rows = float(np.sum(qpos[rows].astype(np.float64) + 1.0))
        attn_scale = lay * vis_all / vis_rows if len(rows) else 0.0
        t["sampled_s"] = t["rebase"] + t["score"] + t["select"] + t["attention"]
        t["full_step_s_est"] = (lay * t["rebase"] + t["score"] + t["select"]
                                + attn_scale * t["attention"])
        t["rows"] = int(len(rows))
        t["attn_scale"] = attn_scale
        return t

    def describe(self, n_rows: int) -> str:
        w = self.w
        return (f"re-base of layer(s) {self.layers} of {w.n_layers} (all {w.T} tokens, scaled by "
                f"{w.n_layers}/{len(self.layers)}); score and select over all {w.n_cand} "
                f"candidates (timed in full); attention of {min(n_rows, w.M)} of {w.M} query rows "
                f"(seeded, first and last included) at those layers, scaled by "
                f"{w.n_layers}/{len(self.layers)} x sum(qpos+1) over all rows / over the sampled "
                f"rows; the full-step time and the rate are extrapolated from this sample; "
                f"numpy fp64")

    def rate(self, workers: int, steps: int, n_rows: int, seed0: int = 0):
        """(tokens/s of the estimated full step, per-step timing dicts)."""
        self.start(workers)
        try:
            times = [self.step(n_rows, row_seed=seed0 + s) for s in range(steps)]
        finally:
            self.stop()
        full = float(np.mean([t["full_step_s_est"] for t in times]))
        return self.w.t_vis / full, times


def cpu_baseline(w, x, layers, n_rows):
    """The oracle on the GPU machine's host, 1 process and all cores, on the GPU arm's own inputs."""
    sample = OracleSample.from_tensors(w, x, layers)
    cores = host_cores()
    try:
        r1, t1 = sample.rate(1, 1, n_rows)
        rn, tn = sample.rate(cores, 1, n_rows)
    finally:
        sample.close()
    return {"value": round(rn, 2), "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": "1 step; " + sample.describe(n_rows) + f"; {cores} worker processes",
            "cpu_model": cpu_model(),
            "sampled_s": round(tn[0]["sampled_s"], 3),
            "full_step_s_est": round(tn[0]["full_step_s_est"], 3),
            "value_is": "extrapolated from the sampled step",
            "single_thread": {"value": round(r1, 2), "unit": UNIT, "cores": 1,
                              "sampled_s": round(t1[0]["sampled_s"], 3),
                              "full_step_s_est": round(t1[0]["full_step_s_est"], 3)}}


def cpu_next_rows(w, k_l, v_l, n_rows: int, seed: int = 0) -> dict:
    """The oracle's scatter-back and shallow-recompute attention on the host (one process),
    on a bounded sample of the same work as `next_rows`, scaled to the full work:

    * scatter_rows of the k repaired rows into one layer of K (seeded fresh rows at the step's
      selected positions), scaled by 2 x L (K and V of every layer);
    * repair_attention of n_rows seeded candidate rows at one layer, scaled by 2 layers x
      sum(pos + 1) over all candidates / over the sampled ones.
    k_l, v_l: fp64 [T, Hkv, D], one layer of the GPU arm's stored cache."""
    import oracle as O
    rng = np.random.default_rng(seed)
    idx = np.sort(rng.choice(np.arange(w.cand0, w.cand0 + w.n_cand), w.k, replace=False))
    rows = rng.standard_normal((1, w.k, w.hkv, w.head_dim))
    t0 = time.perf_counter()
    O.scatter_rows(k_l[None], rows, idx)
    sc_s = (time.perf_counter() - t0) * 2 * w.n_layers
    pos = np.arange(w.cand0, w.cand0 + w.n_cand, dtype=np.int64)
    rsel = W.sample_rows(w.n_cand, n_rows, seed=seed + 1)
    q = rng.standard_normal((1, len(rsel), w.hq, w.head_dim))
    t0 = time.perf_counter()
    O.repair_attention(q, k_l[None], v_l[None], pos[rsel].astype(np.int32))
    nl = min(2, w.n_layers)
    sr_s = (time.perf_counter() - t0) * nl * float(np.sum(pos + 1)) / float(np.sum(pos[rsel] + 1))
    return {"cores": 1, "kind": "oracle", "value_is": "extrapolated from the sample",
            "scatter_back": {"ms_est": round(sc_s * 1e3, 3),
                             "sample": f"scatter_rows of {w.k} rows into 1 layer of K, x {2 * w.n_layers}"},
            "shallow_recompute": {"ms_est": round(sr_s * 1e3, 1),
                                  "sample": f"repair_attention of {len(rsel)} of {w.n_cand} "
                                            f"candidate rows at 1 layer, x {nl} layers x "
                                            "sum(pos+1) over all / over the sampled rows"}}


def run_reference(args, w, ws):
    """The reference arm: the oracle (the paper publishes no code) on the host cores."""
    layers = [w.score_layer]
    x = W.make_inputs(w, seed=args.seed, device="cpu", layers=layers)
    sample = OracleSample.from_tensors(w, x, layers)
    del x
    cores = host_cores()
    try:
        sample.start(cores)
        for s in range(args.warmup):
            sample.step(args.cpu_rows, row_seed=1000 + s)
        wall0 = time.perf_counter()
        times = [sample.step(args.cpu_rows, row_seed=s) for s in range(args.steps)]
        wall = time.perf_counter() - wall0
    finally:
        sample.close()
    full = float(np.mean([t["full_step_s_est"] for t in times]))
    rate = w.t_vis / full
    ms_sampled = 1e3 * float(np.mean([t["sampled_s"] for t in times]))
    desc = (f"each of the {args.steps} timed steps: " + sample.describe(args.cpu_rows)
            + f" (a new row sample per step); {cores} worker processes")
    return {"impl": "reference", "metric": METRIC, "value": round(rate, 2), "unit": UNIT,
            "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(ms_sampled, 3),
            "ms_per_step_is": "wall time of one sampled step as run (the timed region is "
                              "steps x this); value is T_vis / the estimated full-step time",
            "full_step_ms_est": round(1e3 * full, 3),
            "value_is": "extrapolated from the sampled steps (see cpu_baseline.sample)",
            "wall_s_timed_loop": round(wall, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": DATA + " (CPU generator)", "config": config_of(w, ws),
            "cpu_baseline": {"value": round(rate, 2), "unit": UNIT, "cores": cores,
                             "kind": "oracle", "sample": desc, "cpu_model": cpu_model()},
            "e2e": {"value": round(rate, 2), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default=W.BENCH_WORKLOAD, choices=sorted(W.CONFIGS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-fuse", action="store_true",
                    help="run re-base and score as two calls (the standalone score kernel), "
                         "not the fused cs_rebase_and_score launch")
    ap.add_argument("--no-e2e", action="store_true", help="skip the end-to-end (host buffer) leg")
    ap.add_argument("--no-next-rows", action="store_true",
                    help="skip the scatter-back and shallow-recompute measurements")
    ap.add_argument("--layers", type=int, default=None,
                    help="profiling aid: run only the first N layers of the workload (the line "
                         "says so; not a headline number)")
    ap.add_argument("--cpu-rows", type=int, default=256,
                    help="query rows the oracle attends per sampled step")
    args = ap.parse_args()
    w = W.CONFIGS[args.workload]
    if args.layers is not None:
        if not 1 <= args.layers <= w.n_layers:
            ap.error("--layers must be in [1, n_layers]")
        w = w.with_(n_layers=args.layers)
    ws, rank, local = _dist_env()

    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args, w, ws)), flush=True)
        return

    if ws > 1:
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local))
    line, x, pristine = run_gpu(args, w, ws, rank, local)
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        layers = [w.score_layer]
        xs = {"k": pristine[layers], "v": x["v"][layers], "q": x["q"][layers],
              "k_fresh_local": x["k_fresh_local"]}
        line["cpu_baseline"] = cpu_baseline(w, xs, layers, args.cpu_rows)
        if "next_rows" in line:
            f64 = lambda t: t.detach().float().cpu().numpy().astype(np.float64)   # noqa: E731
            line["cpu_baseline"]["next_rows"] = cpu_next_rows(w, f64(xs["k"][0]), f64(xs["v"][0]),
                                                              args.cpu_rows)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
