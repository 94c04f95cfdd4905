"""Benchmark of the BRISK-DLM per-block decode tail on GB300.

A step is one fused decode-tail call (candidates + corrector + verification)
over one block of the decode-stream workload: 128 sequences, block length 32,
vocabulary 126464, width 4096, K = 8, corrector width 256, bf16 logits and
hidden states, greedy Select and verify, per-sequence verifier agreement
U(0.6, 0.98). The timed steps cycle through a pool of distinct pre-generated
blocks (each block's 2.07 GB of logits exceeds the 129 MB L2, so no flush is
needed); the anchor of each block is the last committed token of the block
before it. The metric is accepted (verified) tokens per second.

Under torchrun every rank runs its own 128 sequences (replicas: the method
has no exchange between sequences); the value is the accepted tokens of all
ranks over the slowest rank's time.

``--impl reference`` times the CPU oracle (the plain float64 statement of the
method) on a bounded sample of the same workload instead.
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

METRIC = "verified tokens/sec at 1 GB300 for decode tail; % of HBM roofline on vocab sweep"
UNIT = "accepted tokens/s"
WORKLOAD = "decode_stream"
NAMEPLATE_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
SWEEP_KERNEL_SRC = os.path.join(ROOT, "paper_2609_33390_gb300", "csrc", "sweep.cu")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "ncu_traffic.txt")


# ----------------------------------------------------------------------------- host helpers

def dist_env():
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def shard_sequences(rank: int, world: int, per_rank: int, n_seqs: int):
    """Sequence ids of one rank: ranks take consecutive groups of `per_rank` sequences of the
    stream, wrapping around its `n_seqs` sequences."""
    start = (rank * per_rank) % max(1, n_seqs)
    return [(start + j) % n_seqs for j in range(per_rank)]


def aggregate(total_tokens_local: float, elapsed_local_s: float, reduce_sum, reduce_max):
    """Whole-job throughput: tokens of every rank over the slowest rank's time."""
    tokens = reduce_sum(total_tokens_local)
    elapsed = reduce_max(elapsed_local_s)
    return tokens / elapsed, tokens, elapsed


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return FALLBACK_HBM_GBS, "fallback"


def bf16_peak_tflops() -> float:
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            return float(json.load(f)["bf16_tflops"])
    return 1900.0


def fold_flops_of(wl) -> float:
    """Algorithmic flops of the once-per-weight-set folds: P_e E_in(v) and W_c E_out(v) (k = d),
    the token shares of the gate, candidate and Init pre-activations (2S + S outputs, k = r) and
    the residual rows (S outputs, k = r), for every token v."""
    return 2.0 * wl.V * wl.r * (2 * wl.d + 4 * wl.S)


def sweep_source_hash() -> str:
    """Hash of the sweep source's code: line comments, trailing blanks and empty lines are left
    out, so that an edit of the comments alone keeps a traffic record that is still valid."""
    with open(SWEEP_KERNEL_SRC) as f:
        lines = [ln.split("//", 1)[0].rstrip() for ln in f]
    code = "\n".join(ln for ln in lines if ln)
    return hashlib.sha1(code.encode()).hexdigest()[:12]


def workload_config(wl) -> dict:
    """The workload keys of the bench line's config (the same in both arms)."""
    return {"workload": WORKLOAD, "B": wl.B, "L": wl.L, "V": wl.V, "d": wl.d, "K": wl.K,
            "r": wl.r, "input_dtype": "bf16", "select": wl.select_mode,
            "verify": wl.verify_mode, "parallelism": "replicas"}


def sweep_span_ms(q0, q1, p0, p1) -> float:
    """Milliseconds from the earlier of the two sweep launches' start events to the later of
    their end events (all offsets taken from q0, so either launch may start first)."""
    p_start = q0.elapsed_time(p0)
    return max(q0.elapsed_time(q1), q0.elapsed_time(p1)) - min(0.0, p_start)


def recorded_traffic(workload: str):
    """DRAM bytes per sweep launch from the committed ncu summary, when it was taken on the
    current sweep source (lines: kernel workload bytes_per_launch source_hash)."""
    if not os.path.exists(TRAFFIC_FILE):
        return None
    h = sweep_source_hash()
    with open(TRAFFIC_FILE) as f:
        for line in f:
            parts = line.split()
            if len(parts) >= 4 and parts[0] == "sweep" and parts[1] == workload and parts[3] == h:
                return float(parts[2])
    return None


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""
    QUERY = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.t = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (FileNotFoundError, OSError):
            self.proc = None
            return
        self.t = threading.Thread(target=self._read, daemon=True)
        self.t.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        if self.t is not None:
            self.t.join(timeout=2)

    def summary(self, t0: float, t1: float):
        rows = []
        for ts, line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 10:
                continue
            try:
                rows.append((ts, float(parts[2]), float(parts[3]), parts[5:]))
            except ValueError:
                continue
        inside = [r for r in rows if t0 <= r[0] <= t1 + 0.15]
        used = inside if inside else rows
        if not used:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no nvidia-smi samples"],
                    "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        for r in used:
            for n, v in zip(names, r[3][1:5]):
                if v.strip().lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(r[1] for r in used),
                "sm_max_mhz": max(r[2] for r in used), "reasons": sorted(reasons),
                "samples": len(used), "samples_in_timed_region": len(inside)}


# ----------------------------------------------------------------------------- CPU oracle leg

CPU_SAMPLE_SEQS = 24


def _oracle_sample_worker(spec_json: str) -> str:
    """Runs in a fresh single-threaded interpreter: generates a bounded sample of the workload on
    the CPU and times the oracle's decode tail on it."""
    spec = json.loads(spec_json)
    import numpy as np
    import torch
    torch.set_num_threads(1)
    from paper_2609_33390_gb300 import synth
    from oracle import brisk_oracle as O
    wl = synth.WORKLOADS[spec["workload"]]
    seqs = spec["seqs"]
    block = synth.make_block(wl, "cpu", seqs=seqs, block=spec["block"])
    # corrector weights (small) and on-demand embedding rows of the full vocabulary
    ws = {k: v.to(torch.float64).numpy()
          for k, v in synth.make_corrector_weights(wl, "cpu").items()}
    gen_time = [0.0]

    class Rows:
        def __init__(self, which):
            self.src = synth.EmbeddingRows(wl, which)
            self.cache = {}

        def __getitem__(self, v):
            v = int(v)
            if v not in self.cache:
                t = time.perf_counter()
                self.cache[v] = self.src[v].to(torch.float64).numpy()
                gen_time[0] += time.perf_counter() - t
            return self.cache[v]

    ws.update(E_in=Rows("E_in"), E_out=Rows("E_out"), b_g=0.0, alpha=0.0)
    params = O.params_from_arrays(ws)
    lq = block["logits_q"].to(torch.float64).numpy()
    lp = block["logits_p"].to(torch.float64).numpy()
    hid = block["hidden"].to(torch.float64).numpy()
    hc = block["h_c"].to(torch.float64).numpy()
    x0 = block["x0"].numpy()
    t0 = time.perf_counter()
    acc = 0
    for b in range(len(seqs)):
        _, _, _, _, vr = O.decode_tail_sequence(params, lambda i: lq[b, i], lambda i: lp[b, i],
                                                hid[b], hc[b], int(x0[b]), wl.K, wl.select_mode,
                                                wl.verify_mode)
        acc += vr.accepted_len
    el = time.perf_counter() - t0 - gen_time[0]
    return json.dumps({"accepted": acc, "seconds": el, "seqs": len(seqs)})


def _oracle_cmd(seqs, block, workload):
    spec = json.dumps({"workload": workload, "seqs": list(seqs), "block": block})
    return [sys.executable, "-c",
            "import sys; sys.path.insert(0, %r); import bench; print(bench._oracle_sample_worker(%r))"
            % (ROOT, spec)]


def _oracle_env():
    return dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
                CUDA_VISIBLE_DEVICES="")


def run_oracle_sample(seqs, block=0, workload=WORKLOAD):
    r = subprocess.run(_oracle_cmd(seqs, block, workload), env=_oracle_env(), capture_output=True,
                       text=True, cwd=ROOT)
    if r.returncode != 0:
        raise RuntimeError("oracle sample failed:\n" + r.stderr[-2000:])
    return json.loads(r.stdout.strip().splitlines()[-1])


def run_oracle_parallel(procs, per_proc, block=0, workload=WORKLOAD):
    """`procs` single-threaded oracle processes at once, each on its own `per_proc` sequences;
    fresh interpreters (nothing forked from this CUDA process)."""
    running = [subprocess.Popen(_oracle_cmd(range(j * per_proc, (j + 1) * per_proc), block,
                                            workload),
                                env=_oracle_env(), stdout=subprocess.PIPE, stderr=subprocess.PIPE,
                                text=True, cwd=ROOT) for j in range(procs)]
    res = []
    for pr in running:
        out, err = pr.communicate()
        if pr.returncode != 0:
            raise RuntimeError("oracle sample failed:\n" + err[-2000:])
        res.append(json.loads(out.strip().splitlines()[-1]))
    return res


def cpu_baseline_entry(seqs):
    """The oracle on the host cores: one process per core (up to 16), each timing its own
    sequences; throughput = all accepted tokens / the slowest process's oracle time."""
    cores = max(1, min(16, len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity")
                       else (os.cpu_count() or 1)))
    per = max(1, len(seqs) // 3)
    res = run_oracle_parallel(cores, per)
    acc = sum(r["accepted"] for r in res)
    secs = max(r["seconds"] for r in res)
    n = sum(r["seqs"] for r in res)
    return {"value": acc / secs, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{n} sequences x 1 block of {WORKLOAD} (L=32, V=126464, d=4096, K=8, r=256)"
                      f" over {cores} single-threaded processes, float64 numpy oracle,"
                      f" {secs:.1f} s of the slowest process"}


# ----------------------------------------------------------------------------- reference arm

def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    from paper_2609_33390_gb300 import synth
    wl = synth.WORKLOADS[WORKLOAD]
    per_step = 1
    for w in range(args.warmup):
        run_oracle_sample([w % wl.n_seqs], block=0)
    tot_acc, tot_s = 0, 0.0
    for s in range(args.steps):
        r = run_oracle_sample([(s * per_step) % wl.n_seqs], block=s % wl.n_blocks)
        tot_acc += r["accepted"]
        tot_s += r["seconds"]
    value = tot_acc / tot_s
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * tot_s / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {**workload_config(wl),
                   "sample": "each step times the oracle on one sequence of one block"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": "one sequence of the decode-stream workload per step"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


# ----------------------------------------------------------------------------- GPU arm

def run_ours(args):
    import torch
    from paper_2609_33390_gb300 import build, brisk, synth

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    build.build()
    wl = synth.WORKLOADS[WORKLOAD]
    seqs = shard_sequences(rank, world, wl.B, wl.n_seqs)

    weights = synth.make_weights(wl, dev)
    tail = brisk.DecodeTail.for_workload(wl, weights, dev)
    tail.prepare()               # the first call sets kernel attributes; time the second
    torch.cuda.synchronize()
    t = time.perf_counter()
    tail.prepare()
    torch.cuda.synchronize()
    prepare_ms = 1000.0 * (time.perf_counter() - t)
    fold_flops = fold_flops_of(wl)

    pool_n = max(1, min(args.pool, args.steps + args.warmup))
    pool = []
    for j in range(pool_n):
        blk = synth.make_block(wl, dev, seqs=seqs, block=j % wl.n_blocks)
        pool.append(blk)
    sm, vm = brisk.mode_ids(wl.select_mode, wl.verify_mode)
    nsteps = args.warmup + args.steps
    outs = [tail.alloc_outputs(full=False) for _ in range(nsteps)]
    events = [tuple(torch.cuda.Event(enable_timing=True) for _ in range(4)) for _ in range(nsteps)]
    stream = torch.cuda.current_stream()
    for evs in events:      # create the CUDA events before handing their handles over
        for e in evs:
            e.record(stream)
    torch.cuda.synchronize()

    def step(s):
        blk = pool[s % pool_n]
        x0 = blk["x0"] if s == 0 else outs[s - 1]["next_anchor"]
        tail.tail(blk, sm, vm, out=outs[s], x0=x0, events=events[s])

    sampler = ClockSampler(local if "CUDA_VISIBLE_DEVICES" not in os.environ else 0)
    sampler.start()
    time.sleep(0.3)
    for s in range(args.warmup):
        step(s)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    g0 = torch.cuda.Event(enable_timing=True)
    g1 = torch.cuda.Event(enable_timing=True)
    wall0 = time.time()
    g0.record(stream)
    h0 = time.perf_counter()
    for s in range(args.warmup, nsteps):
        step(s)
    host_enqueue_s = time.perf_counter() - h0
    g1.record(stream)
    torch.cuda.synchronize()
    wall1 = time.time()
    if world > 1:
        torch.distributed.barrier()
    time.sleep(0.25)
    sampler.stop()
    elapsed = g0.elapsed_time(g1) / 1000.0
    status = tail.device_status()
    if status != brisk.OK:
        raise RuntimeError(f"device status {brisk.status_string(status)}")

    acc = sum(int(outs[s]["accepted_len"].sum()) for s in range(args.warmup, nsteps))
    committed = sum(int((outs[s]["accepted_len"] + (outs[s]["correction"] >= 0).int()).sum())
                    for s in range(args.warmup, nsteps))
    # acceptance profile of the timed steps (Sec. 3.2 Eqs. 2-3), counted after the timed region
    acc_counts = torch.zeros(2 * wl.L, dtype=torch.int64, device=dev)
    for s in range(args.warmup, nsteps):
        brisk.acceptance_counts(outs[s]["accepted_len"], wl.L, acc_counts)
    counts_h = acc_counts.cpu().tolist()
    reach_h, accept_h = counts_h[:wl.L], counts_h[wl.L:]
    prof_a = [accept_h[i] / reach_h[i] if reach_h[i] else 0.0 for i in range(wl.L)]
    prof_tpf, _, prof_w = brisk.acceptance_weights(prof_a)
    # the ISD instantiation (App. C.1, Eq. 8), which the paper uses for FPT and the weights
    isd_tpf, _, isd_w = brisk.acceptance_weights(prof_a, *brisk.isd_costs(wl.L))
    # distillation loss of the head (App. C.3) on one block's outputs: kernel time, untimed above
    full = tail.alloc_outputs(full=True)
    tail.tail(pool[0], sm, vm, out=full)
    dl_args = (pool[0]["logits_p"], full["cand_ids"], full["cand_logprob"], full["refined"],
               full["accepted_len"])
    for _ in range(3):
        tail.distill_loss(*dl_args)
    d0, d1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    d0.record(stream)
    for _ in range(20):
        tail.distill_loss(*dl_args)
    d1.record(stream)
    torch.cuda.synchronize()
    distill_us = 1000.0 * d0.elapsed_time(d1) / 20
    # same-state replay diagnostics (App. B) over the block pool: rates and the call's time
    n_fb = n_res = n_int = n_acc = n_reg = 0
    for blk in pool:
        fl = tail.replay(blk, sm)["flags"]
        n_fb += int(((fl & 4) != 0).sum())
        n_int += int(((fl & 4) != 0).logical_and((fl & 8) != 0).sum())
        n_res += int(((fl & 16) != 0).sum())
        n_acc += int(((fl & 1) != 0).logical_and((fl & 4) == 0).sum())
        n_reg += int(((fl & 32) != 0).sum())
    d0.record(stream)
    for _ in range(5):
        tail.replay(pool[0], sm)
    d1.record(stream)
    torch.cuda.synchronize()
    replay_us = 1000.0 * d0.elapsed_time(d1) / 5
    sweep_q_ms = [events[s][0].elapsed_time(events[s][1]) for s in range(args.warmup, nsteps)]
    sweep_p_ms = [events[s][2].elapsed_time(events[s][3]) for s in range(args.warmup, nsteps)]
    # the two launches overlap (the verifier rows fill the room the proposal rows leave), so
    # the sweep's time in a step is the span from the first launch's start to the last one's end
    sweep_ms = [sweep_span_ms(*events[s]) for s in range(args.warmup, nsteps)]

    if world > 1:
        import torch.distributed as dist

        def rsum(x):
            t_ = torch.tensor([float(x)], device=dev, dtype=torch.float64)
            dist.all_reduce(t_, op=dist.ReduceOp.SUM)
            return float(t_.item())

        def rmax(x):
            t_ = torch.tensor([float(x)], device=dev, dtype=torch.float64)
            dist.all_reduce(t_, op=dist.ReduceOp.MAX)
            return float(t_.item())
    else:
        rsum = rmax = float
    value, tokens, elapsed_max = aggregate(acc, elapsed, rsum, rmax)
    committed_all = rsum(committed)

    # roofline of the dominant kernel (the vocabulary sweep)
    sweep_bytes = wl.sweep_bytes()
    mean_sweep_s = statistics.mean(sweep_ms) / 1000.0
    achieved = sweep_bytes / mean_sweep_s / 1e9
    peak, peak_src = measured_peaks()
    traffic = recorded_traffic(WORKLOAD)

    # end to end through the public API: inputs from pinned host memory every step
    e2e = run_e2e(args, tail, pool, wl, sm, vm, dev) if rank == 0 or world > 1 else None
    if world > 1 and e2e is not None:
        e2e["value"] = rsum(e2e["_tokens"]) / rmax(e2e["_seconds"])
    if e2e is not None:
        e2e.pop("_tokens", None)
        e2e.pop("_seconds", None)

    # acceptance of the timed blocks with the corrector's gate closed (base ranking), after
    # the timed region, on the same blocks and anchors
    alpha = tail.params.alpha
    tail.params.alpha = float("-inf")
    acc_off = 0
    for s in range(args.warmup, nsteps):
        blk = pool[s % pool_n]
        x0 = blk["x0"] if s == 0 else outs[s - 1]["next_anchor"]
        acc_off += int(tail.tail(blk, sm, vm, x0=x0)["accepted_len"].sum())
    tail.params.alpha = alpha

    if rank != 0:
        return 0
    graph_loop = run_graph_loop(dev)
    per_config = None if args.no_per_config else run_per_config(dev, args.per_config_steps)
    cpu = None
    if not args.no_cpu_baseline:
        cpu = cpu_baseline_entry(list(range(CPU_SAMPLE_SEQS)))
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1000.0 * elapsed_max / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic",
        "config": {**workload_config(wl),
                   "l2": f"inputs larger than L2 ({sweep_bytes / 1e9:.2f} GB of logits per step,"
                         f" {pool_n} distinct blocks cycled)",
                   "prepare_ms": round(prepare_ms, 1),
                   "prepare_tflops": round(fold_flops / (prepare_ms * 1e-3) / 1e12, 1),
                   "prepare_frac_of_bf16_peak": round(fold_flops / (prepare_ms * 1e-3) / 1e12
                                                      / bf16_peak_tflops(), 3)},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic, "peak_source": peak_src,
                     "kernel": "sweep_kernel (proposal rows + verifier rows, two overlapping "
                               "launches)",
                     "bytes_per_launch": sweep_bytes, "mean_launch_us": 1e6 * mean_sweep_s,
                     "launch_time": "span from the first launch's start to the last one's end",
                     "mean_q_launch_us": 1e3 * statistics.mean(sweep_q_ms),
                     "mean_p_launch_us": 1e3 * statistics.mean(sweep_p_ms),
                     "frac_of_nameplate_8tbs": achieved / NAMEPLATE_HBM_GBS},
        "cpu_baseline": cpu,
        "e2e": e2e,
        "gpu_launches": brisk.kernels_per_tail(tail.dims) * args.steps,
        "clocks": sampler.summary(wall0, wall1),
        "committed_tokens_per_s": committed_all / elapsed_max,
        "host_enqueue_us_per_step": 1e6 * host_enqueue_s / args.steps,
        "accepted_per_sequence_block": tokens / (wl.B * world * args.steps),
        "accepted_per_sequence_block_corrector_off": acc_off / (wl.B * args.steps),
        "acceptance_profile": {"a": [round(x, 4) for x in prof_a[:8]],
                               "positions_shown": min(8, wl.L),
                               "tpf_unit_cost": prof_tpf,
                               "w_bar": [round(x, 4) for x in prof_w[:8]],
                               "tpf_isd_eq8": isd_tpf,
                               "w_bar_isd_eq8": [round(x, 4) for x in isd_w[:8]]},
        "graph_loop": graph_loop,
        "per_config": per_config,
        "distill_loss_us": distill_us,
        "replay": {"first_breakers": n_fb,
                   "intervention_rate_at_breakers": n_int / max(1, n_fb),
                   "rescue_rate_at_breakers": n_res / max(1, n_fb),
                   "regression_rate_at_accepted": n_reg / max(1, n_acc),
                   "call_us": replay_us},
    }
    print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def run_graph_loop(dev, blocks=30):
    """Per-block latency of the decode tail on one sequence (the `single` workload), as direct
    calls and as replays of the captured CUDA graph (App. F), anchors chained on the device."""
    import torch
    from paper_2609_33390_gb300 import brisk, synth
    wl = synth.WORKLOADS["single"]
    tail = brisk.DecodeTail.for_workload(wl, synth.make_weights(wl, dev), dev)
    tail.prepare()
    blk = synth.make_block(wl, dev)
    sm, vm = brisk.mode_ids(wl.select_mode, wl.verify_mode)
    stream = torch.cuda.Stream()
    out = tail.alloc_outputs(full=False)
    anchor = blk["x0"].clone()
    out["next_anchor"] = anchor
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        for _ in range(5):
            tail.tail(blk, sm, vm, out=out, x0=anchor, stream=stream)
        e0.record(stream)
        for _ in range(blocks):
            tail.tail(blk, sm, vm, out=out, x0=anchor, stream=stream)
        e1.record(stream)
    stream.synchronize()
    direct_us = 1000.0 * e0.elapsed_time(e1) / blocks
    g = tail.graph(blk, sm, vm, stream=stream)
    with torch.cuda.stream(stream):
        for _ in range(5):
            g.launch()
        e0.record(stream)
        acc = 0
        for _ in range(blocks):
            g.launch()
        e1.record(stream)
    stream.synchronize()
    graph_us = 1000.0 * e0.elapsed_time(e1) / blocks
    acc = int(g.out["accepted_len"].sum())
    g.close()
    # new inputs every block: double-buffered graphs, the next block copied in on a second stream
    pool = [synth.make_block(wl, dev, block=j) for j in range(4)]
    from paper_2609_33390_gb300.loop import graph_loop_double_buffered
    graph_loop_double_buffered(tail, pool, sm, vm, stream, 5)
    ms, nbytes, _ = graph_loop_double_buffered(tail, pool, sm, vm, stream, blocks)
    return {"workload": "single", "B": wl.B, "L": wl.L, "V": wl.V, "blocks": blocks,
            "direct_us_per_block": direct_us, "graph_us_per_block": graph_us,
            "graph_new_inputs_us_per_block": 1000.0 * ms / blocks,
            "new_inputs": f"{nbytes / 1e6:.1f} MB a block copied from a pool of {len(pool)} "
                          "pre-generated blocks on a second stream into the idle one of two "
                          "buffer sets, overlapped with the running block",
            "kernels_per_block": brisk.kernels_per_tail(tail.dims),
            "accepted_last_block": acc}


PER_CONFIG = ("tiny", "single", "batched_stochastic", "large_vocab")
L2_FLUSH_BYTES = 256 << 20   # twice the 129 MB L2


def run_per_config(dev, steps, names=PER_CONFIG, pool_n=3):
    """Every other workload configuration at its full size, outside the headline's timed region:
    per step (a fused decode-tail call, CUDA events on its stream, L2 flushed by a 256 MB write
    before each step and outside the events) the device time, the span of the two sweep launches
    (events the library records around them) and the accepted tokens; then the same blocks with
    the corrector's gate closed (alpha = -inf: the base ranking, rank 0 under greedy Select), for
    the acceptance the corrector changes."""
    import torch
    from paper_2609_33390_gb300 import brisk, synth
    peak, peak_src = measured_peaks()
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    res = {}
    for name in names:
        wl = synth.WORKLOADS[name]
        tail = brisk.DecodeTail.for_workload(wl, synth.make_weights(wl, dev), dev)
        tail.prepare()
        pool = [synth.make_block(wl, dev, block=j) for j in range(pool_n)]
        sm, vm = brisk.mode_ids(wl.select_mode, wl.verify_mode)
        nsteps = 3 + steps
        outs = [tail.alloc_outputs(full=False) for _ in range(nsteps)]
        evs = [tuple(torch.cuda.Event(enable_timing=True) for _ in range(6)) for _ in range(nsteps)]
        for ev in evs:
            for e in ev:
                e.record(stream)
        torch.cuda.synchronize()
        for s in range(nsteps):
            blk = pool[s % pool_n]
            x0 = blk["x0"] if s == 0 else outs[s - 1]["next_anchor"]
            flush.zero_()
            evs[s][4].record(stream)
            tail.tail(blk, sm, vm, out=outs[s], x0=x0, events=evs[s][:4])
            evs[s][5].record(stream)
        torch.cuda.synchronize()
        st = tail.device_status()
        if st != brisk.OK:
            raise RuntimeError(f"{name}: device status {brisk.status_string(st)}")
        timed = range(3, nsteps)
        step_ms = [evs[s][4].elapsed_time(evs[s][5]) for s in timed]
        span_ms = [sweep_span_ms(*evs[s][:4]) for s in timed]
        acc = sum(int(outs[s]["accepted_len"].sum()) for s in timed)
        # the same blocks and anchors with the gate closed
        alpha = tail.params.alpha
        tail.params.alpha = float("-inf")
        acc_off = 0
        for s in timed:
            blk = pool[s % pool_n]
            x0 = blk["x0"] if s == 0 else outs[s - 1]["next_anchor"]
            o = tail.tail(blk, sm, vm, x0=x0)
            acc_off += int(o["accepted_len"].sum())
        tail.params.alpha = alpha
        torch.cuda.synchronize()
        sweep_s = statistics.mean(span_ms) / 1000.0
        gbs = wl.sweep_bytes() / sweep_s / 1e9
        n_blocks = wl.B * steps
        res[name] = {
            "B": wl.B, "L": wl.L, "V": wl.V, "d": wl.d, "K": wl.K, "r": wl.r,
            "select": wl.select_mode, "verify": wl.verify_mode, "steps": steps,
            "us_per_step_mean": 1000.0 * statistics.mean(step_ms),
            "us_per_step_median": 1000.0 * statistics.median(step_ms),
            "accepted_tokens_per_s": acc / (sum(step_ms) / 1000.0),
            "sweep_bytes": wl.sweep_bytes(), "sweep_span_us": 1e6 * sweep_s,
            "sweep_gbs": gbs, "sweep_frac_of_peak": gbs / peak, "peak_source": peak_src,
            "sweep_frac_of_nameplate_8tbs": gbs / NAMEPLATE_HBM_GBS,
            "sweep_share_of_step": statistics.mean(span_ms) / statistics.mean(step_ms),
            "accepted_per_sequence_block": acc / n_blocks,
            "accepted_per_sequence_block_corrector_off": acc_off / n_blocks,
            "l2": "256 MB written before every step, outside its events",
        }
        del tail, pool, outs
        torch.cuda.empty_cache()
    return res


def run_e2e(args, tail, pool, wl, sm, vm, dev):
    """Same metric through the public API with host buffers. Every step the fused call reads the
    block's logits in place from pinned host memory (the kernels stream them over the host link),
    the other inputs are copied from pinned host memory, and the accepted lengths, tokens and
    corrections are read back. The same loop with every input copied first by the copy engine
    is reported beside it (`copy_inputs`)."""
    import torch
    n = max(1, min(args.e2e_steps, args.steps))
    keys = ("logits_q", "logits_p", "hidden", "h_c", "x0")
    in_place = ("logits_q", "logits_p")
    host = []
    for j in range(min(2, len(pool))):
        host.append({k: pool[j][k].cpu().pin_memory() for k in keys})
    dev_in = {k: torch.empty_like(pool[0][k]) for k in keys}
    out = tail.alloc_outputs(full=False)
    res_host = {k: torch.empty(out[k].shape, dtype=out[k].dtype).pin_memory()
                for k in ("accepted_len", "out_tokens", "correction")}
    h2d = sum(host[0][k].numel() * host[0][k].element_size() for k in keys)
    d2h = sum(v.numel() * v.element_size() for v in res_host.values())
    stream = torch.cuda.current_stream()

    def loop(copy_all):
        torch.cuda.synchronize()
        acc = 0
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        for it in range(n + 1):
            if it == 1:
                torch.cuda.synchronize()
                acc = 0
                e0.record(stream)
            h = host[it % len(host)]
            blk = {}
            for k in keys:
                if copy_all or k not in in_place:
                    dev_in[k].copy_(h[k], non_blocking=True)
                    blk[k] = dev_in[k]
                else:
                    blk[k] = h[k]
            tail.tail(blk, sm, vm, out=out)
            for k, v in res_host.items():
                v.copy_(out[k], non_blocking=True)
            stream.synchronize()
            if it >= 1:
                acc += int(res_host["accepted_len"].sum())
        e1.record(stream)
        torch.cuda.synchronize()
        return acc, e0.elapsed_time(e1) / 1000.0

    acc, secs = loop(copy_all=False)
    acc_c, secs_c = loop(copy_all=True)
    return {"value": acc / secs, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "steps": n, "ms_per_step": 1000.0 * secs / n,
            "logits": "read in place from pinned host memory by the kernels; hidden, h_c, x0 copied",
            "copy_inputs": {"value": acc_c / secs_c, "ms_per_step": 1000.0 * secs_c / n},
            "_tokens": acc, "_seconds": secs}


def run_profile(args):
    """A short run for profilers: `--steps` fused decode-tail calls on one block of the named
    workload (no timing output). Used to capture single kernels under ncu."""
    import torch
    from paper_2609_33390_gb300 import build, brisk, synth
    build.build()
    dev = torch.device("cuda")
    wl = synth.WORKLOADS[args.profile]
    if args.profile_batch:
        wl = wl.with_(B=args.profile_batch)
    if args.profile_vocab:
        wl = wl.with_(V=args.profile_vocab)
    weights = synth.make_weights(wl, dev)
    tail = brisk.DecodeTail.for_workload(wl, weights, dev)
    tail.prepare()
    blk = synth.make_block(wl, dev)
    sm, vm = brisk.mode_ids(wl.select_mode, wl.verify_mode)
    out = tail.alloc_outputs(full=False)
    for _ in range(args.warmup + args.steps):
        tail.tail(blk, sm, vm, out=out)
    torch.cuda.synchronize()
    st = tail.device_status()
    print(json.dumps({"profile": args.profile, "B": wl.B, "V": wl.V, "calls": args.warmup + args.steps,
                      "status": brisk.status_string(st),
                      "accepted": int(out["accepted_len"].sum())}))
    return 0 if st == brisk.OK else 1


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--pool", type=int, default=16, help="distinct pre-generated blocks cycled")
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-per-config", action="store_true",
                    help="skip the measurements of the other four workload configurations")
    ap.add_argument("--per-config-steps", type=int, default=20)
    ap.add_argument("--profile", default=None, help="workload name: short untimed run for ncu")
    ap.add_argument("--profile-batch", type=int, default=0,
                    help="with --profile: sequences per call instead of the workload's (a smaller case)")
    ap.add_argument("--profile-vocab", type=int, default=0,
                    help="with --profile: vocabulary size instead of the workload's (a smaller case)")
    args = ap.parse_args(argv)
    args.warmup = max(3, args.warmup)   # at least 3 untimed warm-up steps
    if args.profile:
        return run_profile(args)
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
