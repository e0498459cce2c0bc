"""Benchmark: ISM attention forward + backward on one packed batch of
synthetic multi-turn dialogues (default: batch 2 x 8192 tokens, 32 query /
8 KV heads, head_dim 128, bf16), reported as effective TFLOP/s counting only
visible (unmasked) query-key pairs: 14 * D * N_vis per step (forward
4 * D * N_vis, backward 10 * D * N_vis).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

For N > 1 launch one process per GPU with torch.distributed.run; every rank
processes its own replica of the batch (weak scaling, no collective on the
data path) and rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2408_00539_gb300 import workloads as wl  # noqa: E402

METRIC = "ISM attn fwd+bwd effective TFLOP/s and % of bf16 tensor peak at seq 8K, 1 GB300"
L2_BYTES = 129 * 2 ** 20


def n_visible(segs) -> int:
    """Visible (row, key) pairs per head, from the segment lengths: a query
    segment [s, e) contributes (e - s) * e pairs, an answer token j
    contributes j + 1 (sequence-relative).  Counting only, no attention."""
    total = 0
    for b in range(segs.num_seqs):
        _, _, se, st = segs.seq(b)
        start = 0
        for e, t in zip(se.tolist(), st.tolist()):
            n = e - start
            if t == wl.QUERY:
                total += n * e
            else:
                total += (start + 1 + e) * n // 2
            start = e
    return total


def n_tile_pairs(segs, tile: int = 128) -> int:
    """Non-empty (q-tile, k-tile) pairs at tile x tile: q-tile t reaches
    k-tiles [0, ceil(kv_end(last row) / tile)) (kv_end non-decreasing)."""
    total = 0
    for b in range(segs.num_seqs):
        _, L, se, st = segs.seq(b)
        for t in range((L + tile - 1) // tile):
            last = min(L, (t + 1) * tile) - 1
            i = int(np.searchsorted(se, last, side="right"))
            kv = int(se[i]) if int(st[i]) == wl.QUERY else last + 1
            total += (kv + tile - 1) // tile
    return total


def ncu_name(kind: str, stored_ds: bool) -> str:
    return {"fwd": "fwd_pair_kernel", "bwd_dkdv": "dkdv_kernel",
            "bwd_dq": "dq_gemm_kernel" if stored_ds else "dq_kernel"}.get(kind, "")


def kernel_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from the committed ncu capture, or None when the
    kernel's source changed since the counters were taken (or no capture of
    this workload exists)."""
    import hashlib
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as fh:
        rec = json.load(fh).get(kernel)
    if not rec or rec.get("workload") != workload:
        return None
    with open(os.path.join(ROOT, rec["source"]), "rb") as fh:
        if hashlib.sha256(fh.read()).hexdigest() != rec["source_sha256"]:
            return None
    return rec["dram_bytes_per_launch"]


def read_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as fh:
            d = json.load(fh)
        return d, "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled every 50 ms from before
    the warm-up on; ``summary`` keeps the samples taken inside the timed
    window (``mark_start`` / ``mark_end``), or, when the window is shorter
    than one sampling interval, the first sample after its start (the GPU is
    still running the same steps then)."""
    Q = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.t0 = self.t1 = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except (FileNotFoundError, OSError):
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def wait_first(self, timeout: float = 2.0):
        """Wait (at most ``timeout`` s) until nvidia-smi has printed a sample,
        so that a short timed window that follows gets one."""
        t_end = time.time() + timeout
        while self.proc is not None and not self.lines and time.time() < t_end:
            time.sleep(0.01)

    def mark_start(self):
        self.t0 = time.time()

    def hold(self, step, sync, limit: float = 1.0):
        """Keep running ``step`` (the timed work, outside the window) until a
        sample taken after the window's start has arrived, at most ``limit``
        seconds, so that short windows still get a clock record."""
        t_end = time.time() + limit
        while self.proc is not None and time.time() < t_end:
            if any(t >= (self.t0 or 0) for t, _ in list(self.lines)):
                break
            step()
            sync()

    def mark_end(self):
        self.t1 = time.time()

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        rows = []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for t, line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((t, float(parts[2]), float(parts[3]), parts[5:9]))
            except ValueError:
                continue
        t0 = self.t0 if self.t0 is not None else -np.inf
        t1 = self.t1 if self.t1 is not None else np.inf
        inside = [r for r in rows if t0 <= r[0] <= t1]
        if not inside:
            inside = [r for r in rows if r[0] >= t0][:1]
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        reasons = sorted({n for r in inside for n, v in zip(names, r[3]) if v.lower() == "active"})
        return {"sm_mhz": float(np.median([r[1] for r in inside])), "sm_max_mhz": max(r[2] for r in inside),
                "reasons": reasons, "samples": len(inside),
                "window_ms": None if self.t1 is None or self.t0 is None else (self.t1 - self.t0) * 1e3}


def dist_setup(args, backend: str = "nccl"):
    """One process per GPU (torchrun's RANK / LOCAL_RANK / WORLD_SIZE /
    MASTER_*); backend "gloo" runs the same bookkeeping on CPU processes."""
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        if backend == "nccl":
            torch.cuda.set_device(local)
            dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        else:
            dist.init_process_group(backend)
    elif torch.cuda.is_available():
        torch.cuda.set_device(0)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    """The slowest rank's time: the whole job's wall time for replicas."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank: float, world: int, steps: int, total_ms: float) -> float:
    """Whole-job rate of N replicas: every rank processes units_per_rank a
    step, over the slowest rank's time."""
    return units_per_rank * world * steps / (total_ms * 1e-3)


# ---------------------------------------------------------------- oracle arm

def oracle_sample(w, q, k, v, do, heads_per_sample: int):
    """Bounded CPU sample: fwd+bwd of the oracle over the first sequence and
    the first `heads_per_sample` query heads of one GQA group."""
    from oracle import ism_oracle as orc
    t0, L, se, st = w.segs.seq(0)
    grp = w.num_heads_q // w.num_heads_kv
    nh = min(heads_per_sample, grp)
    sub = wl.pack([(se, st)])
    qs = q[t0:t0 + L, :nh].contiguous()
    dos = do[t0:t0 + L, :nh].contiguous()
    ks = k[t0:t0 + L, :1].contiguous()
    vs = v[t0:t0 + L, :1].contiguous()
    n_vis = n_visible(sub) * nh
    tic = time.perf_counter()
    orc.attn_fwd(qs, ks, vs, sub, w.softmax_scale)
    orc.attn_bwd(qs, ks, vs, dos, sub, w.softmax_scale)
    dt = time.perf_counter() - tic
    flops = 14 * w.head_dim * n_vis
    return flops / dt / 1e12, dt, f"oracle fwd+bwd of sequence 0 ({L} tokens), {nh} query head(s) of KV head 0"


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


def run_reference(args, w):
    world, rank, _ = dist_setup(args) if args.gpus > 1 else (1, 0, 0)
    if rank != 0:
        return
    q, k, v, do = wl.attention_tensors(w)
    vals, times = [], []
    for i in range(args.warmup + args.steps):
        val, dt, sample = oracle_sample(w, q, k, v, do, heads_per_sample=1)
        if i >= args.warmup:
            vals.append(val)
            times.append(dt)
    value = float(np.mean(vals))
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": float(np.mean(times)) * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "sample": sample},
        "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": cpu_cores(), "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------- CUDA arm

def run_cuda(args, w):
    import torch
    from paper_2408_00539_gb300 import ism

    world, rank, local = dist_setup(args)
    dev = torch.device("cuda", local if world > 1 else 0)
    ism.load()
    peaks, peak_kind = read_peaks()

    q, k, v, do = wl.attention_tensors(w)
    segs = ism.Segments.from_workload(w.segs, dev)
    qd, kd, vd, dod = (t.to(dev) for t in (q, k, v, do))
    n_vis = n_visible(w.segs) * w.num_heads_q
    D = w.head_dim
    flops = 14 * D * n_vis
    o, lse = ism.fwd(segs, qd, kd, vd, w.softmax_scale)
    # backward workspace sized for the stored-dS schedule where it applies
    # (the minimum with --min-workspace: the recompute schedule)
    ws_bytes = ism.bwd_workspace_size(segs, qd, kd, w.softmax_scale, minimal=args.min_workspace)
    stored_ds = ws_bytes > ism.bwd_workspace_size(segs, qd, kd, w.softmax_scale, minimal=True)
    ws_b = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    dq, dk, dv = ism.bwd(segs, qd, kd, vd, o, lse, dod, w.softmax_scale, workspace=ws_b)
    flush = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device=dev)
    # a step builds the batch's plan (one metadata pass) and runs the forward
    # and the backward on it, as a training step over the same segments does
    plan = ism.Plan(segs, w.num_heads_q, w.num_heads_kv, w.head_dim, qd.dtype, dev)

    def step():
        plan.build()
        ism.fwd(segs, qd, kd, vd, w.softmax_scale, out=o, lse=lse, plan=plan)
        ism.bwd(segs, qd, kd, vd, o, lse, dod, w.softmax_scale, dq=dq, dk=dk, dv=dv, workspace=ws_b, plan=plan)

    if args.profile_step and args.rope:
        # the rotary step (usual schedule) for a profiler: same tensors, rotated copies
        cos_np, sin_np = wl.rope_tables(int(np.diff(w.segs.cu_seqlens).max()), D)
        cos_t, sin_t = torch.from_numpy(cos_np).to(dev), torch.from_numpy(sin_np).to(dev)
        q_rot, k_rot = torch.empty_like(qd), torch.empty_like(kd)

        def step():  # noqa: F811
            ism.fwd_rope(segs, qd, kd, vd, cos_t, sin_t, w.softmax_scale, q_rot=q_rot, k_rot=k_rot, out=o, lse=lse)
            ism.bwd_rope(segs, q_rot, k_rot, vd, o, lse, dod, cos_t, sin_t, w.softmax_scale, dq=dq, dk=dk, dv=dv,
                         workspace=ws_b)

    if args.profile_step and args.e4m3:
        # the e4m3 forward alone for a profiler: e4m3 copies of the same Q, K, V
        q8, k8, v8 = (wl.quantize_e4m3(t) for t in (qd, kd, vd))

        def step():  # noqa: F811
            ism.fwd_e4m3(segs, q8[0], k8[0], v8[0], q8[1], k8[1], v8[1], w.softmax_scale)

    # clocks are sampled from the warm-up on (nvidia-smi needs a moment to start)
    clocks = ClockSampler(dev.index) if not args.profile_step else None
    if clocks is not None:
        clocks.__enter__()
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    ism.check_status(dev)
    if args.profile_step:
        # one more step for a profiler to capture, then stop (no timing, no JSON)
        step()
        torch.cuda.synchronize()
        ism.check_status(dev)
        return

    # timed steps: CUDA events around each step only
    stream = torch.cuda.current_stream(dev)
    step_ms = []
    launches0 = ism.kernel_launches()
    barrier(world)
    torch.cuda.synchronize()
    clocks.mark_start()
    for _ in range(args.steps):
        flush.fill_(1)  # evict L2 between timed steps (outside the step's events)
        s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s0.record(stream)
        step()
        s1.record(stream)
        s1.synchronize()
        step_ms.append(s0.elapsed_time(s1))
    torch.cuda.synchronize()
    clocks.mark_end()
    barrier(world)
    launches = ism.kernel_launches() - launches0
    # keep the GPU busy with the same steps a little longer, so that a timed
    # region shorter than the sampling interval still gets a sample
    clocks.hold(step, torch.cuda.synchronize)
    clocks.__exit__(None, None, None)
    ism.check_status(dev)

    # per-kernel times for the rooflines, from separate steps run with the
    # library's kernel-timer hooks (events recorded on its launch stream)
    kinds = {"fwd": ism.KERNEL_FWD, "bwd_dkdv": ism.KERNEL_BWD_DKDV, "bwd_dq": ism.KERNEL_BWD_DQ,
             "bwd_pre": ism.KERNEL_BWD_PRE, "meta": ism.KERNEL_META}
    ktimes = {n: [] for n in kinds}
    for _ in range(max(3, min(args.steps, 10))):
        flush.fill_(1)
        ev = {n: (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for n in kinds}
        for n, kid in kinds.items():
            for e in ev[n]:
                e.record(stream)  # creates the event; the library re-records it around its launch
            ism.set_kernel_timer(kid, *ev[n])
        step()
        torch.cuda.synchronize()
        for n in kinds:
            ktimes[n].append(ev[n][0].elapsed_time(ev[n][1]))
    for kid in kinds.values():
        ism.set_kernel_timer(kid)
    ism.check_status(dev)

    total_ms = max_over_ranks(float(np.sum(step_ms)), world)
    ms_per_step = total_ms / args.steps
    value = job_throughput(flops, world, args.steps, total_ms) / 1e12

    # roofline of each attention kernel; the dominant one (largest share of
    # the step) is the line's "roofline"
    mean_k = {n: float(np.mean(t)) for n, t in ktimes.items()}
    peak_tc = peaks.get("bf16_tflops_sustained" if args.steps * ms_per_step > 2000 else "bf16_tflops")
    T, Hq, Hkv = w.total_tokens, w.num_heads_q, w.num_heads_kv
    ds_bytes = n_tile_pairs(w.segs) * Hq * 128 * 128 * 2 if stored_ds else 0
    rooflines = {}
    for kind, fl in (("fwd", 4), ("bwd_dkdv", 8), ("bwd_dq", 6)):
        kname = ncu_name(kind, stored_ds)
        ms = mean_k[kind]
        if kind == "bwd_dq" and stored_ds:
            # GEMM over the stored dS tiles: reads dS and K once, writes dQ
            nbytes = ds_bytes + T * Hkv * D * 2 + T * Hq * D * 2
            ach = nbytes / (ms * 1e-3) / 1e9
            r = {"bound": "hbm", "achieved": ach, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                 "frac": ach / peaks["hbm_gbs"], "bytes_per_launch": nbytes}
        else:
            fpl = fl * D * n_vis
            ach = fpl / (ms * 1e-3) / 1e12
            r = {"bound": "tensor", "achieved": ach, "peak": peak_tc, "unit": "TFLOP/s", "frac": ach / peak_tc,
                 "flops_per_launch": fpl}
        r.update({"kernel": kname, "traffic": kernel_traffic(kname, w.name), "peak_kind": peak_kind,
                  "ms_per_launch": ms})
        rooflines[kind] = r
    dom = max(rooflines, key=lambda n: mean_k[n])
    roofline = dict(rooflines[dom])

    # end to end through the public API with host buffers
    pin = lambda t: t.pin_memory()  # noqa: E731
    qh, kh, vh, doh = pin(q), pin(k), pin(v), pin(do)
    dqh, dkh, dvh = (torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in (q, k, v))
    h2d = sum(t.numel() * t.element_size() for t in (qh, kh, vh, doh))
    d2h = sum(t.numel() * t.element_size() for t in (dqh, dkh, dvh))

    copy_stream = torch.cuda.Stream(dev)

    def e2e_step():
        # Q, K, V feed the forward; dO is uploaded on a second stream while the
        # forward runs, and the backward waits for it
        qd.copy_(qh, non_blocking=True)
        kd.copy_(kh, non_blocking=True)
        vd.copy_(vh, non_blocking=True)
        copy_stream.wait_stream(stream)
        with torch.cuda.stream(copy_stream):
            dod.copy_(doh, non_blocking=True)
        plan.build()
        ism.fwd(segs, qd, kd, vd, w.softmax_scale, out=o, lse=lse, plan=plan)
        stream.wait_stream(copy_stream)
        ism.bwd(segs, qd, kd, vd, o, lse, dod, w.softmax_scale, dq=dq, dk=dk, dv=dv, workspace=ws_b, plan=plan)
        dqh.copy_(dq, non_blocking=True)
        dkh.copy_(dk, non_blocking=True)
        dvh.copy_(dv, non_blocking=True)

    # (a) one step at a time: upload, fwd+bwd, read back, in series
    for _ in range(2):
        e2e_step()
    torch.cuda.synchronize()
    serial_ms = []
    for _ in range(args.steps):
        flush.fill_(1)
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        e2e_step()
        a1.record(stream)
        a1.synchronize()
        serial_ms.append(a0.elapsed_time(a1))
    serial_total = max_over_ranks(float(np.sum(serial_ms)), world)

    # (b) K steps back to back as a training loop runs them: the inputs of step
    # i+1 are uploaded on one copy stream and the gradients of step i read back
    # on another while step i+1 computes (double-buffered device tensors); the
    # timed region holds every step's uploads and read-backs
    ins = [[torch.empty_like(t) for t in (qd, kd, vd, dod)] for _ in range(2)]
    outs = [[torch.empty_like(t) for t in (dq, dk, dv)] for _ in range(2)]
    ob = [torch.empty_like(o) for _ in range(2)]
    lb = [torch.empty_like(lse) for _ in range(2)]
    up, down = torch.cuda.Stream(dev), torch.cuda.Stream(dev)

    def run_pipelined(n_steps):
        # ev_in: Q, K, V of a step uploaded; ev_in_do: its dO (needed only by the backward)
        ev_in = [torch.cuda.Event() for _ in range(n_steps)]
        ev_in_do = [torch.cuda.Event() for _ in range(n_steps)]
        ev_done = [torch.cuda.Event() for _ in range(n_steps)]
        ev_out = [torch.cuda.Event() for _ in range(n_steps)]
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)

        def upload(i):
            up.wait_event(a0)
            if i >= 2:
                up.wait_event(ev_done[i - 2])  # that buffer set's last user finished
            with torch.cuda.stream(up):
                for dst, src in zip(ins[i % 2][:3], (qh, kh, vh)):
                    dst.copy_(src, non_blocking=True)
                ev_in[i].record(up)
                ins[i % 2][3].copy_(doh, non_blocking=True)
                ev_in_do[i].record(up)

        upload(0)
        for i in range(n_steps):
            bsel = i % 2
            if i + 1 < n_steps:
                upload(i + 1)
            plan.build()  # needs no input: runs while the inputs may still be on their way
            stream.wait_event(ev_in[i])
            if i >= 2:
                stream.wait_event(ev_out[i - 2])  # its gradients were read back
            qb, kb, vb, dob = ins[bsel]
            dqb, dkb, dvb = outs[bsel]
            ism.fwd(segs, qb, kb, vb, w.softmax_scale, out=ob[bsel], lse=lb[bsel], plan=plan)
            stream.wait_event(ev_in_do[i])
            ism.bwd(segs, qb, kb, vb, ob[bsel], lb[bsel], dob, w.softmax_scale, dq=dqb, dk=dkb, dv=dvb,
                    workspace=ws_b, plan=plan)
            ev_done[i].record(stream)
            down.wait_event(ev_done[i])
            with torch.cuda.stream(down):
                for dst, src in zip((dqh, dkh, dvh), outs[bsel]):
                    dst.copy_(src, non_blocking=True)
            ev_out[i].record(down)
        stream.wait_event(ev_out[n_steps - 1])
        a1.record(stream)
        a1.synchronize()
        return a0.elapsed_time(a1)

    run_pipelined(3)
    torch.cuda.synchronize()
    # three runs of the K steps, the median reported: the host side of the
    # copies (pinned buffers, the CPU-GPU link) is shared with whatever else
    # runs on the machine and varies from run to run
    e2e_runs = []
    for _ in range(3):
        barrier(world)
        e2e_runs.append(max_over_ranks(run_pipelined(args.steps), world))
    e2e_total = float(np.median(e2e_runs))
    e2e_value = job_throughput(flops, world, args.steps, e2e_total) / 1e12

    if rank != 0:
        return
    line = {
        "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": w.name, "tokens": w.total_tokens, "n_vis_pairs": n_vis,
                   "flops_per_step": flops, "flop_count": "14*D*N_vis (fwd 4, bwd 10)",
                   "strict_tflops_12D": value * 12 / 14, "l2": "flushed between timed steps (258 MB write)",
                   "pct_of_peak": value / peak_tc * 100, "path": "tensor cores" if ism.has_tensor_cores()
                   else "cuda cores", "bwd_schedule": "stored dS" if stored_ds else "recompute dQ",
                   "bwd_workspace_bytes": ws_bytes,
                   "metadata": "one pass a step (ism_attn_plan_build), shared by the forward and the backward",
                   "parallelism": f"replicas x{world}"},
        "kernel_ms": mean_k,
        "phases": {
            "fwd": {"ms": mean_k["meta"] + mean_k["fwd"], "flops": 4 * D * n_vis,
                    "tflops": 4 * D * n_vis / ((mean_k["meta"] + mean_k["fwd"]) * 1e-3) / 1e12,
                    "kernels": "metadata pass (the plan) + forward"},
            "bwd": {"ms": mean_k["bwd_pre"] + mean_k["bwd_dkdv"] + mean_k["bwd_dq"],
                    "flops": 10 * D * n_vis,
                    "tflops": 10 * D * n_vis / ((mean_k["bwd_pre"] + mean_k["bwd_dkdv"] +
                                                 mean_k["bwd_dq"]) * 1e-3) / 1e12,
                    "kernels": "Delta + dK/dV + dQ on the plan"},
            "note": "per-kernel times from the timer hooks; a step builds the plan (one metadata pass) and "
                    "runs the forward and the backward on it; the headline counts fwd 4*D*N_vis and bwd "
                    "10*D*N_vis"},
        "roofline": roofline,
        "kernel_rooflines": rooflines,
        "e2e": {"value": e2e_value, "unit": "TFLOP/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "ms_per_step": e2e_total / args.steps,
                "ms_per_step_runs": [t / args.steps for t in e2e_runs],
                "how": "median of three runs of K steps back to back through ism.Plan.build/ism.fwd/ism.bwd; step i+1's Q, K, V, dO uploads (pinned host, "
                       "copy stream; the forward waits for Q, K, V, the backward for dO) and step i's dQ, dK, dV "
                       "read-backs (second copy stream) overlap the kernels; double-buffered device tensors; "
                       "inputs (335 MB) exceed L2, no flush",
                "serial": {"value": job_throughput(flops, world, args.steps, serial_total) / 1e12,
                           "ms_per_step": serial_total / args.steps,
                           "how": "each step alone: upload, plan + fwd + bwd, read-back, L2 flushed between steps"}},
        "gpu_launches": int(launches),
        "clocks": clocks.summary(),
    }
    if not args.no_extra:
        line["bwd_min_workspace"] = measure_training_config(dev, w, peaks, steps=args.steps, minimal_workspace=True)
        line["rope"] = measure_training_config(dev, w, peaks, steps=args.steps, rope=True)
        line["configs"] = {wname: measure_training_config(dev, WORKLOADS[wname](), peaks, steps=args.steps)
                           for wname in ("mha_4k", "packed_32k") if WORKLOADS[wname]().name != w.name}
    if not args.no_append:
        line["append"] = measure_append(dev, read_peaks()[0])
        line["session"] = measure_session(dev)
        line["training_cost"] = measure_training_cost(dev, w)
        line["fwd_e4m3"] = measure_fwd_e4m3(dev, w, read_peaks()[0])
    if not args.no_extra:
        # the seconds-long runs come last: the power-capped clocks they leave
        # behind would slow the short measurements taken right after them
        line["sustained"] = measure_sustained(dev, step, flops, peaks)
        del ins, outs, ob, lb
        torch.cuda.empty_cache()
        line["long_context"] = measure_long_context(dev, peaks)
    if world == 1 and not args.no_cpu_baseline:
        val, dt, sample = oracle_sample(w, q, k, v, do, heads_per_sample=4)
        line["cpu_baseline"] = {"value": val, "unit": "TFLOP/s", "cores": cpu_cores(), "kind": "oracle",
                                "sample": sample, "seconds": dt}
    print(json.dumps(line), flush=True)


def measure_append(dev, peaks):
    """Append-prefill of a 512-token query turn against 8 x 16384 cached
    tokens, then answer-token decode steps (reported beside the headline;
    timed with CUDA events per call, caches larger than L2)."""
    import torch
    from paper_2408_00539_gb300 import ism
    a = wl.append_16k()
    B, cap, hq, hkv, d, ln = a.batch, a.capacity, a.num_heads_q, a.num_heads_kv, a.head_dim, a.l_new
    g = torch.Generator(device=dev).manual_seed(a.seed)
    kc = torch.randn((B, cap, hkv, d), generator=g, device=dev, dtype=torch.float32).mul_(a.value_std).bfloat16()
    vc = torch.randn((B, cap, hkv, d), generator=g, device=dev, dtype=torch.float32).mul_(a.value_std).bfloat16()
    qn = torch.randn((B, ln, hq, d), generator=g, device=dev).mul_(a.value_std).bfloat16()
    kn = torch.randn((B, ln, hkv, d), generator=g, device=dev).mul_(a.value_std).bfloat16()
    vn = torch.randn((B, ln, hkv, d), generator=g, device=dev).mul_(a.value_std).bfloat16()
    qd = torch.randn((B, 1, hq, d), generator=g, device=dev).mul_(a.value_std).bfloat16()
    kd = torch.randn((B, 1, hkv, d), generator=g, device=dev).mul_(a.value_std).bfloat16()
    vd = torch.randn((B, 1, hkv, d), generator=g, device=dev).mul_(a.value_std).bfloat16()
    c0 = a.cache_len.copy()
    cl = torch.from_numpy(c0.copy()).to(dev)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device=dev)
    # prefill: cache_len is reset before every call (outside the events)
    pre_ms = []
    for it in range(8):
        cl.copy_(torch.from_numpy(c0))
        flush.fill_(1)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        ism.prefill_append(qn, kn, vn, kc, vc, cl, c0, a.new_seg_end, a.new_seg_type, a.softmax_scale)
        e1.record(stream)
        e1.synchronize()
        if it >= 3:
            pre_ms.append(e0.elapsed_time(e1))
    ism.check_status(dev)
    n_vis_pre = int(B * hq * ln * (int(c0[0]) + ln))  # every new row sees the cache and the whole new query
    pre = float(np.median(pre_ms))
    # decode steps after the prefill
    # decode steps after the prefill, through a prepared call (one C call a
    # step, as a generation loop makes them); the decode kernels are timed by
    # the library's timer hook inside each call
    c_host = (c0 + ln).astype(np.int32)
    cl.copy_(torch.from_numpy(c_host))
    step = ism.AppendStep(qd, kd, vd, kc, vc, cl, c_host, [1], [1], a.softmax_scale)
    dec_us, dec_kernel_us, dec_bytes = [], [], []
    for t in range(a.decode_steps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        k0, k1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        for e in (k0, k1):
            e.record(stream)
        ism.set_kernel_timer(ism.KERNEL_DECODE, k0, k1)
        e0.record(stream)
        step()
        e1.record(stream)
        e1.synchronize()
        ism.set_kernel_timer(ism.KERNEL_DECODE)
        dec_us.append(e0.elapsed_time(e1) * 1e3)
        dec_kernel_us.append(k0.elapsed_time(k1) * 1e3)
        dec_bytes.append(2 * B * (int(c_host[0]) + 1) * hkv * d * 2)
        c_host += 1
    ism.check_status(dev)
    us = float(np.median(dec_us[3:]))
    kus = float(np.median(dec_kernel_us[3:]))
    gbs = float(np.median(np.array(dec_bytes[3:]) / (np.array(dec_kernel_us[3:]) * 1e-6) / 1e9))
    # the same step through the plain binding (argument conversion, workspace
    # and output allocation on every call), over the last 16 positions again
    c_host -= 16
    cl.copy_(torch.from_numpy(c_host))
    plain_us = []
    for t in range(16):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        ism.prefill_append(qd, kd, vd, kc, vc, cl, c_host, [1], [1], a.softmax_scale)
        e1.record(stream)
        e1.synchronize()
        plain_us.append(e0.elapsed_time(e1) * 1e3)
        c_host += 1
    ism.check_status(dev)
    paged = measure_append_paged(dev, a, kc, vc, qn, kn, vn, qd, kd, vd, flush)
    e4m3 = measure_append_e4m3(dev, a, kc, vc, qn, kn, vn, qd, kd, vd, flush, peaks)
    rope = measure_append_rope(dev, a, kc, vc, qn, kn, vn, qd, kd, vd, flush)
    return {"workload": a.name,
            "prefill_ms": pre, "prefill_tflops": 4 * d * n_vis_pre / (pre * 1e-3) / 1e12,
            "prefill_frac_of_bf16_peak": 4 * d * n_vis_pre / (pre * 1e-3) / 1e12 / peaks["bf16_tflops"],
            "decode_us_per_call": us, "decode_kernel_us": kus,
            "decode_us_per_call_plain_binding": float(np.median(plain_us[3:])),
            "decode_hbm_gbs": gbs, "decode_frac_of_hbm": gbs / peaks["hbm_gbs"],
            "decode_steps": a.decode_steps,
            "paged": paged,
            "e4m3": e4m3,
            "rope": rope,
            "note": "decode bytes = K and V cache read once: 2*B*(c+1)*Hkv*D*2 per step; GB/s over the "
                    "split-KV + merge kernels (decode_kernel_us); decode_us_per_call: CUDA events around one "
                    "prepared call (ism.AppendStep), which adds the cache-write kernel and the host time of the "
                    "call; decode_us_per_call_plain_binding: the same through ism.prefill_append"}


def measure_append_paged(dev, a, kc, vc, qn, kn, vn, qd, kd, vd, flush, page_size=256, decode_steps=64):
    """The append-prefill and decode of ``measure_append`` against the same
    cache held in shuffled pages of one pool (block table per sequence)."""
    import torch
    from paper_2408_00539_gb300 import ism
    B, cap = kc.shape[0], kc.shape[1]
    max_pages = (cap + page_size - 1) // page_size
    rng = np.random.Generator(np.random.PCG64(a.seed))
    table = rng.permutation(B * max_pages).reshape(B, max_pages).astype(np.int32)
    rows = (torch.from_numpy(table).to(dev).long()[:, :, None] * page_size +
            torch.arange(page_size, device=dev)[None, None, :]).reshape(B, -1)[:, :cap]
    kp = torch.empty((B * max_pages * page_size,) + tuple(kc.shape[2:]), dtype=kc.dtype, device=dev)
    vp = torch.empty_like(kp)
    kp[rows.reshape(-1)] = kc.reshape((-1,) + tuple(kc.shape[2:]))
    vp[rows.reshape(-1)] = vc.reshape((-1,) + tuple(vc.shape[2:]))
    del rows
    td = torch.from_numpy(table).to(dev)
    c0 = a.cache_len.copy()
    cl = torch.from_numpy(c0.copy()).to(dev)
    stream = torch.cuda.current_stream(dev)
    pre_ms = []
    for it in range(8):
        cl.copy_(torch.from_numpy(c0))
        flush.fill_(1)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        ism.prefill_append_paged(qn, kn, vn, kp, vp, page_size, td, table, cl, c0, a.new_seg_end, a.new_seg_type,
                                 a.softmax_scale)
        e1.record(stream)
        e1.synchronize()
        if it >= 3:
            pre_ms.append(e0.elapsed_time(e1))
    c_host = c0 + a.l_new
    cl.copy_(torch.from_numpy(c_host))
    dec_kernel_us = []
    for t in range(decode_steps):
        k0, k1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        for e in (k0, k1):
            e.record(stream)
        ism.set_kernel_timer(ism.KERNEL_DECODE, k0, k1)
        ism.prefill_append_paged(qd, kd, vd, kp, vp, page_size, td, table, cl, c_host, [1], [1], a.softmax_scale)
        k1.synchronize()
        ism.set_kernel_timer(ism.KERNEL_DECODE)
        dec_kernel_us.append(k0.elapsed_time(k1) * 1e3)
        c_host = c_host + 1
    ism.check_status(dev)
    del kp, vp
    return {"page_size": page_size, "prefill_ms": float(np.median(pre_ms)),
            "decode_kernel_us": float(np.median(dec_kernel_us[3:])), "decode_steps": decode_steps}


def measure_append_rope(dev, a, kc, vc, qn, kn, vn, qd, kd, vd, flush, decode_steps=64):
    """The append-prefill and decode of ``measure_append`` with rotary
    encoding of the new queries and keys fused into the cache-write pass,
    against the same calls without it; the metadata timer gives the plan +
    cache-write kernels alone (L2 flushed before each prefill)."""
    import torch
    from paper_2408_00539_gb300 import ism
    cap, d = kc.shape[1], kc.shape[3]
    cos_np, sin_np = wl.rope_tables(cap, d)
    cos_t, sin_t = torch.from_numpy(cos_np).to(dev), torch.from_numpy(sin_np).to(dev)
    c0 = a.cache_len.copy()
    cl = torch.from_numpy(c0.copy()).to(dev)
    stream = torch.cuda.current_stream(dev)
    out = {}
    for name, call in (("plain", lambda q, k, v, ch, se, st: ism.prefill_append(q, k, v, kc, vc, cl, ch, se, st,
                                                                                  a.softmax_scale)),
                       ("rope", lambda q, k, v, ch, se, st: ism.prefill_append_rope(q, k, v, kc, vc, cl, ch, se, st,
                                                                                     cos_t, sin_t, a.softmax_scale))):
        pre_ms, meta_us = [], []
        for it in range(8):
            cl.copy_(torch.from_numpy(c0))
            flush.fill_(1)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            m0, m1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            for e in (m0, m1):
                e.record(stream)
            ism.set_kernel_timer(ism.KERNEL_META, m0, m1)
            e0.record(stream)
            call(qn, kn, vn, c0, a.new_seg_end, a.new_seg_type)
            e1.record(stream)
            e1.synchronize()
            ism.set_kernel_timer(ism.KERNEL_META)
            if it >= 3:
                pre_ms.append(e0.elapsed_time(e1))
                meta_us.append(m0.elapsed_time(m1) * 1e3)
        c_host = c0 + a.l_new
        cl.copy_(torch.from_numpy(c_host))
        dec_us = []
        for t in range(decode_steps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            call(qd, kd, vd, c_host, [1], [1])
            e1.record(stream)
            e1.synchronize()
            dec_us.append(e0.elapsed_time(e1) * 1e3)
            c_host = c_host + 1
        ism.check_status(dev)
        out[name] = {"prefill_ms": float(np.median(pre_ms)), "prefill_plan_and_cache_write_us": float(np.median(meta_us)),
                     "decode_us_per_call": float(np.median(dec_us[3:]))}
    out["decode_steps"] = decode_steps
    out["note"] = ("rope: new queries and keys rotated at positions cache_len + j (tables [cap, D/2] fp32) inside "
                   "the cache-write kernel; the attention kernels are the same")
    return out


def measure_training_config(dev, w, peaks, steps=20, minimal_workspace=False, rope=False):
    """fwd+bwd steps of one workload timed as the headline is: inputs resident,
    L2 flushed between steps (outside the events), CUDA events around each
    step, per-kernel times from separate steps through the library's timer
    hooks, clocks sampled over the timed steps.  minimal_workspace runs the
    backward with ism_attn_bwd_workspace_size_min bytes (the recompute
    schedule: no stored dS); rope runs the rotary forward and backward
    (queries and keys rotated at their positions, the usual schedule)."""
    import torch
    from paper_2408_00539_gb300 import ism
    q, k, v, do = (t.to(dev) for t in wl.attention_tensors(w))
    segs = ism.Segments.from_workload(w.segs, dev)
    n_vis = n_visible(w.segs) * w.num_heads_q
    D = w.head_dim
    flops = 14 * D * n_vis
    ws_bytes = ism.bwd_workspace_size(segs, q, k, w.softmax_scale, minimal=minimal_workspace)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    o, lse = ism.fwd(segs, q, k, v, w.softmax_scale)
    dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    flush = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)
    plan = ism.Plan(segs, w.num_heads_q, w.num_heads_kv, w.head_dim, q.dtype, dev)

    def step():  # the plan (one metadata pass), the forward and the backward on it
        plan.build()
        ism.fwd(segs, q, k, v, w.softmax_scale, out=o, lse=lse, plan=plan)
        ism.bwd(segs, q, k, v, o, lse, do, w.softmax_scale, dq=dq, dk=dk, dv=dv, workspace=ws, plan=plan)

    if rope:
        cos_np, sin_np = wl.rope_tables(int(np.diff(w.segs.cu_seqlens).max()), D)
        cos_t, sin_t = torch.from_numpy(cos_np).to(dev), torch.from_numpy(sin_np).to(dev)
        q_rot, k_rot = torch.empty_like(q), torch.empty_like(k)

        def step():  # noqa: F811
            plan.build()
            ism.fwd_rope(segs, q, k, v, cos_t, sin_t, w.softmax_scale, q_rot=q_rot, k_rot=k_rot, out=o, lse=lse,
                         plan=plan)
            ism.bwd_rope(segs, q_rot, k_rot, v, o, lse, do, cos_t, sin_t, w.softmax_scale, dq=dq, dk=dk, dv=dv,
                         workspace=ws, plan=plan)

    with ClockSampler(dev.index) as clocks:
        for _ in range(3):
            step()
        torch.cuda.synchronize()
        clocks.wait_first()
        ms = []
        clocks.mark_start()
        for _ in range(steps):
            flush.fill_(1)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            step()
            e1.record(stream)
            e1.synchronize()
            ms.append(e0.elapsed_time(e1))
        clocks.mark_end()
        clocks.hold(step, torch.cuda.synchronize)
    ism.check_status(dev)
    kinds = {"fwd": ism.KERNEL_FWD, "bwd_dkdv": ism.KERNEL_BWD_DKDV, "bwd_dq": ism.KERNEL_BWD_DQ,
             "bwd_pre": ism.KERNEL_BWD_PRE, "meta": ism.KERNEL_META}
    if rope:
        kinds["rope"] = ism.KERNEL_ROPE
    kt = {n: [] for n in kinds}
    for _ in range(5):
        flush.fill_(1)
        ev = {n: (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for n in kinds}
        for n, kid in kinds.items():
            for e in ev[n]:
                e.record(stream)
            ism.set_kernel_timer(kid, *ev[n])
        step()
        torch.cuda.synchronize()
        for n in kinds:
            kt[n].append(ev[n][0].elapsed_time(ev[n][1]))
    for kid in kinds.values():
        ism.set_kernel_timer(kid)
    ism.check_status(dev)
    ms_step = float(np.sum(ms)) / steps
    tflops = flops / (ms_step * 1e-3) / 1e12
    mean_k = {n: float(np.mean(t)) for n, t in kt.items()}
    peak = peaks["bf16_tflops"]
    fracs = {"fwd": 4 * D * n_vis / (mean_k["fwd"] * 1e-3) / 1e12 / peak,
             "bwd_dkdv": 8 * D * n_vis / (mean_k["bwd_dkdv"] * 1e-3) / 1e12 / peak}
    out = {"workload": w.name, "tokens": w.total_tokens, "n_vis_pairs": n_vis, "flops_per_step": flops,
           "ms_per_step": ms_step, "steps": steps, "tflops": tflops, "pct_of_bf16_peak": tflops / peak * 100,
           "bwd_schedule": "recompute dQ" if minimal_workspace else "stored dS", "rope": rope,
           "bwd_workspace_bytes": ws_bytes, "kernel_ms": mean_k, "kernel_frac_of_bf16_peak": fracs,
           "clocks": clocks.summary()}
    del q, k, v, do, o, lse, dq, dk, dv, ws, flush
    torch.cuda.empty_cache()
    return out


def measure_long_context(dev, peaks, length=131072, steps=3):
    """One dialogue of ``length`` tokens (a few hundred turns of the config-2
    recipe, 32 query / 8 KV heads, head_dim 128, bf16) through the forward and
    the minimum-workspace backward: the stored-dS workspace would need
    pairs x 32 heads x 32 KiB (about 0.5 TB at 128K), so long contexts run
    the recompute schedule.  Inputs drawn on the device (seeded); CUDA events
    around each step; the step is far larger than L2."""
    import torch
    from paper_2408_00539_gb300 import ism
    rng = np.random.Generator(np.random.PCG64(131))
    segs_np = wl.pack([wl.draw_dialogue(rng, length, 300, 400)])
    hq, hkv, D = 32, 8, 128
    scale = D ** -0.5
    g = torch.Generator(device=dev).manual_seed(131)
    q = torch.randn((length, hq, D), generator=g, device=dev).mul_(0.5).bfloat16()
    k = torch.randn((length, hkv, D), generator=g, device=dev).mul_(0.5).bfloat16()
    v = torch.randn((length, hkv, D), generator=g, device=dev).mul_(0.5).bfloat16()
    do = torch.randn((length, hq, D), generator=g, device=dev).bfloat16()
    segs = ism.Segments.from_workload(segs_np, dev)
    ws = torch.empty(ism.bwd_workspace_size(segs, q, k, scale, minimal=True), dtype=torch.uint8, device=dev)
    o, lse = ism.fwd(segs, q, k, v, scale)
    dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    stream = torch.cuda.current_stream(dev)
    plan = ism.Plan(segs, hq, hkv, D, q.dtype, dev)
    n_vis = n_visible(segs_np) * hq
    flops = 14 * D * n_vis
    kinds = {"fwd": ism.KERNEL_FWD, "bwd_dkdv": ism.KERNEL_BWD_DKDV, "bwd_dq": ism.KERNEL_BWD_DQ}
    ms, kt = [], {n: [] for n in kinds}
    for it in range(steps + 1):
        ev = {n: (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for n in kinds}
        for n, kid in kinds.items():
            for e in ev[n]:
                e.record(stream)
            ism.set_kernel_timer(kid, *ev[n])
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        plan.build()
        ism.fwd(segs, q, k, v, scale, out=o, lse=lse, plan=plan)
        ism.bwd(segs, q, k, v, o, lse, do, scale, dq=dq, dk=dk, dv=dv, workspace=ws, plan=plan)
        e1.record(stream)
        e1.synchronize()
        if it:
            ms.append(e0.elapsed_time(e1))
            for n in kinds:
                kt[n].append(ev[n][0].elapsed_time(ev[n][1]))
    for kid in kinds.values():
        ism.set_kernel_timer(kid)
    ism.check_status(dev)
    step_ms = float(np.median(ms))
    tflops = flops / (step_ms * 1e-3) / 1e12
    mean_k = {n: float(np.mean(t)) for n, t in kt.items()}
    fr = {"fwd": 4 * D * n_vis / (mean_k["fwd"] * 1e-3) / 1e12 / peaks["bf16_tflops"],
          "bwd_dkdv": 8 * D * n_vis / (mean_k["bwd_dkdv"] * 1e-3) / 1e12 / peaks["bf16_tflops"],
          "bwd_dq": 6 * D * n_vis / (mean_k["bwd_dq"] * 1e-3) / 1e12 / peaks["bf16_tflops"]}
    out = {"workload": f"long_t{length}_hq32_hkv8_d128", "segments": int(segs_np.seg_end.shape[0]),
           "n_vis_pairs": n_vis, "ms_per_step": step_ms, "steps": steps, "tflops": tflops,
           "pct_of_bf16_peak": tflops / peaks["bf16_tflops"] * 100, "bwd_schedule": "recompute dQ",
           "bwd_workspace_bytes": int(ws.numel()), "kernel_ms": mean_k, "kernel_frac_of_bf16_peak": fr,
           "note": "dQ kernel recomputes S and dP: 6*D*N_vis; dK/dV 8*D*N_vis; forward 4*D*N_vis"}
    del q, k, v, do, o, lse, dq, dk, dv, ws
    torch.cuda.empty_cache()
    return out


def measure_sustained(dev, step, flops, peaks, seconds=3.0):
    """The headline step run back to back, as a training loop runs it (no L2
    flush), for at least ``seconds``: the rate once the clocks have settled
    under the power limit, against the sustained bf16 peak."""
    import torch
    probe = []
    stream = torch.cuda.current_stream(dev)
    for _ in range(5):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        step()
        e1.record(stream)
        e1.synchronize()
        probe.append(e0.elapsed_time(e1))
    n = int(np.ceil(seconds * 1e3 / float(np.median(probe))))
    with ClockSampler(dev.index) as clocks:
        torch.cuda.synchronize()
        clocks.mark_start()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(n):
            step()
        e1.record(stream)
        e1.synchronize()
        clocks.mark_end()
    total = e0.elapsed_time(e1)
    tflops = flops * n / (total * 1e-3) / 1e12
    return {"steps": n, "seconds": total * 1e-3, "ms_per_step": total / n, "tflops": tflops,
            "frac_of_bf16_sustained_peak": tflops / peaks["bf16_tflops_sustained"],
            "bf16_sustained_peak_tflops": peaks["bf16_tflops_sustained"], "clocks": clocks.summary(),
            "note": "steps back to back without an L2 flush (inputs 335 MB exceed L2), one event pair around all"}


def measure_training_cost(dev, w, reps=3):
    """What one ISM pass saves in training against a prefix-LM, which needs
    one sample per answer turn (history and query as a bidirectional prefix,
    then the answer): tokens, visible pairs and the measured fwd+bwd time of
    the same kernels on both batches (random values, same heads)."""
    import torch
    from paper_2408_00539_gb300 import ism
    out = {}
    for name, segs_np in (("ism_one_pass", w.segs), ("prefix_lm_triplets", wl.triplet_expansion(w.segs))):
        T = segs_np.total_tokens
        g = torch.Generator(device=dev).manual_seed(w.seed)
        q = torch.randn((T, w.num_heads_q, w.head_dim), generator=g, device=dev).mul_(w.value_std).bfloat16()
        k = torch.randn((T, w.num_heads_kv, w.head_dim), generator=g, device=dev).mul_(w.value_std).bfloat16()
        v = torch.randn((T, w.num_heads_kv, w.head_dim), generator=g, device=dev).mul_(w.value_std).bfloat16()
        do = torch.randn((T, w.num_heads_q, w.head_dim), generator=g, device=dev).bfloat16()
        segs = ism.Segments.from_workload(segs_np, dev)
        ms = []
        for it in range(reps + 1):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            o, lse = ism.fwd(segs, q, k, v, w.softmax_scale)
            ism.bwd(segs, q, k, v, o, lse, do, w.softmax_scale)
            e1.record()
            e1.synchronize()
            if it:
                ms.append(e0.elapsed_time(e1))
        ism.check_status(dev)
        out[name] = {"samples": segs_np.num_seqs, "tokens": T, "n_vis_pairs": n_visible(segs_np) * w.num_heads_q,
                     "fwd_bwd_ms": float(np.median(ms))}
        del q, k, v, do, o, lse
        torch.cuda.empty_cache()
    a, b = out["ism_one_pass"], out["prefix_lm_triplets"]
    out["tokens_ratio"] = b["tokens"] / a["tokens"]
    out["flops_ratio"] = b["n_vis_pairs"] / a["n_vis_pairs"]
    out["time_ratio"] = b["fwd_bwd_ms"] / a["fwd_bwd_ms"]
    return out


def measure_gemm_peaks(dev, n=8192, reps=20):
    """Dense e4m3 and bf16 GEMM rates of the library GEMMs (torch._scaled_mm and
    torch.matmul, i.e. cuBLASLt) on n x n x n products, timed back to back as a
    burst like the measured bf16 peak: the e4m3 forward's roofline takes the
    e4m3 figure, and the bf16 one shows how this run compares with the
    recorded peak.  None where the e4m3 GEMM is not available."""
    import torch
    out = {"n": n, "reps": reps}
    a = torch.randn(n, n, device=dev, dtype=torch.bfloat16)
    b = torch.randn(n, n, device=dev, dtype=torch.bfloat16)
    stream = torch.cuda.current_stream(dev)

    def rate(fn):
        for _ in range(3):
            fn()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        e1.synchronize()
        return 2.0 * n ** 3 * reps / (e0.elapsed_time(e1) * 1e-3) / 1e12

    out["bf16_tflops"] = rate(lambda: torch.matmul(a, b))
    try:
        a8 = a.to(torch.float8_e4m3fn)
        b8 = b.to(torch.float8_e4m3fn).t().contiguous().t()  # column-major second operand
        one = torch.tensor(1.0, device=dev)
        out["e4m3_tflops"] = rate(lambda: torch._scaled_mm(a8, b8, scale_a=one, scale_b=one, out_dtype=torch.bfloat16))
    except Exception as e:  # noqa: BLE001 - reported, the derived peak is used instead
        out["e4m3_tflops"] = None
        out["e4m3_error"] = str(e).splitlines()[0][:200]
    del a, b
    torch.cuda.empty_cache()
    return out


def measure_fwd_e4m3(dev, w, peaks, reps=10):
    """The forward on e4m3 copies of the workload's Q, K, V (per-tensor scales,
    fp8 tensor cores), against the bf16 forward of the same inputs; L2 flushed
    between calls, CUDA events around each."""
    import torch
    from paper_2408_00539_gb300 import ism
    q, k, v, _ = wl.attention_tensors(w)
    segs = ism.Segments.from_workload(w.segs, dev)
    qb, kb, vb = (t.to(dev) for t in (q, k, v))
    q8, k8, v8 = (wl.quantize_e4m3(t) for t in (qb, kb, vb))
    flush = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)

    def timed(fn):
        ms = []
        for it in range(reps + 2):
            flush.fill_(1)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn()
            e1.record(stream)
            e1.synchronize()
            if it >= 2:
                ms.append(e0.elapsed_time(e1))
        return float(np.median(ms))

    ms8 = timed(lambda: ism.fwd_e4m3(segs, q8[0], k8[0], v8[0], q8[1], k8[1], v8[1], w.softmax_scale))
    ms16 = timed(lambda: ism.fwd(segs, qb, kb, vb, w.softmax_scale))
    ism.check_status(dev)
    flops = 4 * w.head_dim * n_visible(w.segs) * w.num_heads_q
    tflops8 = flops / (ms8 * 1e-3) / 1e12
    gemm = measure_gemm_peaks(dev)
    derived = 2 * peaks["bf16_tflops"]  # e4m3 dense rate = 2x bf16 (nominal 4.5 vs 2.25 PFLOP/s)
    if gemm.get("e4m3_tflops"):
        peak8, kind = gemm["e4m3_tflops"], ("measured in this run: cuBLASLt e4m3 GEMM (torch._scaled_mm), "
                                            f"{gemm['n']}^3, {gemm['reps']} back to back")
    else:
        peak8, kind = derived, ("derived, not measured: measured bf16 burst peak x 2, the nominal dense "
                                "fp8/bf16 ratio (4.5 / 2.25 PFLOP/s)")
    return {"workload": w.name, "ms": ms8, "tflops": tflops8,
            "frac_of_e4m3_peak": tflops8 / peak8, "e4m3_peak_tflops": peak8, "e4m3_peak_kind": kind,
            "frac_of_derived_e4m3_peak": tflops8 / derived, "gemm_peaks_this_run": gemm,
            "bf16_fwd_ms": ms16, "speedup_over_bf16": ms16 / ms8,
            "note": "fwd call incl. metadata pass"}


def measure_append_e4m3(dev, a, kc, vc, qn, kn, vn, qd, kd, vd, flush, peaks, decode_steps=64):
    """The append-prefill and decode of ``measure_append`` with e4m3 queries
    and caches (per-tensor factors): fp8 tensor cores for the prefill, half
    the cache bytes for the decode."""
    import torch
    from paper_2408_00539_gb300 import ism
    _, ks = wl.quantize_e4m3(kc)
    _, vs = wl.quantize_e4m3(vc)
    k8, v8 = (kc.float() / ks).to(torch.float8_e4m3fn), (vc.float() / vs).to(torch.float8_e4m3fn)
    q8, qs = wl.quantize_e4m3(qn)
    kn8, vn8 = (kn.float() / ks).to(torch.float8_e4m3fn), (vn.float() / vs).to(torch.float8_e4m3fn)
    qd8, qds = wl.quantize_e4m3(qd)
    kd8, vd8 = (kd.float() / ks).to(torch.float8_e4m3fn), (vd.float() / vs).to(torch.float8_e4m3fn)
    B, hkv, d = kc.shape[0], kc.shape[2], kc.shape[3]
    c0 = a.cache_len.copy()
    cl = torch.from_numpy(c0.copy()).to(dev)
    stream = torch.cuda.current_stream(dev)
    pre_ms = []
    for it in range(8):
        cl.copy_(torch.from_numpy(c0))
        flush.fill_(1)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        ism.prefill_append_e4m3(q8, kn8, vn8, k8, v8, cl, c0, a.new_seg_end, a.new_seg_type, qs, ks, vs,
                                a.softmax_scale)
        e1.record(stream)
        e1.synchronize()
        if it >= 3:
            pre_ms.append(e0.elapsed_time(e1))
    c_host = c0 + a.l_new
    cl.copy_(torch.from_numpy(c_host))
    dec_kernel_us, dec_bytes = [], []
    for t in range(decode_steps):
        k0, k1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        for e in (k0, k1):
            e.record(stream)
        ism.set_kernel_timer(ism.KERNEL_DECODE, k0, k1)
        ism.prefill_append_e4m3(qd8, kd8, vd8, k8, v8, cl, c_host, [1], [1], qds, ks, vs, a.softmax_scale)
        k1.synchronize()
        ism.set_kernel_timer(ism.KERNEL_DECODE)
        dec_kernel_us.append(k0.elapsed_time(k1) * 1e3)
        dec_bytes.append(2 * B * (int(c_host[0]) + 1) * hkv * d)
        c_host = c_host + 1
    ism.check_status(dev)
    kus = float(np.median(dec_kernel_us[3:]))
    gbs = float(np.median(np.array(dec_bytes[3:]) / (np.array(dec_kernel_us[3:]) * 1e-6) / 1e9))
    return {"prefill_ms": float(np.median(pre_ms)), "decode_kernel_us": kus, "decode_hbm_gbs": gbs,
            "decode_frac_of_hbm": gbs / peaks["hbm_gbs"], "decode_steps": decode_steps,
            "note": "decode bytes = e4m3 K and V cache read once: 2*B*(c+1)*Hkv*D per step"}


def measure_session(dev):
    """A serving session in the shape of the paper's latency experiment
    (Section 3.6): per turn, the query is appended in one prefill call (the
    attention share of time to first token) and the answer generated by
    single-token decode calls (time per output token), the KV cache growing
    to the whole dialogue.  Each call is timed alone with CUDA events and a
    synchronise after it, as a generation loop must wait for its token.  The
    query turns run twice: under ISM (bidirectional query segment) and as a
    causal chunk, the comparison the paper makes between the ISM and the
    causal fine-tuned models."""
    import torch
    from paper_2408_00539_gb300 import ism
    s = wl.latency_session()
    B, hq, hkv, d, cap = s.batch, s.num_heads_q, s.num_heads_kv, s.head_dim, s.capacity
    g = torch.Generator(device=dev).manual_seed(s.seed)

    def rnd(*shape):
        return torch.randn(shape, generator=g, device=dev).mul_(s.value_std).bfloat16()

    kc, vc = rnd(B, cap, hkv, d), rnd(B, cap, hkv, d)
    qn, kn, vn = rnd(B, s.q_len, hq, d), rnd(B, s.q_len, hkv, d), rnd(B, s.q_len, hkv, d)
    qd, kd, vd = rnd(B, 1, hq, d), rnd(B, 1, hkv, d), rnd(B, 1, hkv, d)
    ws = torch.empty(max(ism.append_workspace_size(qn, kn, s.softmax_scale),
                         ism.append_workspace_size(qd, kd, s.softmax_scale)), dtype=torch.uint8, device=dev)
    o_pre, o_dec = torch.empty_like(qn), torch.empty_like(qd)
    l_pre = torch.empty((hq, B, s.q_len), dtype=torch.float32, device=dev)
    l_dec = torch.empty((hq, B, 1), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def timed(fn):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        fn()
        e1.record(stream)
        e1.synchronize()
        return e0.elapsed_time(e1)

    result = {}
    for mode, qtype in (("ism", wl.QUERY), ("causal", wl.ANSWER)):
        cl = torch.zeros((B,), dtype=torch.int32, device=dev)
        c_host = np.zeros((B,), dtype=np.int32)  # advanced in place: the prepared calls hold it
        prefill = ism.AppendStep(qn, kn, vn, kc, vc, cl, c_host, [s.q_len], [qtype], s.softmax_scale,
                                 out=o_pre, lse=l_pre, workspace=ws)
        decode = ism.AppendStep(qd, kd, vd, kc, vc, cl, c_host, [1], [wl.ANSWER], s.softmax_scale,
                                out=o_dec, lse=l_dec, workspace=ws)
        ttft, tpot = [], []
        for t in range(s.turns):
            ttft.append(timed(prefill))
            c_host += s.q_len
            if mode == "ism":
                turn = []
                for _ in range(s.a_len):
                    turn.append(timed(decode))
                    c_host += 1
                tpot.append(float(np.mean(turn)) * 1e3)
            else:  # the answer tokens' K / V are already in the cache from the first pass
                c_host += s.a_len
                cl.fill_(int(c_host[0]))
        ism.check_status(dev)
        result[mode] = (ttft, tpot)
    ttft_i, tpot = result["ism"]
    ttft_c, _ = result["causal"]
    return {"workload": s.name, "heads": f"{hq}/{hkv}", "head_dim": d,
            "context_tokens": s.capacity,
            "ttft_ms_ism": float(np.mean(ttft_i)), "ttft_ms_causal": float(np.mean(ttft_c)),
            "ttft_ism_over_causal": float(np.mean(ttft_i) / np.mean(ttft_c)),
            "ttft_ms_first_last_turn": [float(ttft_i[0]), float(ttft_i[-1])],
            "tpot_us": float(np.mean(tpot)), "tpot_us_first_last_turn": [tpot[0], tpot[-1]],
            "note": "one attention layer per call (query chunk: append plan, cache write, forward; answer token: cache "
                    "write, tensor-core decode, combine) through a prepared "
                    "ism.AppendStep (one C call a step); the first turn's calls include warm-up"}


def profile_decode(dtype: str, steps: int):
    """Only the single-token steps of the 8 x 16K cache workload (the decode of
    ``measure_append``), ``steps`` of them, printing nothing: for ncu.  bf16
    caches, or e4m3 ones with per-tensor factors."""
    import torch
    from paper_2408_00539_gb300 import ism
    dev = "cuda:0"
    a = wl.append_16k()
    B, cap, hq, hkv, d = a.batch, a.capacity, a.num_heads_q, a.num_heads_kv, a.head_dim
    g = torch.Generator(device=dev).manual_seed(a.seed)

    def rnd(shape):
        x = torch.randn(shape, generator=g, device=dev).mul_(a.value_std)
        return x.to(torch.float8_e4m3fn) if dtype == "e4m3" else x.bfloat16()
    kc, vc = rnd((B, cap, hkv, d)), rnd((B, cap, hkv, d))
    qd, kd, vd = rnd((B, 1, hq, d)), rnd((B, 1, hkv, d)), rnd((B, 1, hkv, d))
    c_host = a.cache_len.copy() + a.l_new
    cl = torch.from_numpy(c_host.copy()).to(dev)
    for _ in range(steps):
        if dtype == "e4m3":
            ism.prefill_append_e4m3(qd, kd, vd, kc, vc, cl, c_host, [1], [1], 1.0, 1.0, 1.0, a.softmax_scale)
        else:
            ism.prefill_append(qd, kd, vd, kc, vc, cl, c_host, [1], [1], a.softmax_scale)
        c_host = c_host + 1
    torch.cuda.synchronize()
    ism.check_status(dev)


WORKLOADS = {"gqa_8k": wl.gqa_8k, "mha_4k": wl.mha_4k, "packed_32k": wl.packed_32k,
             # one 4K dialogue of the same recipes: small enough for full ncu captures
             "gqa_4k_b1": lambda: wl.gqa_8k(batch=1, seqlen=4096),
             "mha_4k_b1": lambda: wl.mha_4k(batch=1),
             # one long dialogue (few hundred turns): with --min-workspace, the recompute schedule
             "long_32k": lambda: wl.long_dialogue(32768)}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="cuda", choices=["cuda", "reference"])
    ap.add_argument("--workload", default="gqa_8k", choices=sorted(WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-append", action="store_true", help="skip the append-prefill / decode measurement")
    ap.add_argument("--no-extra", action="store_true",
                    help="skip the sustained run, the minimum-workspace backward and the other training configs")
    ap.add_argument("--profile-step", action="store_true",
                    help="run the warm-up steps and one more step, print nothing (for ncu)")
    ap.add_argument("--rope", action="store_true", help="with --profile-step: the rotary forward and backward")
    ap.add_argument("--e4m3", action="store_true", help="with --profile-step: the e4m3 forward alone")
    ap.add_argument("--min-workspace", action="store_true",
                    help="backward with the minimum workspace (recompute schedule) in the headline step")
    ap.add_argument("--profile-decode", choices=["bf16", "e4m3"],
                    help="run only warm-up + steps single-token steps on the 8 x 16K cache, print nothing (for ncu)")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    if args.profile_decode:
        profile_decode(args.profile_decode, args.warmup + args.steps)
        return
    w = WORKLOADS[args.workload]()
    if args.impl == "reference":
        run_reference(args, w)
    else:
        run_cuda(args, w)


if __name__ == "__main__":
    main()
