"""Benchmark of the WISE attention hot path on one or more GB300s.

One benchmark step is one recurrent trajectory of the 4K workload (batch 1,
L=4096, 32 heads, head_dim 128, block 128, T=32): the discovery steps run
dense attention with the block-mass epilogue, one selection builds the
support (sink + diagonal + 95% mass coverage, cap 8), and every late step runs
support-restricted attention.  Every step of the trajectory has its own
Q/K/V (2.9 GB in total, far above the 129 MB L2), resident in HBM before the
timed region starts.

Reported (one JSON line on rank 0):
  value            late-step attention ms per recurrent step (sparse kernel,
                   CUDA events on the launching stream around the late steps
                   after the first, which run back to back as in the
                   trajectory, divided by their number; mean over trajectories)
  dense_ms         the library's own dense kernel (no mass) on the same late
                   inputs, timed the same way; speedup = dense_ms / value
  discovery_ms     the dense kernel with the block-mass epilogue on the
                   discovery steps' inputs, timed the same way (as many
                   launches as dense_ms); discovery_event_ms keeps the events
                   around each discovery step of the timed trajectories
  roofline         the sparse kernel's algorithmic tensor FLOPs per launch
                   over its mean launch time, against the measured bf16 peak
  e2e              the same late step through the C ABI with Q/K/V copied from
                   pinned host memory and O copied back inside the timed region
  cpu_baseline     the fp64 oracle timed on a bounded sample on the host cores
Multi-GPU: every rank runs an independent replica (the path has no exchange
step).  Times are maxima over ranks; in that time the job completes one step
per rank, so `value` and `e2e` (ms per late step of the whole job) are the
maximum divided by the number of ranks, while ms_per_step, dense_ms, the
speedups and the roofline stay per replica.

--impl reference times the fp64 oracle (the reference arm of this build) on
a bounded sample of the same workload.
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
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

WORKLOAD = "4k"
METRIC = "late-step attention ms/step (sparse, 4K)"
WORKLOAD_DESC = ("4k: batch 1, L=4096, 32 heads, head_dim 128, block 128, T=32, discovery 0-3, "
                 "sink+diagonal+95% coverage cap 8")
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def sparse_traffic_bytes():
    """DRAM bytes per launch of the sparse kernel from the committed ncu
    summary, or None when the kernel source changed since that capture."""
    import hashlib
    src = os.path.join(ROOT, "paper_2609_27373_gb300", "csrc", "attn_kernel.cuh")
    prof = os.path.join(ROOT, "profiles", "attn_sparse_4k.md")
    try:
        sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        fields = dict(line.split(":", 1) for line in open(prof) if line.count(":") == 1 and " " not in line.split(":")[0])
    except (OSError, ValueError):
        return None
    if fields.get("source_sha256_16", "").strip() != sha:
        return None
    try:
        return int(fields["traffic_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


def aggregate_over_ranks(values, world, device="cpu"):
    """Per-rank times (ms) -> (max over ranks, whole-job time per step).

    Every rank runs an independent replica, so in the slowest rank's time the
    job completes `world` steps: the job's time per step is max / world.  With
    world > 1 the process group must be initialised (NCCL with CUDA tensors,
    gloo with CPU tensors)."""
    import torch
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    mx = [float(x) for x in t.tolist()]
    return mx, [v / world for v in mx]


def load_peaks():
    try:
        with open(PEAKS_FILE) as f:
            d = json.load(f)
        return d, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


# --------------------------------------------------------------------------- FLOP accounting

def pair_count(block: int, diagonal: bool) -> int:
    """Query-key pairs of one (query block, key block) tile: B^2 off the
    diagonal, B(B+1)/2 on it (causal mask, Eq. 2)."""
    return block * (block + 1) // 2 if diagonal else block * block


def sparse_flops(idx: np.ndarray, counts: np.ndarray, n_heads: int, head_dim: int, block: int) -> float:
    """4*d FLOPs (QK^T and PV) per computed query-key pair over the support."""
    B, Hkv, nb, _ = idx.shape
    group = n_heads // Hkv
    total = 0
    for b in range(B):
        for g in range(Hkv):
            for q in range(nb):
                for kb in idx[b, g, q, : counts[b, g, q]]:
                    total += pair_count(block, kb == q)
    return 4.0 * head_dim * total * group


def dense_flops(batch: int, n_heads: int, seqlen: int, head_dim: int) -> float:
    return 4.0 * head_dim * batch * n_heads * seqlen * (seqlen + 1) / 2


# --------------------------------------------------------------------------- clocks

class ClockSampler:
    """Samples SM clocks and throttle reasons with nvidia-smi while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, path: str):
        self.path = path
        self.proc = None
        try:
            self.f = open(path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(gpu_index), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax.append(float(parts[2]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower().startswith("active"):
                        reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# --------------------------------------------------------------------------- oracle (CPU) arm

def oracle_late_step_ms(wl, late_inputs, idx, counts, n_heads_sample: int):
    """fp64 oracle on `n_heads_sample` heads of one late step, scaled to the
    full step (work is uniform across heads).  Returns (ms, cores, seconds)."""
    from oracle import oracle as orc
    Q, K, V = late_inputs
    units = [(b, h, q) for b in range(wl.batch) for h in range(n_heads_sample) for q in range(wl.n_blocks)]
    t0 = time.perf_counter()
    orc.sparse_attention(Q, K, V, idx, counts, wl.block, units=units)
    sec = time.perf_counter() - t0
    scale = (wl.batch * wl.n_heads * wl.n_blocks) / len(units)
    return 1e3 * sec * scale, orc.max_threads(), sec


def run_reference(args):
    """Reference arm: the fp64 oracle runs the same trajectory on the host
    cores (its own discovery masses and selection), and each timed step is
    one whole late step of the 4K workload."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    from oracle import oracle as orc
    from paper_2609_27373_gb300 import synth
    wl = synth.WORKLOADS[WORKLOAD]
    traj = synth.Trajectory(wl)
    mass = None
    for t in range(wl.n_discovery):
        Q, K, V = traj.step(t)
        _, m = orc.full_attention(Q, K, V, wl.block, with_mass=True)
        mass = m if mass is None else mass + m
    idx, counts = orc.select_support(mass.astype(np.float32), wl.n_kv_heads, wl.block, wl.sel_mode, wl.n_sink,
                                     wl.n_local, wl.topk, wl.eta, wl.cap)
    Q, K, V = traj.step(wl.n_discovery)
    times = []
    for s in range(args.warmup + args.steps):
        ms, cores, _ = oracle_late_step_ms(wl, (Q, K, V), idx, counts, wl.n_heads)
        if s >= args.warmup:
            times.append(ms)
    value = statistics.median(times)
    line = {
        "impl": "reference", "metric": METRIC, "value": value,
        "unit": "ms", "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": value, "higher_is_better": False, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD_DESC, "parallelism": "replicas x1"},
        "cpu_baseline": {"value": value, "unit": "ms", "cores": cores, "kind": "oracle",
                         "sample": "one whole late step of the 4K workload per timed step"},
        "e2e": {"value": value, "unit": "ms", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


# --------------------------------------------------------------------------- GPU arm

def run_profile_sequence(name=WORKLOAD):
    """Fixed launch sequence for profilers: n_discovery dense+mass launches,
    one selection, two sparse launches and one plain dense launch of a
    workload, then (4K workload only) one Freeze-A store and two
    stored-Freeze-A P V launches (about 1 GB on the device at 4K, under 1.5 GB
    for the other workloads)."""
    import torch
    from paper_2609_27373_gb300 import synth, wise
    wl = synth.WORKLOADS[name]
    shape, sel = wise.shape_of(wl), wise.select_of(wl)
    layer = wise.WiseAttention(shape, sel, wl.n_discovery)
    traj = synth.Trajectory(wl)
    for t in range(wl.n_discovery + 1):
        Q, K, V = (torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).cuda() for x in traj.step(t))
        O = torch.empty_like(Q)
        layer.step(t, Q, K, V, O)
    wise.wise_sparse_attn(shape, Q, K, V, layer.idx, layer.counts, O)
    wise.wise_full_attn_accumulate(shape, Q, K, V, O)
    if name != WORKLOAD:
        status = wise.wise_get_status()
        if status != wise.WISE_OK:
            raise RuntimeError(wise.status_string(status))
        return 0
    # Freeze-A with the distribution stored once, then two late-step P V launches
    n_units = wl.batch * wl.n_heads * (wl.seqlen // 128)
    P = torch.empty((n_units, wise.freeze_tile_cap(shape, wl.cap), 128, 128), dtype=torch.bfloat16, device="cuda")
    inv_l = torch.empty((n_units, 128), dtype=torch.float32, device="cuda")
    wise.wise_freeze_a_probs(shape, Q, K, layer.idx, layer.counts, P, inv_l)
    for _ in range(2):
        wise.wise_frozen_pv(shape, P, inv_l, V, layer.idx, layer.counts, O)
    status = wise.wise_get_status()
    if status != wise.WISE_OK:
        raise RuntimeError(wise.status_string(status))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--clocks-dir", default=None,
                    help="directory for the nvidia-smi clock samples of the timed region (default: the temp dir)")
    ap.add_argument("--profile", action="store_true",
                    help="no timing: the 4K discovery steps, one selection, then 2 late sparse and 1 dense launches "
                         "(a small, fixed launch sequence for ncu captures)")
    ap.add_argument("--profile-workload", default=WORKLOAD,
                    help="workload of --profile (4k, 4k_b32, 4k_b4_d96, 16k, 32k_gqa, tiny)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("at least 3 warm-up steps")
    if args.impl == "reference":
        return run_reference(args)
    if args.profile:
        return run_profile_sequence(args.profile_workload)

    import torch
    import torch.distributed as dist
    from paper_2609_27373_gb300 import synth, wise

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    def barrier():
        if world > 1:
            dist.barrier()

    wl = synth.WORKLOADS[WORKLOAD]
    shape, sel = wise.shape_of(wl), wise.select_of(wl)
    n_late = wl.steps - wl.n_discovery

    # ---- inputs: the whole trajectory, generated on the host, resident in HBM
    traj = synth.Trajectory(wl)
    host_steps, dev_steps = [], []
    for t in range(wl.steps):
        q, k, v = traj.step(t)
        host_steps.append((q, k, v))
        dev_steps.append(tuple(torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).cuda() for x in (q, k, v)))
    O = torch.empty(host_steps[0][0].shape, dtype=torch.bfloat16, device="cuda")
    layer = wise.WiseAttention(shape, sel, wl.n_discovery)
    stream = torch.cuda.current_stream()

    def per_call_ms(calls):
        """Mean time per call of `calls` run back to back on the stream between
        one pair of CUDA events.  Consecutive attention launches overlap their
        set-up with the end of the previous one (programmatic dependent
        launch), as they do in a trajectory; an event recorded between two
        launches would keep them apart."""
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for c in calls:
            c()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / len(calls)

    def trajectory(ev=None):
        """One trajectory.  With `ev`: events around each discovery step and the
        first late step (it also runs the selection), then one pair around the
        remaining late steps, which run back to back."""
        layer.selected = False
        for t in range(wl.steps):
            Q, K, V = dev_steps[t]
            if ev is not None and t <= wl.n_discovery + 1:
                ev[t][0].record(stream)
            layer.step(t, Q, K, V, O)
            if ev is not None and t <= wl.n_discovery:
                ev[t][1].record(stream)
        if ev is not None:
            ev[wl.n_discovery + 1][1].record(stream)

    for _ in range(args.warmup):
        trajectory()
    torch.cuda.synchronize()
    idx_h, counts_h = layer.idx.cpu().numpy(), layer.counts.cpu().numpy()
    flops_sparse = sparse_flops(idx_h, counts_h, wl.n_heads, wl.head_dim, wl.block)
    flops_dense = dense_flops(wl.batch, wl.n_heads, wl.seqlen, wl.head_dim)
    density = flops_sparse / flops_dense

    clocks = ClockSampler(local, os.path.join(args.clocks_dir or tempfile.gettempdir(), f"wise_clocks_rank{rank}.csv"))
    time.sleep(0.3)

    # ---- timed: K trajectories
    evs = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(wl.steps)]
           for _ in range(args.steps)]
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    t_start.record(stream)
    for k in range(args.steps):
        trajectory(evs[k])
    t_end.record(stream)
    torch.cuda.synchronize()
    barrier()
    total_ms = t_start.elapsed_time(t_end)
    disc_ms, sel_ms, late_ms = [], [], []
    for k in range(args.steps):
        for t in range(wl.n_discovery):
            disc_ms.append(evs[k][t][0].elapsed_time(evs[k][t][1]))
        # the late steps after the first, back to back (the first also ran the
        # selection: timed alone below)
        late_ms.append(evs[k][wl.n_discovery + 1][0].elapsed_time(evs[k][wl.n_discovery + 1][1]) / (n_late - 1))
    # the first late step also ran the selection; time the selection alone
    sel_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    for k in range(args.steps):
        sel_ev[k][0].record(stream)
        wise.wise_select_support(shape, sel, layer.blockmass, layer.idx, layer.counts)
        sel_ev[k][1].record(stream)
    torch.cuda.synchronize()
    sel_ms = [a.elapsed_time(b) for a, b in sel_ev]
    late_only = late_ms  # late steps without the selection

    # ---- own dense kernel on the same late inputs
    dense_calls = [lambda t=t: wise.wise_full_attn_accumulate(shape, *dev_steps[t], O)
                   for t in range(wl.n_discovery, wl.steps)]
    dense_ms = [per_call_ms(dense_calls) for _ in range(max(1, args.steps // 2))]

    # ---- the discovery steps back to back, as they run in a trajectory (the
    # per-step events above keep consecutive launches apart), timed like the
    # dense baseline: as many launches (passes over the discovery steps' own
    # inputs), into a scratch mass so that the layer's own stays as selected
    disc_mass = torch.zeros_like(layer.blockmass)
    disc_calls = [lambda t=t % wl.n_discovery: wise.wise_full_attn_accumulate(shape, *dev_steps[t], O, disc_mass, t)
                  for t in range(len(dense_calls))]
    disc_b2b_ms = [per_call_ms(disc_calls) for _ in range(max(1, args.steps // 2))]

    # ---- end to end through host buffers (pinned), late steps
    pinned = [tuple(torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).pin_memory() for x in host_steps[t])
              for t in range(wl.n_discovery, min(wl.steps, wl.n_discovery + 4))]
    # Pipelined over steps like a serving loop: step i's inputs are copied in
    # on one stream while step i-1 computes and step i-2's output is copied
    # out on a third; device inputs and outputs are double-buffered.  Every
    # step's copies stay inside the timed region.
    O_host = [torch.empty(O.shape, dtype=torch.bfloat16).pin_memory() for _ in range(2)]
    dev_in = [tuple(torch.empty_like(x) for x in dev_steps[0]) for _ in range(2)]
    dev_out = [torch.empty_like(O) for _ in range(2)]
    h2d = sum(x.numel() * x.element_size() for x in pinned[0])
    d2h = O_host[0].numel() * O_host[0].element_size()
    e2e_iters = max(8, args.steps)
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    ev_in = [torch.cuda.Event() for _ in range(e2e_iters)]
    ev_done = [torch.cuda.Event() for _ in range(e2e_iters)]
    ev_out = [torch.cuda.Event() for _ in range(e2e_iters)]
    e_start, e_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    e_start.record(stream)
    s_in.wait_stream(stream)
    s_out.wait_stream(stream)
    for i in range(e2e_iters):
        buf = i & 1
        hq, hk, hv = pinned[i % len(pinned)]
        with torch.cuda.stream(s_in):
            if i >= 2:
                s_in.wait_event(ev_done[i - 2])  # step i-2 no longer reads this input buffer
            for dst, src in zip(dev_in[buf], (hq, hk, hv)):
                dst.copy_(src, non_blocking=True)
            ev_in[i].record(s_in)
        stream.wait_event(ev_in[i])
        if i >= 2:
            stream.wait_event(ev_out[i - 2])  # step i-2's output has been copied out
        wise.wise_sparse_attn(shape, *dev_in[buf], layer.idx, layer.counts, dev_out[buf], stream=stream)
        ev_done[i].record(stream)
        with torch.cuda.stream(s_out):
            s_out.wait_event(ev_done[i])
            O_host[buf].copy_(dev_out[buf], non_blocking=True)
            ev_out[i].record(s_out)
    stream.wait_stream(s_in)
    stream.wait_stream(s_out)
    e_end.record(stream)
    torch.cuda.synchronize()
    e2e_ms = e_start.elapsed_time(e_end) / e2e_iters

    # ---- sparse kernel with every admissible block (the matched-backend row)
    nb = shape.n_blocks
    all_idx, all_counts = synth.all_blocks_support(wl.batch, wl.n_kv_heads, nb)
    all_idx, all_counts = torch.from_numpy(all_idx).cuda(), torch.from_numpy(all_counts).cuda()
    all_blocks_ms = per_call_ms([lambda t=t: wise.wise_sparse_attn(shape, *dev_steps[t], all_idx, all_counts, O)
                                 for t in range(wl.n_discovery, wl.steps)])

    # ---- routing diagnostic: share of each late step's full attention kept
    # by the frozen support (the step's own block mass, then the support sum)
    diag_mass = torch.empty((wl.batch, wl.n_heads, nb, nb), dtype=torch.float32, device="cuda")
    retained = torch.empty((wl.batch, wl.n_heads, nb), dtype=torch.float32, device="cuda")
    ret = []
    for t in range(wl.n_discovery, wl.steps, 4):
        Q, K, V = dev_steps[t]
        wise.wise_full_attn_accumulate(shape, Q, K, V, O, diag_mass, 0)
        wise.wise_support_mass(shape, diag_mass, layer.idx, layer.counts, retained)
        ret.append(float(retained.mean()))
    retained_mass = statistics.mean(ret)

    # ---- the paper's own working set (union over the discovery window of each
    # step's 95 % coverage set, Eq. 6) and the intervention controls, each with
    # its density, retained late-step mass and late-step sparse time
    step_mass = torch.empty((wl.n_discovery, wl.batch, wl.n_heads, nb, nb), dtype=torch.float32, device="cuda")
    for t in range(wl.n_discovery):
        wise.wise_full_attn_accumulate(shape, *dev_steps[t], O, step_mass[t], 0)
    ws_idx = {k: torch.empty((wl.batch, wl.n_kv_heads, nb, nb), dtype=torch.int32, device="cuda")
              for k in ("union", "static", "mass_matched", "size_matched")}
    ws_cnt = {k: torch.empty((wl.batch, wl.n_kv_heads, nb), dtype=torch.int32, device="cuda") for k in ws_idx}
    forced = dict(n_sink=wl.n_sink, n_local=wl.n_local)
    wise.wise_select_working_set(shape, wise.WS_UNION, step_mass, ws_idx["union"], ws_cnt["union"], eta=wl.eta,
                                 **forced)
    wise.wise_select_working_set(shape, wise.WS_STATIC, step_mass[:1], ws_idx["static"], ws_cnt["static"],
                                 eta=wl.eta, **forced)
    for k, mode in (("mass_matched", wise.WS_MASS_MATCHED), ("size_matched", wise.WS_SIZE_MATCHED)):
        wise.wise_select_working_set(shape, mode, step_mass[:1], ws_idx[k], ws_cnt[k], ref_idx=ws_idx["union"],
                                     ref_counts=ws_cnt["union"], **forced)
    admissible = wl.batch * wl.n_kv_heads * nb * (nb + 1) / 2
    supports = {}
    for k in ws_idx:
        rm = []
        for t in range(wl.n_discovery, wl.steps, 4):
            wise.wise_full_attn_accumulate(shape, *dev_steps[t], O, diag_mass, 0)
            wise.wise_support_mass(shape, diag_mass, ws_idx[k], ws_cnt[k], retained)
            rm.append(float(retained.mean()))
        sp_k = per_call_ms([lambda t=t, k=k: wise.wise_sparse_attn(shape, *dev_steps[t], ws_idx[k], ws_cnt[k], O)
                            for t in range(wl.n_discovery, wl.steps)])
        supports[k] = {"density": round(float(ws_cnt[k].sum()) / admissible, 4),
                       "retained_mass": round(statistics.mean(rm), 4),
                       "sparse_ms": round(sp_k, 5)}

    # ---- stability of the rolling working set at the discovery endpoint
    # (appendix "Stability of the Deployed Working Set"): W(t) = union of the
    # eta sets of steps t-3..t; Jaccard of W(t_d - 1) and W(t_d)
    roll = []
    for t in (wl.n_discovery - 2, wl.n_discovery - 1):
        r_idx = torch.empty((wl.batch, wl.n_kv_heads, nb, nb), dtype=torch.int32, device="cuda")
        r_cnt = torch.empty((wl.batch, wl.n_kv_heads, nb), dtype=torch.int32, device="cuda")
        wise.wise_select_working_set(shape, wise.WS_UNION, step_mass[max(0, t - 3):t + 1].contiguous(), r_idx, r_cnt,
                                     eta=wl.eta, **forced)
        roll.append((r_idx, r_cnt))
    inter_union = torch.empty((wl.batch, 2), dtype=torch.int64, device="cuda")
    wise.wise_support_overlap(shape, roll[0][0], roll[0][1], roll[1][0], roll[1][1], inter_union)
    rolling_jaccard = statistics.mean(1.0 if u == 0 else i / u for i, u in inter_union.cpu().tolist())

    # ---- Freeze-A control: the selected support with the within-support
    # distribution of the last discovery step, applied to each late step's V
    Q_td, K_td, _ = dev_steps[wl.n_discovery - 1]
    freeze_a_ms = per_call_ms([lambda t=t: wise.wise_freeze_a_attn(shape, Q_td, K_td, dev_steps[t][2], layer.idx,
                                                                   layer.counts, O)
                               for t in range(wl.n_discovery, wl.steps)])

    # ---- Freeze-A with the distribution stored once (row-max-relative bf16
    # tiles + 1/sum per row) and a block-sparse P V product per late step:
    # HBM-bound, reported against the measured copy bandwidth
    n_units = wl.batch * wl.n_heads * (wl.seqlen // 128)
    tile_cap = wise.freeze_tile_cap(shape, wl.cap)
    P_frz = torch.empty((n_units, tile_cap, 128, 128), dtype=torch.bfloat16, device="cuda")
    inv_l = torch.empty((n_units, 128), dtype=torch.float32, device="cuda")
    pr_ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    wise.wise_freeze_a_probs(shape, Q_td, K_td, layer.idx, layer.counts, P_frz, inv_l)  # warm-up
    pr_ev[0].record(stream)
    wise.wise_freeze_a_probs(shape, Q_td, K_td, layer.idx, layer.counts, P_frz, inv_l)
    pr_ev[1].record(stream)
    pv_calls = [lambda t=t: wise.wise_frozen_pv(shape, P_frz, inv_l, dev_steps[t][2], layer.idx, layer.counts, O)
                for t in range(wl.n_discovery, wl.steps)]
    per_call_ms(pv_calls)  # warm-up
    frozen_pv_ms = per_call_ms(pv_calls)
    # Algorithmic bytes per launch: the stored tiles of every walk, V once
    # (every key block is selected by some query tile of its head), O, inv_l.
    walk_tiles = 0
    for b in range(wl.batch):
        for g in range(wl.n_kv_heads):
            for q in range(nb):
                walk_tiles += int(counts_h[b, g, q])  # block 128: one tile per list entry
    walk_tiles *= wl.n_heads // wl.n_kv_heads
    v_bytes = wl.batch * wl.n_kv_heads * wl.seqlen * wl.head_dim * 2
    o_bytes = wl.batch * wl.n_heads * wl.seqlen * wl.head_dim * 2
    frz_bytes = walk_tiles * 128 * 128 * 2 + v_bytes + o_bytes + n_units * 128 * 4
    hbm_peak = float(load_peaks()[0]["hbm_gbs"])
    frz_gbs = frz_bytes / (frozen_pv_ms * 1e-3) / 1e9
    frozen = {"store_ms": round(pr_ev[0].elapsed_time(pr_ev[1]), 5), "pv_ms": round(frozen_pv_ms, 5),
              "pv_roofline": {"bound": "hbm", "achieved": round(frz_gbs, 1), "peak": hbm_peak, "unit": "GB/s",
                              "frac": round(frz_gbs / hbm_peak, 4), "bytes_per_launch": frz_bytes},
              "stored_bytes": P_frz.numel() * 2 + inv_l.numel() * 4}
    del P_frz, inv_l

    # ---- the paper's default block of 32 keys: the 4K workload at B = 32 with
    # the same key budget per query block, its own discovery and selection,
    # then late steps timed.  Kernels compute 128 x 128 tiles with 4 x 4
    # sub-block masks, so `tile_density` (tiles touched / causal tiles) is the
    # share of tensor work against the dense kernel.
    wl32 = synth.WORKLOADS["4k_b32"]
    shape32, sel32 = wise.shape_of(wl32), wise.select_of(wl32)
    layer32 = wise.WiseAttention(shape32, sel32, wl32.n_discovery)
    traj32 = synth.Trajectory(wl32)
    late32 = 8
    steps32 = [tuple(torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).cuda() for x in traj32.step(t))
               for t in range(wl32.n_discovery + late32)]
    O32 = torch.empty_like(steps32[0][0])
    for t in range(wl32.n_discovery + 1):
        layer32.step(t, *steps32[t], O32)
    calls32 = [lambda t=t: wise.wise_sparse_attn(shape32, *steps32[t], layer32.idx, layer32.counts, O32)
               for t in range(wl32.n_discovery, wl32.n_discovery + late32)]
    per_call_ms(calls32)  # warm-up
    b32_ms = per_call_ms(calls32)
    i32, c32 = layer32.idx.cpu().numpy(), layer32.counts.cpu().numpy()
    f32 = sparse_flops(i32, c32, wl32.n_heads, wl32.head_dim, wl32.block)
    tiles32 = 0
    for b in range(wl32.batch):
        for g in range(wl32.n_kv_heads):
            for qt in range(wl32.n_blocks // 4):
                tiles32 += len({int(v) // 4 for q in range(4 * qt, 4 * qt + 4) for v in i32[b, g, q, :c32[b, g, q]]})
    causal_tiles = wl32.batch * wl32.n_kv_heads * (wl32.seqlen // 128) * (wl32.seqlen // 128 + 1) // 2
    block32 = {"workload": "4k_b32: the 4K workload at block 32, sink+diagonal+95% coverage cap 32",
               "late_ms": round(b32_ms, 5), "tflops_effective": round(f32 / (b32_ms * 1e-3) / 1e12, 2),
               "density": round(f32 / dense_flops(wl32.batch, wl32.n_heads, wl32.seqlen, wl32.head_dim), 4),
               "tile_density": round(tiles32 / causal_tiles, 4), "speedup_vs_dense": round(statistics.mean(dense_ms) / b32_ms, 4)}
    del steps32, layer32, O32

    # ---- the other benchmark workloads at their full sizes: own discovery
    # and selection, then late steps timed against the dense kernel on the
    # same inputs (context for the 4K line; parity is tested separately)
    other = {}
    for name in ("tiny", "4k_b4_d96", "16k", "32k_gqa"):
        wo = synth.WORKLOADS[name]
        sh_o, sel_o = wise.shape_of(wo), wise.select_of(wo)
        lay_o = wise.WiseAttention(sh_o, sel_o, wo.n_discovery)
        tr_o = synth.Trajectory(wo)
        n_t = 4
        st_o = [tuple(torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).cuda() for x in tr_o.step(t))
                for t in range(wo.n_discovery + n_t)]
        O_o = torch.empty_like(st_o[0][0])
        for t in range(wo.n_discovery + 1):
            lay_o.step(t, *st_o[t], O_o)
        sp_calls = [lambda t=t: wise.wise_sparse_attn(sh_o, *st_o[t], lay_o.idx, lay_o.counts, O_o)
                    for t in range(wo.n_discovery, wo.n_discovery + n_t)]
        dn_calls = [lambda t=t: wise.wise_full_attn_accumulate(sh_o, *st_o[t], O_o)
                    for t in range(wo.n_discovery, wo.n_discovery + n_t)]
        per_call_ms(sp_calls + dn_calls)  # warm-up
        sp = per_call_ms(sp_calls)
        dn = per_call_ms(dn_calls)
        f_o = sparse_flops(lay_o.idx.cpu().numpy(), lay_o.counts.cpu().numpy(), wo.n_heads, wo.head_dim, wo.block)
        other[name] = {"late_ms": round(sp, 5), "dense_ms": round(dn, 5), "speedup_vs_dense": round(dn / sp, 4),
                       "tflops_effective": round(f_o / (sp * 1e-3) / 1e12, 2),
                       "density": round(f_o / dense_flops(wo.batch, wo.n_heads, wo.seqlen, wo.head_dim), 4)}
        del st_o, lay_o, O_o

    # ---- the whole trajectory as one CUDA graph (discovery, selection, late
    # steps), replayed; its launches carry no host-side gaps
    graph = {"ms": None, "note": None}
    try:
        for _ in range(2):
            trajectory()
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            trajectory()
        g.replay()
        torch.cuda.synchronize()
        g_start, g_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        reps = max(3, args.steps // 2)
        g_start.record(stream)
        for _ in range(reps):
            g.replay()
        g_end.record(stream)
        torch.cuda.synchronize()
        graph["ms"] = g_start.elapsed_time(g_end) / reps
    except Exception as exc:  # report, do not fail the bench line
        graph["note"] = f"capture failed: {type(exc).__name__}: {exc}"[:200]
    clk = clocks.stop()
    status = wise.wise_get_status()
    if status != wise.WISE_OK:
        raise RuntimeError(f"kernel status: {wise.status_string(status)}")

    dense = statistics.mean(dense_ms)
    # max over ranks; `value` and `e2e` are per late step of the whole job
    (rank_value, step_ms, rank_e2e), (value, _, e2e_ms) = aggregate_over_ranks(
        [statistics.mean(late_only), total_ms / args.steps, e2e_ms], world, device="cuda")

    peaks, peak_kind = load_peaks()
    peak = float(peaks["bf16_tflops"])
    achieved = flops_sparse / (rank_value * 1e-3) / 1e12  # per GPU: one replica's kernel
    launches = args.steps * (wl.steps + 1)  # n_discovery dense + 1 select + n_late sparse per trajectory

    line = {
        "metric": METRIC,
        "value": round(value, 5),
        "unit": "ms",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(step_ms, 4),
        "higher_is_better": False,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": WORKLOAD_DESC,
                   "step": "one T=32 trajectory: 4 dense+mass, 1 selection, 28 sparse",
                   "l2": "every recurrent step has its own Q/K/V (2.9 GB rotating, > L2)",
                   "parallelism": f"replicas x{world}"},
        "dense_ms": round(dense, 5),
        "speedup_vs_dense": round(dense / rank_value, 4),
        "setup_inclusive_speedup": round(n_late * dense / (statistics.mean(sel_ms) + n_late * rank_value), 4),
        "trajectory_speedup": round(wl.steps * dense / step_ms, 4),
        "discovery_ms": round(statistics.mean(disc_b2b_ms), 5),
        "discovery_event_ms": round(statistics.mean(disc_ms), 5),
        "select_ms": round(statistics.mean(sel_ms), 5),
        "tflops_effective": round(achieved, 2),
        "dense_tflops": round(flops_dense / (dense * 1e-3) / 1e12, 2),
        "density": round(density, 4),
        "retained_mass": round(retained_mass, 4),
        "all_blocks_ms": round(all_blocks_ms, 5),
        "block_density": round(float(layer.counts.sum()) / (wl.batch * wl.n_kv_heads * nb * (nb + 1) / 2), 4),
        "supports": supports,
        "rolling_jaccard_at_discovery_end": round(rolling_jaccard, 4),
        "block32": block32,
        "other_workloads": other,
        "freeze_a_ms": round(freeze_a_ms, 5),
        "freeze_a_stored": frozen,
        "all_blocks_vs_dense": round(all_blocks_ms / dense, 4),
        "graph_trajectory_ms": None if graph["ms"] is None else round(graph["ms"], 4),
        "graph_trajectory_speedup": None if graph["ms"] is None else round(wl.steps * dense / graph["ms"], 4),
        **({"graph_note": graph["note"]} if graph["note"] else {}),
        "roofline": {"bound": "tensor", "achieved": round(achieved, 2), "peak": peak, "unit": "TFLOP/s",
                     "frac": round(achieved / peak, 4), "traffic": sparse_traffic_bytes(),
                     "peak_kind": f"{peak_kind} bf16 burst", "kernel": "wise_sparse_attn"},
        "e2e": {"value": round(e2e_ms, 5), "unit": "ms", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "pipeline": "H2D, compute and D2H of consecutive late steps overlapped on three streams"},
        "gpu_launches": launches,
        "clocks": clk,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        # whole late steps (all heads) until about 10 s of CPU time are spent
        per, spent, n = [], 0.0, 0
        while spent < 10.0 and n < n_late:
            ms, cores, sec = oracle_late_step_ms(wl, host_steps[wl.n_discovery + n], idx_h, counts_h, wl.n_heads)
            per.append(ms)
            spent += sec
            n += 1
        line["cpu_baseline"] = {"value": round(statistics.mean(per), 1), "unit": "ms", "cores": cores,
                                "kind": "oracle",
                                "sample": f"{n} whole late steps of the 4K workload ({spent:.1f} s)"}
    if rank == 0:
        print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
