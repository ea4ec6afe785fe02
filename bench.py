#!/usr/bin/env python3
"""Benchmark of the RefAdapt-DiT hot path on GB300: ms per denoising step.

One step = Algorithm 1 over every block of the workload's block stack: target
Q change, gate, reference-cache materialisation and joint attention with the
reference mass (all through the C ABI). Default workload: the video shape
(40 blocks, H=24, d=128, text 512 + 16,380 reference + 16,380 target tokens,
4 denoising steps, per-head target-to-reference logit bias), the largest
configuration; synthetic seeded bf16 inputs pre-generated in HBM for every
step of the trajectory (each block's inputs, 613 MB, exceed L2).

Timed steps cycle through the trajectory (step 0 is a full refresh), so
--steps 4 times every step of the video trajectory once. The same steps are
also timed with an always-refresh gate (delta_max = 1) for the speedup, and
with every launch on one stream in Algorithm 1's block order (the schedule a
model whose block b query depends on block b - 1 allows).

Prints one JSON line (rank 0). Its "workloads" object carries the image-edit
(60 blocks, 256 + 2x4096 + 4096 tokens, 8 steps) and heavy-reference (60
blocks, 256 + 4x4096 + 4096 tokens, 8 steps) workloads timed the same way in
the same run; its "dit_stack" object times the same algorithm over a stack of
random-weight DiT blocks around the attention on the image-edit row partition
(QKV, output projection, MLP, LayerNorms; --dit prints that measurement as its
own line with the CPU oracle beside it; --no-dit skips it). --impl reference
times the CPU oracle instead (a bounded sample per step, extrapolated).
"""
import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

WORKLOAD_NAMES = {
    "c1": "single joint-attention block: B=1, H=8, d=64, text 32 + ref 256 + tgt 256, 4 steps",
    "c2": "multi-reference image edit: 60 blocks, H=24, d=128, text 256 + ref 2x4096 + tgt 4096, 8 steps",
    "c3": "video: 40 blocks, H=24, d=128, text 512 + ref 16380 + tgt 16380, 4 steps, ref bias U(-3,0)",
    "c4": "heavy reference: 60 blocks, H=24, d=128, text 256 + ref 4x4096 + tgt 4096, 8 steps",
}
ROLES = ("text", "ref", "tgt")


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=8)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default="c3", choices=sorted(WORKLOAD_NAMES))
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-refresh-baseline", action="store_true")
    ap.add_argument("--no-graph", action="store_true")
    ap.add_argument("--no-serial", action="store_true",
                    help="skip the one-stream (no overlap) timing of the same steps")
    ap.add_argument("--no-nested", action="store_true",
                    help="skip the image-edit and heavy-reference workloads the video run nests in its line")
    ap.add_argument("--cpu-budget-s", type=float, default=12.0)
    ap.add_argument("--sweep", action="store_true",
                    help="time the sweep workload grid (tokens x reference fraction x reuse fraction); "
                         "one JSON line per point")
    ap.add_argument("--ablation", action="store_true",
                    help="time the controller-cue variants (product, change, exposure, anchor x exposure, "
                         "fixed interval 3) on the workload; one JSON line per variant")
    ap.add_argument("--diagnostics", action="store_true",
                    help="also time the trajectory with the staleness diagnostics on (every 8th target row)")
    ap.add_argument("--dit", action="store_true",
                    help="time the DiT-block stack (QKV / output projection / MLP GEMMs, LayerNorms and the "
                         "attention hot path) under Algorithm 1 on the workload's row partition; one JSON line")
    ap.add_argument("--no-dit", action="store_true",
                    help="skip the DiT-block stack summary that the default run adds to its line")
    ap.add_argument("--blocks", type=int, default=0,
                    help="run only the first N blocks of the stack (small profiling cases)")
    ap.add_argument("--separate-cache-update", action="store_true",
                    help="refresh each materialising block's cache slot with its own refadapt_ref_cache_update "
                         "launch before the attention instead of inside it")
    ap.add_argument("--trace", default=None,
                    help="write the main trajectory's observation record (per step and block: modes, gbar, the "
                         "exposure the gate read, a_b) as JSON lines to this file, after the timed region")
    ap.add_argument("--nvtx", action="store_true",
                    help="NVTX ranges around every block's decision and attention (for timeline profilers)")
    ap.add_argument("--out", default=None, help="also write the JSON line to this file")
    args = ap.parse_args()
    EXEC_OPTS["fused_cache"] = not args.separate_cache_update
    EXEC_OPTS["nvtx"] = bool(args.nvtx)
    return args


# Executor options every timed schedule shares (set from the command line).
EXEC_OPTS = {"fused_cache": True, "nvtx": False}


def launches_per_block(t):
    """Kernels one block of step t launches: the gate (t = 0) or the Q change
    with the gate in the same launch (t >= 1; the Q change's cluster path,
    which every workload here takes), the attention, and the cache update
    unless it is fused into the attention."""
    return 2 + (0 if EXEC_OPTS["fused_cache"] else 1)


# ----------------------------------------------------------------------------- helpers
def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16": float(p["bf16_tflops"]),
                "bf16_sustained": float(p["bf16_tflops_sustained"]), "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16": 1900.0, "bf16_sustained": 1700.0, "source": "fallback"}


def source_hash(*rel):
    h = hashlib.sha256()
    for r in rel:
        with open(os.path.join(ROOT, r), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


ATTN_SOURCES = ("paper_2609_32415_gb300/csrc/joint_attn.cu", "paper_2609_32415_gb300/csrc/tc_ptx.cuh")


def recorded_traffic(config, modes=None):
    """DRAM bytes per attention launch from the committed ncu summary, or None
    when the kernel source changed since the counters were taken. A record with
    separate launch kinds is averaged over the timed launches' modes (`modes`:
    one list of per-sample modes per launch). Kinds: "materialise" (a sample in
    COMPUTE or FULL: all rows, and the kernel writes the cache slot),
    "refresh" (a BOUNDARY sample: all rows, no cache write) and "reuse"; a
    record without "materialise" counts every launch that runs reference rows
    as "refresh"."""
    path = os.path.join(ROOT, "profiles", "attn_traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
    except Exception:
        return None
    if rec.get("source_hash") != source_hash(*ATTN_SOURCES):
        return None
    r = rec.get("per_launch", {}).get(config)
    if r is None or "bytes" in r:
        return r
    if not modes or "refresh" not in r or "reuse" not in r:
        return None

    def kind(m):
        m = [int(x) for x in m]
        if "materialise" in r and any(x in (2, 3) for x in m):
            return "materialise"
        return "refresh" if any(x != 0 for x in m) else "reuse"

    kinds = [kind(m) for m in modes]
    mix = {k: kinds.count(k) for k in ("materialise", "refresh", "reuse") if k in r}
    out = {"bytes": int(round(sum(r[k]["bytes"] for k in kinds) / len(kinds))),
           "mix": {k + "_launches": v for k, v in mix.items()}, "capture": r.get("capture")}
    out.update({k: r[k] for k in mix})
    return out


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons during a region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index=0):
        self.proc = None
        self.file = None
        self.sel = []
        try:
            import torch
            uuid = str(torch.cuda.get_device_properties(device_index).uuid)
            self.sel = ["-i", uuid if uuid.startswith("GPU-") else "GPU-" + uuid]
        except Exception:
            self.sel = []

    def start(self):
        try:
            self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            cmd = ["nvidia-smi", "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
                   "-lms", "200"] + self.sel
            self.proc = subprocess.Popen(cmd, stdout=self.file, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.file.flush()
        self.file.seek(0)
        rows = [ln.strip().split(",") for ln in self.file.read().splitlines() if ln.strip()]
        os.unlink(self.file.name)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                smax.append(float(r[2]))
            except ValueError:
                continue
            for name, v in zip(names, r[5:9]):
                if v.strip().lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def reduce_max_ms(local_ms, device="cpu"):
    """Max over ranks of a per-rank timed region (the job's time), on whatever
    process group is initialised; the local value when running alone."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(local_ms)
    t = torch.tensor([float(local_ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_ms_per_step(max_total_ms, steps, world_size):
    """Whole-job ms per denoising step: every rank runs `steps` steps of its own
    trajectory (weak scaling), so the job completes steps x world_size steps in
    the slowest rank's time."""
    return max_total_ms / (steps * world_size)


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


# ----------------------------------------------------------------------------- work model
def step_rows(wl, modes_tb):
    """Executed query rows of one step, summed over blocks and samples, from
    the per-block modes [n_blocks][B] (App. A.4: reuse skips reference rows)."""
    rows = 0
    for b_modes in modes_tb:
        for m in b_modes:
            rows += (wl.n_text + wl.n_tgt) if int(m) == 0 else wl.N
    return rows


def attn_flops(wl, mode):
    nq = (wl.n_text + wl.n_tgt) if int(mode) == 0 else wl.N
    return 4 * wl.d * wl.H * nq * wl.N


def expected_schedule(wl):
    """Modes the workload's drift recipe is expected to produce (closed-form
    expectation of the score; used only by the CPU reference leg)."""
    from paper_2609_32415_gb300 import synth
    m_est = synth._uniform_mass(wl.n_ref, wl.n_text + wl.n_tgt, wl.bias)
    sched, a_full = [], 0
    for t in range(wl.n_steps):
        if t == 0:
            sched.append([3] * wl.n_blocks)
            continue
        if t - a_full >= wl.delta_max:
            a_full = t
            sched.append([3] * wl.n_blocks)
            continue
        row, crossed = [], False
        for b in range(wl.n_blocks):
            if crossed:
                row.append(2)
                continue
            if wl.forced_boundary >= 0:
                c = b >= wl.forced_boundary
            else:
                c = synth._expected_gbar(wl.tgt_drift[b], t, m_est) >= wl.theta
            row.append(1 if c else 0)
            crossed = c
        sched.append(row)
    return sched


# ----------------------------------------------------------------------------- our arm
def make_inputs(wl, device):
    from paper_2609_32415_gb300 import synth
    traj = synth.Trajectory(wl, device=device)
    inputs = []
    for t in range(wl.n_steps):
        row = []
        for b in range(wl.n_blocks):
            row.append(traj.get(t, b))
        inputs.append(row)
    traj.forget()
    return inputs


def union_length(intervals):
    """Total length of the union of [start, end] intervals (overlaps counted once)."""
    busy, cur_a, cur_b = 0.0, None, None
    for a, b in sorted(intervals):
        if cur_b is None or a > cur_b:
            if cur_b is not None:
                busy += cur_b - cur_a
            cur_a, cur_b = a, b
        else:
            cur_b = max(cur_b, b)
    if cur_b is not None:
        busy += cur_b - cur_a
    return busy


def time_trajectory(wl, inputs, warmup, steps, delta_max=None, attn_timing=False, clocks=None,
                    barrier=None, cue="product", theta=None, diagnostics=False, diag_row_stride=8, overlap=True,
                    trace_path=None):
    """Run warmup + timed steps (cycling the trajectory); returns timing dict.
    overlap=False keeps every launch of a step on one stream in Algorithm 1's
    block order (each block's Q change, gate, cache update, then attention):
    the schedule a model whose block b query comes from block b - 1 allows."""
    import torch
    from paper_2609_32415_gb300 import Executor, roles_from_joint
    dm = wl.delta_max if delta_max is None else delta_max
    th = wl.theta if theta is None else theta
    ex = Executor(wl.n_blocks, wl.B, wl.H, wl.d, wl.n_text, wl.n_ref, wl.n_tgt, th, dm, wl.eps,
                  mass_rows=wl.mass_rows, forced_boundary=wl.forced_boundary, bias=wl.bias,
                  log_steps=wl.n_steps, cue=cue, diagnostics=diagnostics, diag_row_stride=diag_row_stride,
                  overlap=overlap, **EXEC_OPTS)
    views = [[roles_from_joint(inputs[t][b], wl.offsets(), wl.n) for b in range(wl.n_blocks)]
             for t in range(wl.n_steps)]
    T = wl.n_steps
    for i in range(warmup):
        ex.step(i % T, views[i % T])
    torch.cuda.synchronize()
    ev = []
    if attn_timing:
        pool = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                for _ in range(steps * wl.n_blocks)]
        it = iter(pool)

        def hook(phase, t, b):
            if phase == "pre":
                pair = next(it)
                pair[0].record()
                ev.append((t, b, pair))
            else:
                ev[-1][2][1].record()
        ex.attn_hook = hook
    step_ev = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
    if barrier:
        barrier()
    torch.cuda.synchronize()
    if clocks:
        clocks.start()
    t0 = time.perf_counter()
    step_ev[0].record()
    launches = 0
    for k in range(steps):
        t = (warmup + k) % T
        ex.step(t, views[t])
        launches += wl.n_blocks * launches_per_block(t)
        step_ev[k + 1].record()
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    clk = clocks.stop() if clocks else None
    if barrier:
        barrier()
    ex.attn_hook = None
    ex.check()
    if trace_path:
        with open(trace_path, "w") as f:
            for rec in ex.trace(wl.n_steps):
                f.write(json.dumps(rec) + "\n")
    total_ms = step_ev[0].elapsed_time(step_ev[-1])
    per_step = [step_ev[k].elapsed_time(step_ev[k + 1]) for k in range(steps)]
    modes = ex.modes.cpu().numpy()
    res = {"total_ms": total_ms, "per_step_ms": per_step, "wall_s": wall, "modes": modes,
           "gbar": ex.gbar.cpu().numpy(), "launches": launches, "clocks": clk,
           "steps_t": [(warmup + k) % T for k in range(steps)]}
    if attn_timing:
        # Consecutive attentions may overlap (two streams): the attention time
        # is the union of the launches' [start, end] intervals, every event
        # read against the step's first event (the time at least one attention
        # kernel runs); the plain sum of launch durations is kept beside it.
        flops, ms_sum, iv = 0, 0.0, []
        for (t, b, (e0, e1)) in ev:
            ms_sum += e0.elapsed_time(e1)
            iv.append((step_ev[0].elapsed_time(e0), step_ev[0].elapsed_time(e1)))
            flops += sum(attn_flops(wl, m) for m in modes[t, b])
        res["attn_ms"] = union_length(iv)
        res["attn_ms_sum_of_launches"] = ms_sum
        res["attn_flops"] = flops
        res["attn_launches"] = len(ev)
        res["attn_launch_tb"] = [(t, b) for (t, b, _) in ev]
    del ex
    return res


def time_graphs(wl, inputs, warmup, steps):
    """The same trajectory with every denoising step captured once as a CUDA
    graph (one graph per trajectory step) and replayed."""
    import torch
    from paper_2609_32415_gb300 import Executor, roles_from_joint
    T = wl.n_steps
    ex = Executor(wl.n_blocks, wl.B, wl.H, wl.d, wl.n_text, wl.n_ref, wl.n_tgt, wl.theta, wl.delta_max, wl.eps,
                  mass_rows=wl.mass_rows, forced_boundary=wl.forced_boundary, bias=wl.bias, log_steps=T,
                  **EXEC_OPTS)
    views = [[roles_from_joint(inputs[t][b], wl.offsets(), wl.n) for b in range(wl.n_blocks)] for t in range(T)]
    for t in range(T):                            # eager pass: first-call set-up of every entry point
        ex.step(t, views[t])
    torch.cuda.synchronize()
    graphs = [ex.capture_step(t, views[t]) for t in range(T)]
    for i in range(warmup):
        graphs[i % T].replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for k in range(steps):
        graphs[(warmup + k) % T].replay()
    e1.record()
    torch.cuda.synchronize()
    ex.check()
    modes = ex.modes.cpu().numpy()
    del graphs, ex
    return {"ms_per_step": e0.elapsed_time(e1) / steps, "modes": modes}


def host_memory_share():
    """Bytes of host memory available to this rank: MemAvailable divided by the
    ranks on this node (LOCAL_WORLD_SIZE); None when it cannot be read."""
    try:
        with open("/proc/meminfo") as f:
            for ln in f:
                if ln.startswith("MemAvailable:"):
                    avail = int(ln.split()[1]) * 1024
                    break
            else:
                return None
    except OSError:
        return None
    return avail // max(1, int(os.environ.get("LOCAL_WORLD_SIZE", "1")))


class PinnedArena:
    """Page-locked host memory handed out from a few large blocks of torch's
    pinned allocator. That allocator rounds every request up to a power of
    two, so one 612 MB buffer per (step, block) would pin 1 GiB each (the
    video trajectory: 171 GB of the host's 199 GB); blocks of a power-of-two
    size are used whole and sub-allocated in order instead."""

    def __init__(self, total_bytes, largest_bytes, block_bytes=16 << 30):
        import torch
        self.torch = torch
        need = max(int(total_bytes), int(largest_bytes), 1)
        size = 1 << (need - 1).bit_length()
        self.block = min(size, max(block_bytes, 1 << (int(largest_bytes) - 1).bit_length()))
        self.blocks, self.used = [], self.block
        self.pinned = 0

    def take(self, numel, dtype):
        nbytes = (numel * self.torch.empty((), dtype=dtype).element_size() + 511) // 512 * 512
        if self.used + nbytes > self.block:
            self.blocks.append(self.torch.empty(self.block, dtype=self.torch.uint8, pin_memory=True))
            self.pinned += self.block
            self.used = 0
        out = self.blocks[-1][self.used:self.used + numel * self.torch.empty((), dtype=dtype).element_size()]
        self.used += nbytes
        return out.view(dtype)


def time_e2e(wl, inputs, warmup, steps, keep=None):
    """Same steps through the public API with host-resident inputs and results.

    Host side: one page-locked buffer per (step, block) with that block's
    inputs, written by the CPU (a staging copy from the device-generated
    trajectory, then a host memcpy), and one page-locked output buffer per
    block. Per step: the step's gates run first on every block's target Q
    (copied during the previous step, behind that block's data)
    (Executor.gate_block: a gate reads only that block's target queries, its
    previous-step mass partials and the controller state of the blocks before
    it); one device->host read of the step's modes (and gbar) follows; then,
    per block, the text Q/K/V and target K/V are copied, plus the reference
    Q/K/V only when a sample materialises (COMPUTE or FULL; a reusing or
    boundary block reads its reference Q/K/V from the cache), on a copy stream, triple-buffered and overlapped with
    the attentions (Executor.attend_block), up to two blocks ahead;
    consecutive attentions alternate between two high-priority streams; every
    executed row of the block's attention output (text and target rows, and
    reference rows where a sample is not REUSE) goes back to the host on a
    second copy stream as soon as the attention ends. A step ends when its
    last output is on the host.

    Two measurements over the same buffers: the first trajectory right after
    the host buffers were written (no untimed pass over them: what a caller's
    first trajectory sees, with the device's translations of freshly pinned
    host memory still cold), then, after `warmup` more steps, `steps` timed
    steps (steady state).

    With `keep` (a list) nothing is timed: one trajectory runs step by step
    through the same pipeline and `keep` receives, per step, the modes read
    by the host and a copy of every block's host outputs (for tests)."""
    import torch
    from paper_2609_32415_gb300 import Executor
    T, nb = wl.n_steps, wl.n_blocks
    off = wl.offsets()
    # Host layout per (t, b): [target Q | text Q, K, V, target K, V | reference Q, K, V]
    parts = {"tq": [(0, "tgt")], "base": [(0, "text"), (1, "text"), (2, "text"), (1, "tgt"), (2, "tgt")],
             "ref": [(0, "ref"), (1, "ref"), (2, "ref")]}
    shape = {r: (wl.B, wl.H, wl.n[r], wl.d) for r in ROLES}
    size = {k: sum(math.prod(shape[r]) for _, r in v) for k, v in parts.items()}
    per_block = size["tq"] + size["base"] + size["ref"]

    def views(flat, start, kind):
        out, o = {}, start
        for z, r in parts[kind]:
            out[(z, r)] = flat[o:o + math.prod(shape[r])].view(shape[r])
            o += math.prod(shape[r])
        return out

    o_base, o_ref = size["tq"], size["tq"] + size["base"]
    # Page-locked host trajectory (cudaHostAlloc through torch's pinned
    # allocator, sub-allocated from large blocks), written by the CPU: each
    # block's bytes go device -> a staging buffer, then a host memcpy into the
    # block's own buffer.
    out_elems = sum(math.prod(shape[r]) for r in ROLES)
    need = 2 * (T * nb * per_block + nb * out_elems)
    share = host_memory_share()
    if share is not None and need > 0.8 * share:
        raise RuntimeError("host memory: the e2e trajectory needs %.1f GB pinned per rank, %.1f GB available to this "
                           "rank" % (need / 1e9, share / 1e9))
    arena = PinnedArena(need, 2 * per_block)
    stage = torch.empty(per_block, dtype=torch.bfloat16, pin_memory=True)
    stage_v = {"tq": views(stage, 0, "tq"), "base": views(stage, o_base, "base"), "ref": views(stage, o_ref, "ref")}
    # Page-locked host outputs, one set per block (each step overwrites them).
    hout = [{r: arena.take(math.prod(shape[r]), torch.bfloat16).view(shape[r]) for r in ROLES} for _ in range(nb)]
    bufs, host = [], []
    for t in range(T):
        brow, hrow = [], []
        for b in range(nb):
            X = inputs[t][b]
            for kind in stage_v:
                for (z, r), h in stage_v[kind].items():
                    h.copy_(X[z, :, :, off[r]:off[r] + wl.n[r], :])
            buf = arena.take(per_block, torch.bfloat16)
            buf.copy_(stage)
            brow.append(buf)
            hrow.append({k: buf[o:o + size[k]] for k, o in (("tq", 0), ("base", o_base), ("ref", o_ref))})
        bufs.append(brow)
        host.append(hrow)
    del stage, stage_v
    torch.cuda.synchronize()
    dev = torch.device("cuda")
    # Device staging: each block's target Q for the current and the previous
    # step (read as q_{t-1}), NSLOT slots for the rest of a block and NOUT
    # output slots.
    tq = [[torch.empty(size["tq"], dtype=torch.bfloat16, device=dev) for _ in range(nb)] for _ in range(2)]
    NSLOT = 3  # the copy stream may run two blocks ahead of the attentions
    slots = [torch.empty(size["base"] + size["ref"], dtype=torch.bfloat16, device=dev) for _ in range(NSLOT)]
    slot_v = [{**views(x, 0, "base"), **views(x, size["base"], "ref")} for x in slots]
    NOUT = 3
    osl = [{r: torch.empty(shape[r], dtype=torch.bfloat16, device=dev) for r in ROLES} for _ in range(NOUT)]
    ex = Executor(nb, wl.B, wl.H, wl.d, wl.n_text, wl.n_ref, wl.n_tgt, wl.theta, wl.delta_max, wl.eps,
                  mass_rows=wl.mass_rows, forced_boundary=wl.forced_boundary, bias=wl.bias, log_steps=T,
                  **EXEC_OPTS)
    comp = torch.cuda.current_stream()
    copy = torch.cuda.Stream()
    back = torch.cuda.Stream()  # device -> host results
    # consecutive blocks' attentions on two high-priority streams (as in
    # Executor.step): block b + 1 may start in block b's last wave
    lo_pri, hi_pri = torch.cuda.Stream.priority_range()
    attn_streams = [torch.cuda.Stream(priority=hi_pri) for _ in range(2)]
    gates_done = torch.cuda.Event()
    attn_join = [torch.cuda.Event() for _ in range(2)]
    back_join = torch.cuda.Event()
    slot_free = [torch.cuda.Event() for _ in range(NSLOT)]
    out_free = [torch.cuda.Event() for _ in range(NOUT)]
    tq_free = [torch.cuda.Event() for _ in range(2)]
    for e in slot_free + out_free + tq_free:
        e.record(comp)
    modes_host = torch.empty((nb, wl.B), dtype=torch.int32, pin_memory=True)
    gbar_host = torch.empty((nb, wl.B), dtype=torch.float32, pin_memory=True)
    decided = torch.cuda.Event()
    h2d, d2h = [0], [0]
    PREFETCH = NSLOT  # blocks whose text and target K/V are copied before the step's modes are read

    def copy_base(t, b, s):
        copy.wait_event(slot_free[s])
        with torch.cuda.stream(copy):
            slots[s][:size["base"]].copy_(host[t][b]["base"], non_blocking=True)
        h2d[0] += size["base"] * 2

    tq_ready = [None, None]  # copy-stream event after a step parity's target queries (None: not copied yet)

    def copy_tq(t_dst, p, b_range):
        with torch.cuda.stream(copy):
            for b in b_range:
                tq[p][b].copy_(host[t_dst][b]["tq"], non_blocking=True)
            e = torch.cuda.Event()
            e.record(copy)
        h2d[0] += size["tq"] * 2 * len(b_range)
        return e

    def one_step(t, counter, t_next):
        li = t % ex.log_steps
        p = counter[1] % 2  # alternates per call (the step index may wrap)
        counter[1] += 1
        if tq_ready[p] is None:  # first step: nothing was prefetched
            copy.wait_event(tq_free[p])
            tq_ready[p] = copy_tq(t, p, range(nb))
        comp.wait_event(tq_ready[p])
        tq_ready[p] = None
        for b in range(nb):
            ex.gate_block(t, b, tq[p][b].view(shape["tgt"]), log_index=li)
        tq_free[1 - p].record(comp)  # the gates of this step have read the previous step's queries
        modes_host.copy_(ex.modes[li], non_blocking=True)
        gbar_host.copy_(ex.gbar[li], non_blocking=True)
        d2h[0] += modes_host.numel() * 4 + gbar_host.numel() * 4
        decided.record(comp)
        first = counter[0]
        for b in range(min(PREFETCH, nb)):
            copy_base(t, b, (first + b) % NSLOT)
        gates_done.record(comp)
        for st in attn_streams:
            st.wait_event(gates_done)
        decided.synchronize()
        # reference rows are read only by materialising samples (COMPUTE,
        # FULL); they run (and come back) for every sample that is not REUSE
        ref_in = [bool(((modes_host[b] == 2) | (modes_host[b] == 3)).any()) for b in range(nb)]
        ref_out = [bool((modes_host[b] != 0).any()) for b in range(nb)]
        copy.wait_event(tq_free[1 - p])  # the next step's queries go where the previous step's were
        for b in range(nb):
            s = counter[0] % NSLOT
            o = counter[0] % NOUT
            counter[0] += 1
            if b >= PREFETCH:
                copy_base(t, b, s)
            with torch.cuda.stream(copy):
                if ref_in[b]:
                    slots[s][size["base"]:].copy_(host[t][b]["ref"], non_blocking=True)
                    h2d[0] += size["ref"] * 2
                ready = torch.cuda.Event()
                ready.record(copy)
            tq_ready[1 - p] = copy_tq(t_next, 1 - p, [b])  # the next step's target Q of this block, behind its data
            st = attn_streams[b % 2]
            st.wait_event(ready)
            st.wait_event(out_free[o])
            sv = slot_v[s]
            x = {"text": (sv[(0, "text")], sv[(1, "text")], sv[(2, "text")]),
                 "ref": (sv[(0, "ref")], sv[(1, "ref")], sv[(2, "ref")]),
                 "tgt": (tq[p][b].view(shape["tgt"]), sv[(1, "tgt")], sv[(2, "tgt")])}
            with torch.cuda.stream(st):
                ex.attend_block(t, b, x, osl[o], log_index=li)
                slot_free[s].record(st)
                done = torch.cuda.Event()
                done.record(st)
            back.wait_event(done)
            with torch.cuda.stream(back):
                for r in (("text", "ref", "tgt") if ref_out[b] else ("text", "tgt")):
                    hout[b][r].copy_(osl[o][r], non_blocking=True)
                    d2h[0] += osl[o][r].numel() * 2
                out_free[o].record(back)
        for st, j in zip(attn_streams, attn_join):  # the next step's gates read this step's mass partials
            j.record(st)
            comp.wait_event(j)
        back_join.record(back)  # the step ends when its last result is on the host
        comp.wait_event(back_join)

    counter = [0, 0]  # blocks, steps
    seq = [i % T for i in range(T + warmup + steps + 1)]

    def timed(k0, k):
        h2d[0] = d2h[0] = 0
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(k + 1)]
        ev[0].record()
        for i in range(k):
            one_step(seq[k0 + i], counter, seq[k0 + i + 1])
            ev[i + 1].record()
        torch.cuda.synchronize()
        return (ev[0].elapsed_time(ev[-1]) / k, [round(ev[i].elapsed_time(ev[i + 1]), 3) for i in range(k)],
                int(h2d[0] // k), int(d2h[0] // k))

    torch.cuda.synchronize()
    if keep is not None:
        for i in range(T):
            one_step(seq[i], counter, seq[i + 1])
            torch.cuda.synchronize()
            keep.append({"t": seq[i], "modes": modes_host.clone(),
                         "out": [{r: hout[b][r].clone() for r in ROLES} for b in range(nb)]})
        ex.check()
        del host, slots, slot_v, osl, tq, ex, bufs, hout, arena
        return keep
    first_ms, first_steps, first_h2d, first_d2h = timed(0, T)
    for i in range(warmup):
        one_step(seq[T + i], counter, seq[T + i + 1])
    torch.cuda.synchronize()
    ms, per_step, h2d_b, d2h_b = timed(T + warmup, steps)
    ex.check()
    pinned_gb = arena.pinned / 1e9
    del host, slots, slot_v, osl, tq, ex, bufs, hout, arena
    pipeline = ("per step: the step's gates first (every block's target Q copied during the previous step), one "
                "read of the modes, then per block text Q/K/V + target K/V and reference Q/K/V only where a "
                "sample materialises (COMPUTE or FULL), plus the next step's target Q; every executed output row "
                "(text and target, reference where a sample is not REUSE) back to the host behind each attention; bytes are the "
                "mean over the timed steps")
    return {"value": ms, "unit": "ms/step", "per_step_ms": per_step, "h2d_bytes_per_step": h2d_b,
            "d2h_bytes_per_step": d2h_b,
            "host_buffers": "pinned (cudaHostAlloc, %.1f GB in 16 GiB blocks), one buffer per (step, block) and "
                            "one output set per block, written by the CPU; timed after the first trajectory over "
                            "them and %d warm-up steps" % (pinned_gb, warmup),
            "pipeline": pipeline,
            "first_use": {"value": first_ms, "unit": "ms/step", "per_step_ms": first_steps,
                          "h2d_bytes_per_step": first_h2d, "d2h_bytes_per_step": first_d2h,
                          "steps": T,
                          "host_buffers": "the same buffers, timed from their first use: no untimed pass over "
                                          "them, no pinned range set aside"}}


def _q_delta_launch_ms(pairs, B, H, eps, reps, gate_mpl=0):
    """Average duration of one refadapt_q_delta launch over `reps` launches
    rotating over `pairs` (current, previous), queued behind a GPU-side sleep
    so they run back to back; the best of three runs. gate_mpl > 0 times
    refadapt_q_delta_gate instead (the gate of block 0, step 1, on mass
    partials of that length), the call the executor makes."""
    import torch
    from paper_2609_32415_gb300 import api
    ws = api.q_delta_workspace(B, H)
    out = torch.empty((B, H), dtype=torch.float32, device="cuda")
    if gate_mpl > 0:
        state = api.new_state(B, "cuda")
        mode = torch.zeros(B, dtype=torch.int32, device="cuda")
        mass = torch.full((B, H, gate_mpl), 0.01, dtype=torch.float32, device="cuda")

        def call(a, b):
            api.refadapt_q_delta_gate(a, b, out, ws, 1, 0, state, mode, 0.1, 1000, mass, 128 * gate_mpl, eps)
    else:
        def call(a, b):
            api.refadapt_q_delta(a, b, out, ws, eps)
    for a, b in pairs:                           # warm-up
        call(a, b)
    runs = []
    for _ in range(3):
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda._sleep(20_000_000)            # ~10 ms: the host queues every launch meanwhile
        e0.record()
        for i in range(reps):
            a, b = pairs[i % len(pairs)]
            call(a, b)
        e1.record()
        torch.cuda.synchronize()
        runs.append(e0.elapsed_time(e1) / reps)
    return min(runs)


def time_q_delta_long(n_tgt=16380, H=24, d=128, eps=1e-6, reps=64):
    """The same kernel on a longer read: the video workload's target-query
    shape (16,380 rows; 2 x 100.6 MB per launch), four rotating seeded pairs
    (805 MB > L2)."""
    import torch
    g = torch.Generator(device="cuda")
    g.manual_seed(0x5EED)
    pairs = []
    for _ in range(4):
        prev = (torch.randn((1, H, n_tgt, d), generator=g, device="cuda") / d ** 0.5).to(torch.bfloat16)
        cur = (prev.float() + 0.4 * torch.randn((1, H, n_tgt, d), generator=g, device="cuda") / d ** 0.5
               ).to(torch.bfloat16)
        pairs.append((cur, prev))
    ms = _q_delta_launch_ms(pairs, 1, H, eps, reps)
    byts = 4 * n_tgt * H * d
    del pairs
    return {"bytes": byts, "ms": ms, "gbs": byts / ms / 1e6}


def time_q_delta(wl, inputs, reps=64):
    """HBM roofline of the Q-change reduction alone: target Q of step 1 vs step
    0, rotating over 8 blocks (8 x 50 MB > L2, so every launch reads HBM; a
    stack cut to fewer blocks is padded with seeded pairs of the same shape).
    The launches are queued behind a GPU-side sleep so they run back to back;
    the average launch duration is the events' span divided by the launches."""
    import torch
    from paper_2609_32415_gb300 import roles_from_joint
    nb = min(8, wl.n_blocks)
    pairs = [(roles_from_joint(inputs[1][b], wl.offsets(), wl.n)["tgt"][0],
              roles_from_joint(inputs[0][b], wl.offsets(), wl.n)["tgt"][0]) for b in range(nb)]
    g = torch.Generator(device="cuda")
    g.manual_seed(0x0DE17A)
    shape = (wl.B, wl.H, wl.n_tgt, wl.d)
    while len(pairs) < 8:
        prev = (torch.randn(shape, generator=g, device="cuda") / wl.d ** 0.5).to(torch.bfloat16)
        cur = (prev.float() + 0.3 * torch.randn(shape, generator=g, device="cuda") / wl.d ** 0.5).to(torch.bfloat16)
        pairs.append((cur, prev))
    ms = _q_delta_launch_ms(pairs, wl.B, wl.H, wl.eps, reps)
    from paper_2609_32415_gb300 import api
    ms_gate = _q_delta_launch_ms(pairs, wl.B, wl.H, wl.eps, reps,
                                 gate_mpl=api.refadapt_mass_partial_len(wl.n_text, wl.n_tgt))
    byts = 4 * wl.n_tgt * wl.H * wl.d * wl.B
    # Context: a library streaming read of the same number of bytes (torch's
    # sum over one contiguous buffer), timed the same way.
    bufs = [torch.ones(byts // 2, dtype=torch.bfloat16, device="cuda") for _ in range(8)]
    lib_runs = []
    for _ in range(3):
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda._sleep(20_000_000)
        e0.record()
        for i in range(reps):
            bufs[i % 8].sum(dtype=torch.float32)
        e1.record()
        torch.cuda.synchronize()
        lib_runs.append(e0.elapsed_time(e1) / reps)
    del bufs
    return {"bytes": byts, "ms": ms, "gbs": byts / ms / 1e6, "lib_read_gbs": byts / min(lib_runs) / 1e6,
            "ms_with_gate": ms_gate}


def cpu_oracle_sample(wl, X, budget_s):
    """Time the CPU oracle on a bounded sample of one block: target query rows
    of every head against all keys, plus Eq. 1 over the block's target Q.
    Returns seconds per query row (one head) and seconds per block of Eq. 1."""
    import numpy as np
    import torch
    import oracle

    def widen(t):
        return oracle.bf16_to_f64(t.contiguous().cpu().view(torch.int16).numpy().view(np.uint16))

    off = wl.offsets()
    q = widen(X[0, 0, :, off["tgt"]:off["tgt"] + wl.n_tgt, :])
    k = widen(X[1, 0])
    v = widen(X[2, 0])
    nth = oracle.default_threads()
    r0, r1 = wl.n_text, wl.n_text + wl.n_ref
    rows = 8
    elapsed = 0.0
    used = 0
    while True:
        t0 = time.perf_counter()
        oracle.joint_attention(q[:, :rows], k, v, 1.0 / math.sqrt(wl.d), ref_range=(r0, r1), nthreads=nth)
        dt = time.perf_counter() - t0
        elapsed, used = dt, rows
        if dt > budget_s / 4 or rows >= wl.n_tgt:
            break
        rows = min(wl.n_tgt, max(rows * 2, int(rows * (budget_s / 3) / max(dt, 1e-3))))
    per_row = elapsed / (used * wl.H)
    qp = q[:, :min(wl.n_tgt, 4096)]
    t0 = time.perf_counter()
    oracle.q_change(qp, qp * 1.01, wl.eps)
    qd_s = (time.perf_counter() - t0) * (wl.n_tgt / qp.shape[1]) * wl.B
    return {"per_row_s": per_row, "q_change_block_s": qd_s, "rows": used, "heads": wl.H,
            "threads": nth, "sample_s": elapsed}


def make_wl(name, rank=0, blocks=0):
    """The named workload with this rank's seed (replicas draw their own
    trajectories), optionally cut to its first `blocks` blocks."""
    from paper_2609_32415_gb300 import synth
    wl = synth.make_workload(name, seed=rank) if name in ("c3", "c4") else synth.make_workload(name)
    if name not in ("c3", "c4"):
        wl.seed = rank
    if blocks > 0:
        wl.n_blocks = min(wl.n_blocks, blocks)
        wl.ref_drift = wl.ref_drift[:wl.n_blocks]
        wl.tgt_drift = wl.tgt_drift[:wl.n_blocks]
    return wl


def config_dict(wl, args, ws):
    """The line's `config` (both arms print the same one)."""
    return {"workload": WORKLOAD_NAMES[wl.name] + (" (first %d blocks)" % wl.n_blocks if args.blocks > 0 else ""),
            "name": wl.name, "B": wl.B, "H": wl.H, "d": wl.d,
            "tokens": {"text": wl.n_text, "ref": wl.n_ref, "tgt": wl.n_tgt},
            "blocks": wl.n_blocks, "trajectory_steps": wl.n_steps, "theta": round(wl.theta, 6),
            "delta_max": wl.delta_max,
            "l2": "inputs larger than L2 (%.0f MB per block)" % (3 * wl.B * wl.H * wl.N * wl.d * 2 / 1e6),
            "resident_steps": wl.n_steps,
            "parallelism": "replicas" if ws > 1 else "single GPU"}


def q_delta_summary(qd, peaks):
    return {"bound": "hbm", "kernel": "q_delta_cluster_kernel", "achieved": round(qd["gbs"], 1),
            "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": round(qd["gbs"] / peaks["hbm_gbs"], 4),
            "bytes_per_launch": qd["bytes"], "launch_ms": round(qd["ms"], 5),
            "same_bytes_torch_sum_gbs": round(qd["lib_read_gbs"], 1),
            "with_gate_launch_ms": round(qd["ms_with_gate"], 5),
            "peak_kind": "%s HBM copy" % peaks["source"]}


def run_nested(name, args, peaks):
    """Another workload timed the same way inside the same run (attention-only
    steps, gated and always-refresh, and the Q change): one object of the
    line."""
    import torch
    wl = make_wl(name)
    inputs = make_inputs(wl, "cuda")
    torch.cuda.synchronize()
    clocks = Clocks(0)
    main = time_trajectory(wl, inputs, args.warmup, args.steps, attn_timing=True, clocks=clocks)
    refresh = time_trajectory(wl, inputs, args.warmup, args.steps, delta_max=1)
    qd = time_q_delta(wl, inputs)
    del inputs
    torch.cuda.empty_cache()
    ms = main["total_ms"] / args.steps
    tf = main["attn_flops"] / (main["attn_ms"] * 1e-3) / 1e12
    sched = expected_schedule(wl)
    return {"workload": WORKLOAD_NAMES[name], "name": name, "blocks": wl.n_blocks,
            "trajectory_steps": wl.n_steps, "theta": round(wl.theta, 6), "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(ms, 3),
            "per_step_ms": [round(x, 3) for x in main["per_step_ms"]],
            "modes_per_step": {str(t): [int(x) for x in main["modes"][t, :, 0]] for t in sorted(set(main["steps_t"]))},
            "schedule_matches_expected": all([int(x) for x in main["modes"][t, :, 0]] == sched[t]
                                             for t in set(main["steps_t"])),
            "attn_tflops": round(tf, 1), "attn_frac_of_bf16_peak": round(tf / peaks["bf16_sustained"], 4),
            "attn_launch_ms": round(main["attn_ms"] / main["attn_launches"], 4),
            "always_refresh_ms_per_step": round(refresh["total_ms"] / args.steps, 3),
            "speedup_vs_always_refresh": round(refresh["total_ms"] / main["total_ms"], 3),
            "q_delta_roofline": q_delta_summary(qd, peaks),
            "clocks": main["clocks"]}


def main_ours(args):
    import torch
    import torch.distributed as dist
    import __graft_entry__ as ge
    from paper_2609_32415_gb300 import synth
    ws, rank, local = dist_env()
    if ws > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", init_method="env://")
        barrier = dist.barrier
    else:
        barrier = None
    ge.build()
    wl = make_wl(args.config, rank, args.blocks)
    peaks = load_peaks()
    inputs = make_inputs(wl, "cuda")
    torch.cuda.synchronize()
    clocks = Clocks(local)
    main = time_trajectory(wl, inputs, args.warmup, args.steps, attn_timing=True, clocks=clocks,
                           barrier=barrier, trace_path=args.trace if rank == 0 else None)
    total_ms = reduce_max_ms(main["total_ms"], device="cuda")
    ms_per_step = job_ms_per_step(total_ms, args.steps, ws)
    refresh = None
    if not args.no_refresh_baseline:
        refresh = time_trajectory(wl, inputs, args.warmup, args.steps, delta_max=1, barrier=barrier)
    serial = None
    if not args.no_serial:
        serial = time_trajectory(wl, inputs, args.warmup, args.steps, overlap=False, barrier=barrier)
    qd = time_q_delta(wl, inputs)
    qd_long = time_q_delta_long(H=wl.H, d=wl.d, eps=wl.eps) if (wl.d == 128 and wl.n_tgt < 16380) else None
    diag = None
    if args.diagnostics:
        diag = time_trajectory(wl, inputs, args.warmup, args.steps, diagnostics=True, diag_row_stride=8)
    graph = None
    if not args.no_graph:
        try:
            graph = time_graphs(wl, inputs, args.warmup, args.steps)
        except Exception as exc:
            graph = {"ms_per_step": None, "error": str(exc)[:200]}
    e2e = None
    if not args.no_e2e:
        try:
            e2e = time_e2e(wl, inputs, args.warmup, args.steps)
        except Exception as exc:  # host memory or pinning limits: report, do not guess
            e2e = {"value": None, "unit": "ms/step", "error": str(exc)[:200],
                   "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        s = cpu_oracle_sample(wl, inputs[1][0], args.cpu_budget_s)
        rows_step = [step_rows(wl, main["modes"][t]) for t in main["steps_t"]]
        per_step_s = [r * wl.H * s["per_row_s"] + wl.n_blocks * s["q_change_block_s"] for r in rows_step]
        cpu = {"value": round(1000.0 * statistics.mean(per_step_s), 1), "unit": "ms/step", "cores": s["threads"],
               "kind": "oracle",
               "sample": "fp64 C oracle, %d target query rows x %d heads of block 0 (step 1) against all %d keys "
                         "(%.1f s) plus Eq. 1 over the block's target Q; extrapolated per query row to the "
                         "executed rows of the timed steps" % (s["rows"], s["heads"], wl.N, s["sample_s"])}
    del inputs
    torch.cuda.empty_cache()
    nested = {}
    if rank == 0 and ws == 1 and not args.no_nested and args.config == "c3" and args.blocks == 0:
        for name in ("c2", "c4"):
            try:
                nested[name] = run_nested(name, args, peaks)
            except Exception as exc:  # report, do not guess
                nested[name] = {"error": str(exc)[:200]}
            torch.cuda.empty_cache()
    dit = None
    if rank == 0 and ws == 1 and not args.no_dit:
        # The DiT-block stack around the same attention on the image-edit row
        # partition (one line of its own with --dit); its inputs and weights
        # replace the attention trajectory in HBM.
        try:
            dit_wl = synth.make_workload("c2")
            if args.blocks > 0:
                dit_wl.n_blocks = min(dit_wl.n_blocks, args.blocks)
            d = run_dit(args, dit_wl, with_cpu=False, with_context=False)
            dit = {k: d[k] for k in ("workload", "value", "unit", "block", "theta", "per_step_ms", "gemm_tflops",
                                     "gemm_frac_of_bf16_peak", "gemm_share_of_step", "attn_tflops",
                                     "always_refresh_ms_per_step", "speedup_vs_always_refresh", "clocks")
                   if k in d}
        except Exception as exc:  # report, do not guess
            dit = {"error": str(exc)[:200]}
    if rank != 0:
        if ws > 1:
            dist.barrier()
            dist.destroy_process_group()
        return
    attn_tflops = main["attn_flops"] / (main["attn_ms"] * 1e-3) / 1e12
    traffic = recorded_traffic(args.config, [list(main["modes"][t, b]) for t, b in main["attn_launch_tb"]])
    per_launch_flops = main["attn_flops"] / main["attn_launches"]
    qsum = q_delta_summary(qd, peaks)
    if qd_long is not None:
        qsum["longer_read"] = {"shape": "video target query, 16,380 rows x %d heads x d %d" % (wl.H, wl.d),
                               "bytes_per_launch": qd_long["bytes"], "launch_ms": round(qd_long["ms"], 5),
                               "achieved": round(qd_long["gbs"], 1),
                               "frac": round(qd_long["gbs"] / peaks["hbm_gbs"], 4)}
    line = {
        "metric": "ms per denoising step (attention TFLOP/s and %% of bf16 peak, vs always-refresh)",
        "value": round(ms_per_step, 3),
        "unit": "ms/step",
        "n_gpus": ws,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_per_step, 3),
        "higher_is_better": False,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded bf16 Q/K/V with the workload's drift recipe; no datasets or weights)",
        "config": config_dict(wl, args, ws),
        "per_step_ms": [round(x, 3) for x in main["per_step_ms"]],
        "timed_trajectory_steps": main["steps_t"],
        "modes_per_step": {str(t): [int(x) for x in main["modes"][t, :, 0]] for t in sorted(set(main["steps_t"]))},
        "attn_tflops": round(attn_tflops, 1),
        "attn_frac_of_bf16_peak": round(attn_tflops / peaks["bf16_sustained"], 4),
        "roofline": {"bound": "tensor", "kernel": "joint_attn_kernel<128>",
                     "achieved": round(attn_tflops, 1), "peak": peaks["bf16_sustained"],
                     "unit": "TFLOP/s", "frac": round(attn_tflops / peaks["bf16_sustained"], 4),
                     "traffic": None if traffic is None else traffic["bytes"],
                     "traffic_capture": traffic,
                     "flops_per_launch": int(per_launch_flops),
                     "launch_ms": round(main["attn_ms"] / main["attn_launches"], 4),
                     "peak_kind": "%s, sustained bf16 (kernel timed inside a long step)" % peaks["source"]},
        "q_delta_roofline": qsum,
        "gpu_launches": main["launches"],
        "clocks": main["clocks"],
        "e2e": None if e2e is None else {k: v for k, v in e2e.items() if k != "first_use"},
        "cpu_baseline": cpu,
    }
    if e2e is not None and e2e.get("first_use") is not None:
        line["e2e_unpadded"] = e2e["first_use"]
    if serial is not None:
        line["ms_per_step_serial"] = round(serial["total_ms"] / args.steps, 3)
        line["serial_schedule"] = ("one stream, Algorithm 1's block order: each block's Q change, gate, cache "
                                   "update, then its attention (no work of block b under block b - 1's attention)")
    if diag is not None:
        dms = diag["total_ms"] / args.steps
        line["diagnostics_ms_per_step"] = round(dms, 3)
        line["diagnostics_overhead"] = round(dms / (main["total_ms"] / args.steps) - 1.0, 4)
    if graph is not None:
        line["cuda_graph_ms_per_step"] = None if graph.get("ms_per_step") is None else round(graph["ms_per_step"], 3)
        if graph.get("error"):
            line["cuda_graph_error"] = graph["error"]
        elif "modes" in graph:
            timed = sorted(set(main["steps_t"]))   # steps both runs executed
            line["cuda_graph_modes_match"] = bool((graph["modes"][timed] == main["modes"][timed]).all())
    if refresh is not None:
        rms = refresh["total_ms"] / args.steps
        line["always_refresh_ms_per_step"] = round(rms, 3)
        line["speedup_vs_always_refresh"] = round(rms / (main["total_ms"] / args.steps), 3)
    sched = expected_schedule(wl)
    line["schedule_matches_expected"] = all(
        [int(x) for x in main["modes"][t, :, 0]] == sched[t] for t in set(main["steps_t"]))
    if nested:
        line["workloads"] = nested
    if dit is not None:
        line["dit_stack"] = dit
    emit(line, args)
    if ws > 1:
        dist.barrier()
        dist.destroy_process_group()


def emit(line, args):
    s = json.dumps(line)
    print(s, flush=True)
    if args.out:
        with open(args.out, "w") as f:
            f.write(s + "\n")


# ----------------------------------------------------------------------------- reference arm
def main_reference(args):
    """The CPU oracle as it stands, on the host cores: each step a bounded sample
    of the workload, extrapolated to one denoising step over the schedule the
    workload's recipe gives (the GPU arm reports whether its executed schedule
    is that one: schedule_matches_expected)."""
    ws, rank, _ = dist_env()
    if rank != 0:
        return
    from oracle import build as oracle_build
    from paper_2609_32415_gb300 import synth
    oracle_build.build()
    wl = make_wl(args.config, 0, args.blocks)
    sched = expected_schedule(wl)
    traj = synth.Trajectory(wl, device="cpu")
    X = traj.get(1, 0)
    per_step_budget = max(1.0, min(args.cpu_budget_s, 150.0 / max(1, args.steps + args.warmup)))
    vals = []
    last = None
    for i in range(args.warmup + args.steps):
        t = i % wl.n_steps
        s = cpu_oracle_sample(wl, X, per_step_budget)
        ms = 1000.0 * (step_rows(wl, [[m] for m in sched[t]]) * wl.H * s["per_row_s"]
                       + wl.n_blocks * s["q_change_block_s"])
        if i >= args.warmup:
            vals.append(ms)
        last = s
    value = round(statistics.mean(vals), 1)
    line = {
        "impl": "reference",
        "metric": "ms per denoising step (attention TFLOP/s and %% of bf16 peak, vs always-refresh)",
        "value": value, "unit": "ms/step", "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": value, "higher_is_better": False, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64", "data": "synthetic (seeded bf16 inputs widened to fp64)",
        "config": config_dict(wl, args, ws),
        "schedule": {str(t): sched[t] for t in range(wl.n_steps)},
        "cpu_baseline": {"value": value, "unit": "ms/step", "cores": last["threads"], "kind": "oracle",
                         "sample": "per step: %d target query rows x %d heads of one block against all %d keys "
                                   "plus Eq. 1 over the block's target Q, extrapolated to the executed rows of "
                                   "the workload's schedule" % (last["rows"], last["heads"], wl.N)},
        "e2e": {"value": value, "unit": "ms/step", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    emit(line, args)


def main_sweep(args):
    """Sweep workload: 8 blocks, 8 steps per point; ms per step, attention
    roofline fraction and speedup over always-refresh for every grid point."""
    import torch
    import __graft_entry__ as ge
    from paper_2609_32415_gb300 import synth
    ge.build()
    peaks = load_peaks()
    lines = []
    for total, frac, reuse in synth.sweep_points():
        wl = synth.make_workload("c5", total=total, ref_frac=frac, reuse_frac=reuse)
        inputs = make_inputs(wl, "cuda")
        main = time_trajectory(wl, inputs, args.warmup, args.steps, attn_timing=True)
        refresh = time_trajectory(wl, inputs, args.warmup, args.steps, delta_max=1)
        tf = main["attn_flops"] / (main["attn_ms"] * 1e-3) / 1e12
        line = {"workload": "sweep", "tokens": total, "ref_frac": frac, "reuse_frac": reuse,
                "n_text": wl.n_text, "n_ref": wl.n_ref, "n_tgt": wl.n_tgt, "blocks": wl.n_blocks,
                "ms_per_step": round(main["total_ms"] / args.steps, 3),
                "always_refresh_ms_per_step": round(refresh["total_ms"] / args.steps, 3),
                "speedup_vs_always_refresh": round(refresh["total_ms"] / main["total_ms"], 3),
                "attn_tflops": round(tf, 1), "attn_frac_of_bf16_peak": round(tf / peaks["bf16_sustained"], 4),
                "modes_step1": [int(x) for x in main["modes"][1, :, 0]]}
        print(json.dumps(line), flush=True)
        lines.append(line)
        del inputs
        torch.cuda.empty_cache()
    if args.out:
        with open(args.out, "w") as f:
            for line in lines:
                f.write(json.dumps(line) + "\n")


def main_ablation(args):
    """Controller ablation (paper Sec. 5.3, Tab. 4) on a synthetic trajectory:
    the trigger cue changes, everything else (executor, stopping rule,
    bounded-age fallback, threshold) is shared; Fixed R3 refreshes every 3 steps
    and reuses otherwise. Reports ms per step, speedup over full computation
    and the fraction of reusing block-steps."""
    import torch
    import __graft_entry__ as ge
    from paper_2609_32415_gb300 import synth
    ge.build()
    wl = synth.make_workload(args.config)
    if args.blocks > 0:
        wl.n_blocks = min(wl.n_blocks, args.blocks)
        wl.ref_drift, wl.tgt_drift = wl.ref_drift[:wl.n_blocks], wl.tgt_drift[:wl.n_blocks]
    inputs = make_inputs(wl, "cuda")
    full = time_trajectory(wl, inputs, args.warmup, args.steps, delta_max=1)
    variants = [("product", "product", None, None), ("change", "change", None, None),
                ("exposure", "exposure", None, None), ("anchor_q_x_exposure", "anchor_product", None, None),
                ("fixed_r3", "product", float("inf"), 3)]
    lines = []
    for name, cue, theta, dm in variants:
        r = time_trajectory(wl, inputs, args.warmup, args.steps, cue=cue, theta=theta, delta_max=dm)
        reuse = float((r["modes"][1:] == 0).mean())
        line = {"workload": args.config, "variant": name, "theta": wl.theta if theta is None else theta,
                "ms_per_step": round(r["total_ms"] / args.steps, 3),
                "full_computation_ms_per_step": round(full["total_ms"] / args.steps, 3),
                "speedup_vs_full": round(full["total_ms"] / r["total_ms"], 3),
                "reuse_fraction_steps_1_on": round(reuse, 3)}
        print(json.dumps(line), flush=True)
        lines.append(line)
    if args.out:
        with open(args.out, "w") as f:
            for line in lines:
                f.write(json.dumps(line) + "\n")
    del inputs
    torch.cuda.empty_cache()


# ----------------------------------------------------------------------------- DiT-block stack
def dit_gemm_flops(wl, C, F, name, modes):
    """FLOPs of one named GEMM launch of a DiT block for the per-sample modes
    (reference rows skipped on REUSE; only their query on BOUNDARY)."""
    tot = 0
    for m in modes:
        m = int(m)
        ref = 0 if m == 0 else wl.n_ref
        if name == "qkv":
            tot += 2 * (wl.n_text + wl.n_tgt) * C * 3 * C
        elif name == "qkv_ref":
            tot += 0 if m == 0 else 2 * wl.n_ref * C * (C if m == 1 else 3 * C)
        elif name == "o_proj":
            tot += 2 * (wl.n_text + wl.n_tgt + ref) * C * C
        elif name in ("mlp1", "mlp2"):
            tot += 2 * (wl.n_text + wl.n_tgt + ref) * C * F
    return tot


def dit_tables(wl, device):
    """Pre-generated stack inputs, AdaLN vectors and weights (nothing is drawn
    inside a timed region)."""
    from paper_2609_32415_gb300 import synth
    di = synth.DiTInputs(wl, device=device)
    h_in = [{r: x.clone() for r, x in di.h_in(t).items()} for t in range(wl.n_steps)]
    mods = {(t, b): di.mods(t, b) for t in range(wl.n_steps) for b in range(wl.n_blocks)}
    weights = [di.weights(b) for b in range(wl.n_blocks)]
    return di, h_in, mods, weights


def time_dit(wl, tables, warmup, steps, theta, delta_max, timing=False, clocks=None):
    import torch
    from paper_2609_32415_gb300 import DiTExecutor
    di, h_in, mods, weights = tables
    ex = DiTExecutor(wl.n_blocks, wl.B, wl.H, wl.d, wl.n_text, wl.n_ref, wl.n_tgt, theta, delta_max,
                     log_steps=wl.n_steps)
    T = wl.n_steps

    def mods_fn(t, b):
        return mods[(t, b)]

    def w_fn(b):
        return weights[b]

    for i in range(warmup):
        ex.step(i % T, h_in[i % T], mods_fn, w_fn)
    torch.cuda.synchronize()
    gemm_ev, attn_ev = [], []
    if timing:
        def ghook(phase, name, t, b):
            if phase == "pre":
                e = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                e[0].record()
                gemm_ev.append((name, t, b, e))
            else:
                gemm_ev[-1][3][1].record()

        def ahook(phase, t, b):
            if phase == "pre":
                e = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                e[0].record()
                attn_ev.append((t, b, e))
            else:
                attn_ev[-1][2][1].record()
        ex.gemm_hook, ex.attn_hook = ghook, ahook
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
    torch.cuda.synchronize()
    if clocks:
        clocks.start()
    ev[0].record()
    for k in range(steps):
        t = (warmup + k) % T
        ex.step(t, h_in[t], mods_fn, w_fn)
        ev[k + 1].record()
    torch.cuda.synchronize()
    clk = clocks.stop() if clocks else None
    ex.gemm_hook = ex.attn_hook = None
    ex.check()
    modes = ex.modes.cpu().numpy()
    res = {"total_ms": ev[0].elapsed_time(ev[-1]), "per_step_ms": [ev[k].elapsed_time(ev[k + 1]) for k in range(steps)],
           "modes": modes, "gbar": ex.gbar.cpu().numpy(), "clocks": clk,
           "steps_t": [(warmup + k) % T for k in range(steps)]}
    if timing:
        g_ms, g_fl = 0.0, 0
        for name, t, b, (e0, e1) in gemm_ev:
            g_ms += e0.elapsed_time(e1)
            g_fl += dit_gemm_flops(wl, ex.C, ex.F, name, modes[t, b])
        a_ms, a_fl = 0.0, 0
        for t, b, (e0, e1) in attn_ev:
            a_ms += e0.elapsed_time(e1)
            a_fl += sum(attn_flops(wl, m) for m in modes[t, b])
        res.update(gemm_ms=g_ms, gemm_flops=g_fl, gemm_launches=len(gemm_ev), attn_ms=a_ms, attn_flops=a_fl,
                   attn_launches=len(attn_ev))
    del ex
    return res


def calibrate_dit_theta(wl, tables):
    """theta just above the largest step-1 score among the first half of the
    stack (scores taken with every block reusing at step 1), so the first
    half reuses at step 1 and the boundary falls in the second half."""
    r = time_dit(wl, tables, 0, 2, float("inf"), max(2, wl.delta_max))
    g = r["gbar"][1, :, 0]
    half = max(1, wl.n_blocks // 2)
    return float(max(g[:half])) * 1.0001, [round(float(x), 5) for x in g]


def cublas_context_tflops(M, K, N, reps=20):
    """torch.matmul (cuBLAS) on one GEMM shape of the stack, timed the same
    way: context for the tcgen05 GEMM's rate."""
    import torch
    a = torch.randn((M, K), device="cuda").to(torch.bfloat16)
    w = torch.randn((N, K), device="cuda").to(torch.bfloat16)
    out = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    for _ in range(3):
        torch.matmul(a, w.t(), out=out)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda._sleep(10_000_000)
    e0.record()
    for _ in range(reps):
        torch.matmul(a, w.t(), out=out)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    del a, w, out
    return 2.0 * M * N * K / ms / 1e9


def dit_cpu_oracle_sample(wl, tables, budget_s):
    """Time the CPU oracle's DiT block (oracle/dit.py, fp64) on a bounded
    sample: R target rows of block 0 through the modulated LN + QKV + norm +
    RoPE, their attention against all N keys, and the output projection + MLP.
    Returns seconds per row for the linear part and per query row for the
    attention, and the sample size."""
    import numpy as np
    import torch
    import oracle
    from oracle import dit as odit

    def f64(t):
        return oracle.bf16_to_f64(t.contiguous().cpu().view(torch.int16).numpy().view(np.uint16))

    di, h_in, mods, weights = tables
    W = {k: (f64(v) if k.startswith("w_") else v.double().cpu().numpy()) for k, v in weights[0]["image"].items()}
    md = {k: v[0].double().cpu().numpy() for k, v in mods[(1, 0)]["image"].items()}
    C = wl.H * wl.d
    rng = np.random.default_rng(0)
    keys = rng.standard_normal((wl.H, wl.N, wl.d)) / math.sqrt(wl.d)
    vals = rng.standard_normal((wl.H, wl.N, wl.d)) / math.sqrt(wl.d)
    nth = oracle.default_threads()
    R = 4
    while True:
        h = f64(h_in[1]["tgt"][0, :R])
        pos = wl.n_text + wl.n_ref + np.arange(R)
        t0 = time.perf_counter()
        q, _, _ = odit.qkv_project(h, md, W, pos, wl.H, wl.d)
        t1 = time.perf_counter()
        o, _ = oracle.joint_attention(q, keys, vals, 1.0 / math.sqrt(wl.d),
                                      ref_range=(wl.n_text, wl.n_text + wl.n_ref), nthreads=nth)
        t2 = time.perf_counter()
        odit.post_attention(h, odit.round_bf16(o), md, W)
        t3 = time.perf_counter()
        total = t3 - t0
        if total > budget_s / 3 or R >= 256:
            break
        R = min(256, max(R * 2, int(R * (budget_s / 2.5) / max(total, 1e-3))))
    return {"lin_s_per_row": ((t1 - t0) + (t3 - t2)) / R, "attn_s_per_row": (t2 - t1) / R, "rows": R,
            "sample_s": total, "threads": nth, "C": C}


def run_dit(args, wl, with_cpu=True, with_context=True):
    """Time the DiT-block stack on the workload's row partition (theta
    calibrated as below) against always-refresh; returns the summary dict."""
    import torch
    peaks = load_peaks()
    tables = dit_tables(wl, "cuda")
    torch.cuda.synchronize()
    theta, g1 = calibrate_dit_theta(wl, tables)
    clocks = Clocks(0)
    main = time_dit(wl, tables, args.warmup, args.steps, theta, wl.delta_max, timing=True, clocks=clocks)
    refresh = None if args.no_refresh_baseline else time_dit(wl, tables, args.warmup, args.steps, theta, 1)
    C = wl.H * wl.d
    gt = main["gemm_flops"] / (main["gemm_ms"] * 1e-3) / 1e12
    at = main["attn_flops"] / (main["attn_ms"] * 1e-3) / 1e12
    ms = main["total_ms"] / args.steps
    line = {
        "workload": "DiT-block stack: " + WORKLOAD_NAMES[wl.name] + (
            " (first %d blocks)" % wl.n_blocks if args.blocks > 0 else ""),
        "block": "dual-stream MMDiT, C=%d, MLP 4C, random weights (%.1f GB)" % (
            C, sum(v.numel() * v.element_size() for w in tables[3] for st in w.values() for v in st.values()) / 1e9),
        "metric": "ms per denoising step of the DiT-block stack, vs always-refresh",
        "value": round(ms, 3), "unit": "ms/step", "higher_is_better": False, "steps": args.steps,
        "warmup": args.warmup, "dtype": "bf16", "data": "synthetic (seeded inputs, AdaLN vectors and weights)",
        "theta": round(theta, 6), "theta_recipe": "just above the largest step-1 score of the first half of the stack",
        "step1_scores_all_reuse": g1,
        "per_step_ms": [round(x, 3) for x in main["per_step_ms"]],
        "timed_trajectory_steps": main["steps_t"],
        "modes_per_step": {str(t): [int(x) for x in main["modes"][t, :, 0]] for t in sorted(set(main["steps_t"]))},
        "gemm_tflops": round(gt, 1), "gemm_frac_of_bf16_peak": round(gt / peaks["bf16_sustained"], 4),
        "gemm_share_of_step": round(main["gemm_ms"] / main["total_ms"], 4),
        "attn_tflops": round(at, 1), "attn_share_of_step": round(main["attn_ms"] / main["total_ms"], 4),
        "peak": peaks["bf16_sustained"], "peak_kind": "%s, sustained bf16" % peaks["source"],
        "clocks": main["clocks"],
    }
    if with_context:
        line["same_shape_cublas_tflops"] = round(cublas_context_tflops(wl.n_text + wl.n_ref + wl.n_tgt, C, 3 * C), 1)
    if with_cpu:
        smp = dit_cpu_oracle_sample(wl, tables, args.cpu_budget_s)
        per_step = []
        for t in main["steps_t"]:
            ms_t = 0.0
            for b_modes in main["modes"][t]:
                for m in b_modes:
                    rows = wl.N if int(m) != 0 else wl.n_text + wl.n_tgt
                    ms_t += 1000.0 * rows * (smp["lin_s_per_row"] + smp["attn_s_per_row"])
            per_step.append(ms_t)
        line["cpu_baseline"] = {
            "value": round(statistics.mean(per_step), 1), "unit": "ms/step", "cores": smp["threads"], "kind": "oracle",
            "sample": "fp64 DiT-block oracle, %d target rows of block 0 through LN + QKV + norm + RoPE, their "
                      "attention against all %d keys, output projection + MLP (%.1f s); extrapolated per row to "
                      "the executed rows of every block of the timed steps" % (smp["rows"], wl.N, smp["sample_s"])}
    if refresh is not None:
        rms = refresh["total_ms"] / args.steps
        line["always_refresh_ms_per_step"] = round(rms, 3)
        line["speedup_vs_always_refresh"] = round(rms / ms, 3)
    del tables
    torch.cuda.empty_cache()
    return line


def main_dit(args):
    import __graft_entry__ as ge
    from paper_2609_32415_gb300 import synth
    ge.build()
    wl = synth.make_workload(args.config)
    if args.blocks > 0:
        wl.n_blocks = min(wl.n_blocks, args.blocks)
    emit(run_dit(args, wl, with_cpu=not args.no_cpu_baseline), args)

def main():
    args = parse_args()
    if args.dit:
        main_dit(args)
        return
    if args.ablation:
        main_ablation(args)
        return
    if args.sweep:
        main_sweep(args)
        return
    if args.impl == "reference":
        main_reference(args)
    else:
        main_ours(args)


if __name__ == "__main__":
    main()
