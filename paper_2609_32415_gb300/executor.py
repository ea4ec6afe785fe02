"""Algorithm 1's host loop over the C ABI: one denoising step = for each block,
Q change -> gate -> cache materialisation -> joint attention, enqueued with the
decisions kept on the device (no host sync inside a step). The Q change and the
gate are one launch from step 1 on (refadapt_q_delta_gate); the cache
materialisation rides in the attention (fused_cache). By default a block's
decision runs on a side stream beside the previous block's attention, and
consecutive attentions alternate between two streams (see
Executor.step); overlap=False keeps every launch on the caller's stream.

Per block b the executor owns the cache state of paper Eq. 11: reference K and
V, the cached reference hidden state (here the reference query, which is what
restoring the hidden state at a boundary produces in this hot path) and a_b.
REUSE and BOUNDARY blocks read reference Q/K/V from that cache slot (the
values of the last materialisation). COMPUTE / FULL blocks read this step's
reference rows, and the joint-attention kernel copies them into the slot in
the same pass (fused_cache, the default); fused_cache=False refreshes the slot
with refadapt_ref_cache_update first and the attention reads the slot.
"""
import contextlib

import torch

from . import api
from ._lib import RA_MODE_BOUNDARY, RA_MODE_COMPUTE, RA_MODE_FULL, RA_MODE_REUSE  # noqa: F401

ROLES = ("text", "ref", "tgt")


def roles_from_joint(X, offsets, n):
    """Role views of a joint tensor X[3, B, H, N, d] (q, k, v stacked).

    Returns dict role -> (q, k, v), each a [B, H, n_role, d] view."""
    out = {}
    for r in ROLES:
        o, k = offsets[r], n[r]
        out[r] = (X[0, :, :, o:o + k, :], X[1, :, :, o:o + k, :], X[2, :, :, o:o + k, :])
    return out


CUES = {"product": 0, "change": 1, "exposure": 2, "anchor_product": 0}


class Executor:
    """Algorithm 1 over a block stack.

    ``cue`` picks the reactivation trigger of the controller ablation (paper
    Sec. 5.3, Tab. 4): "product" (D x M, the method), "change" (target-Q change
    only), "exposure" (M only), or "anchor_product" (the change of the target
    query to its value at the block's last materialisation, App. A.2, times M;
    the executor keeps that anchor per block). The fixed-interval baseline is
    theta = inf with delta_max = the interval.

    ``diagnostics`` adds, after every block, the staleness diagnostics of
    Sec. 3.3 / App. A.2 on the target rows 0, k, 2k, ... (k =
    ``diag_row_stride``), all through the same entry points: E_K, E_V (Eq. 7,
    this step's reference K, V against the cache slot, refadapt_q_delta), a
    second attention pass of the text and sampled target rows with the fresh
    reference K/V (Eq. 8; its mass partials give the fresh exposure), and I_KV
    (Eq. 10, refadapt_q_delta of the executed target output against it).
    Logged per step in E_K, E_V, I_KV [steps, blocks, B, H] and M_fresh_part
    [steps, blocks, B, H, tiles].

    ``sample_stride`` k > 1 takes D and M over the sampled target-query rows
    0, k, 2k, ... (Eq. 4, Algorithm 1 "sampled target queries"): D from the
    strided target Q views, M from the attention's mass partials over those
    rows only. k = 1 uses every row.

    ``overlap`` (default) runs step() on three streams of its own (a side
    stream for the decisions, and the cache updates when they are not fused;
    two higher-priority streams for the attentions), forked from and joined
    to the caller's stream per step; the results equal the one-stream order
    bit for bit.

    ``fused_cache`` (default) lets the attention of a materialising block
    write its cache slot (refadapt_joint_attn's ref_fresh arguments) instead
    of a refadapt_ref_cache_update launch before it; the results are the same.
    """

    def __init__(self, n_blocks, B, H, d, n_text, n_ref, n_tgt, theta, delta_max, eps=1e-6,
                 mass_rows=0, forced_boundary=-1, softmax_scale=0.0, bias=None, log_steps=8,
                 device="cuda", cue="product", diagnostics=False, diag_row_stride=1, sample_stride=1,
                 overlap=True, fused_cache=True, nvtx=False):
        if cue not in CUES:
            raise ValueError("unknown cue %r" % (cue,))
        self.cue = cue
        self.n_blocks, self.B, self.H, self.d = n_blocks, B, H, d
        self.n = {"text": n_text, "ref": n_ref, "tgt": n_tgt}
        self.theta, self.delta_max, self.eps = float(theta), int(delta_max), float(eps)
        self.mass_rows, self.forced_boundary = int(mass_rows), int(forced_boundary)
        self.softmax_scale = float(softmax_scale)
        dev = torch.device(device)
        self.bias = None if bias is None else torch.as_tensor(bias, dtype=torch.float32, device=dev).contiguous()
        shape = (n_blocks, B, H, n_ref, d)
        self.cache_k = torch.zeros(shape, dtype=torch.bfloat16, device=dev)
        self.cache_v = torch.zeros(shape, dtype=torch.bfloat16, device=dev)
        self.cache_x = torch.zeros(shape, dtype=torch.bfloat16, device=dev)
        self.a_b = torch.full((n_blocks, B), -1, dtype=torch.int32, device=dev)
        self.mpl = api.refadapt_mass_partial_len(n_text, n_tgt)
        self.mass = torch.zeros((n_blocks, B, H, self.mpl), dtype=torch.float32, device=dev)
        k = self.sample_stride = max(1, int(sample_stride))
        self.mass_row_count = (n_tgt + k - 1) // k + ((n_text + k - 1) // k if mass_rows == 1 else 0)
        self.D = torch.zeros((n_blocks, B, H), dtype=torch.float32, device=dev)
        self.log_steps = int(log_steps)
        self.modes = torch.full((self.log_steps, n_blocks, B), -1, dtype=torch.int32, device=dev)
        self.gbar = torch.zeros((self.log_steps, n_blocks, B), dtype=torch.float32, device=dev)
        self.M = torch.zeros((self.log_steps, n_blocks, B, H), dtype=torch.float32, device=dev)
        self.workspace = api.q_delta_workspace(B, H, dev)
        self.state = api.new_state(B, dev)
        # overlap: step() runs each block's decision (Q change with the gate)
        # on a side stream one block ahead, in the previous attention's tail
        # wave (SMs its last wave leaves idle); see step().
        self.overlap = bool(overlap)
        self.fused_cache = bool(fused_cache)
        if self.overlap:
            # The attentions run on a high-priority stream and the side work on
            # a default-priority one: the CTA scheduler serves pending attention
            # CTAs first, so the side kernels take only SMs the attention leaves
            # idle.
            # Consecutive blocks' attentions alternate between two such
            # streams: they share no data, so block b + 1's first CTAs may take
            # the SMs block b's last wave leaves idle.
            lo, hi = torch.cuda.Stream.priority_range()
            self._mains = [torch.cuda.Stream(device=dev, priority=hi) for _ in range(2)]
            self._side = torch.cuda.Stream(device=dev, priority=lo)
            self._fork = torch.cuda.Event()
            self._join = [torch.cuda.Event() for _ in range(2)]
            self._decided = [torch.cuda.Event() for _ in range(n_blocks)]
            self._attn_done = [torch.cuda.Event() for _ in range(n_blocks)]
        self.err = torch.zeros(1, dtype=torch.int32, device=dev)
        self._prev_qtgt = [None] * n_blocks
        self.anchor = (torch.zeros((n_blocks, B, H, n_tgt, d), dtype=torch.bfloat16, device=dev)
                       if cue == "anchor_product" else None)
        self.diagnostics = bool(diagnostics)
        self.diag_row_stride = int(diag_row_stride)
        if self.diagnostics:
            # diagnostics run on the attention streams: one set per block parity
            self.workspace_diag = [api.q_delta_workspace(B, H, dev) for _ in range(2)]
            k = self.diag_row_stride
            n_s = (n_tgt + k - 1) // k
            self.n_tgt_sampled = n_s
            self.E_K = torch.zeros((self.log_steps, n_blocks, B, H), dtype=torch.float32, device=dev)
            self.E_V = torch.zeros_like(self.E_K)
            self.I_KV = torch.zeros_like(self.E_K)
            self.mpl_fresh = api.refadapt_mass_partial_len(n_text, n_s)
            self.M_fresh_part = torch.zeros((self.log_steps, n_blocks, B, H, self.mpl_fresh), dtype=torch.float32,
                                            device=dev)
            self._o_fresh = [{"text": torch.empty((B, H, n_text, d), dtype=torch.bfloat16, device=dev),
                              "tgt": torch.empty((B, H, n_s, d), dtype=torch.bfloat16, device=dev)} for _ in range(2)]
        self._out = [None, None]
        self.attn_hook = None   # optional callable(phase in {"pre", "post"}, t, b), e.g. CUDA events
        self.nvtx = bool(nvtx)

    def _range(self, name):
        """An NVTX range around the launches it encloses (nvtx=True), for
        timeline profilers; nothing otherwise."""
        return torch.cuda.nvtx.range(name) if self.nvtx else contextlib.nullcontext()

    def scratch_outputs(self, parity=0):
        """A set of O buffers (text, ref, tgt) reused by every block of one
        parity (step() gives blocks of the two parities different sets: their
        attentions may run at the same time)."""
        if self._out[parity] is None:
            self._out[parity] = {r: torch.empty((self.B, self.H, self.n[r], self.d), dtype=torch.bfloat16,
                                                device=self.cache_k.device) for r in ROLES}
        return self._out[parity]

    def block(self, t, b, x, out, log_index=None, stream=None):
        """Enqueue block b of step t. x: dict role -> (q, k, v) [B, H, n, d] views;
        out: dict role -> O [B, H, n, d]."""
        self.gate_block(t, b, x["tgt"][0], log_index, stream)
        self.attend_block(t, b, x, out, log_index, stream)

    def gate_block(self, t, b, qt, log_index=None, stream=None):
        """The decision half of block b of step t (Eq. 1 on the target query qt,
        then Algorithm 1's gate into modes[.., b]). It reads only qt, the
        previous step's target query and mass partials of this block and the
        controller state left by the gates of blocks < b, so a step's gates may
        all be enqueued before its attentions (the host can then read the
        modes first, e.g. to skip copying reference rows a reusing block does
        not read). The caller keeps qt alive until step t + 1's gate of this
        block has been enqueued (it is read as q_{t-1})."""
        li = (t % self.log_steps) if log_index is None else log_index
        mode = self.modes[li, b]
        have_prev = t >= 1 and self._prev_qtgt[b] is not None
        with self._range("t%d b%d decision" % (t, b)):
            self._decide(t, b, qt, li, mode, have_prev, stream)
        self._prev_qtgt[b] = qt

    def _decide(self, t, b, qt, li, mode, have_prev, stream):
        if have_prev:
            # Eq. 1 and the decision in one call (one launch on the cluster path)
            ref_q = self.anchor[b] if self.anchor is not None else self._prev_qtgt[b]
            k = self.sample_stride
            api.refadapt_q_delta_gate(qt[:, :, ::k, :] if k > 1 else qt, ref_q[:, :, ::k, :] if k > 1 else ref_q,
                                      self.D[b], self.workspace, t, b, self.state, mode, self.theta,
                                      self.delta_max, self.mass[b], self.mass_row_count, eps=self.eps,
                                      forced_boundary=self.forced_boundary, gbar_out=self.gbar[li, b],
                                      m_out=self.M[li, b], cue=CUES[self.cue], stream=stream)
        else:
            api.refadapt_gate(t, b, self.state, mode, self.theta, self.delta_max, self.B, self.H,
                              mass_row_count=self.mass_row_count, forced_boundary=self.forced_boundary,
                              gbar_out=self.gbar[li, b], m_out=self.M[li, b], cue=CUES[self.cue], stream=stream)
        if self.anchor is not None:
            # Materialising blocks move their anchor to this step's target Q (the
            # V copy is skipped: source and destination coincide).
            an = self.anchor[b]
            api.refadapt_ref_cache_update(qt, an, an, an, mode, t, None, stream=stream)

    def attend_block(self, t, b, x, out, log_index=None, stream=None):
        """The attention half of block b of step t, after gate_block(t, b): the
        reference cache update (materialising samples) and the joint attention
        with the mass partials. x[ref] is read only for samples whose mode is
        COMPUTE or FULL."""
        if not self.fused_cache:
            self.update_cache(t, b, x, log_index, stream)
        self.attend(t, b, x, out, log_index, stream)

    def update_cache(self, t, b, x, log_index=None, stream=None):
        """Block b's reference cache update of step t (after its gate):
        materialising samples copy their reference K, V and query into the
        cache slot and stamp a_b = t."""
        li = (t % self.log_steps) if log_index is None else log_index
        qr, kr, vr = x["ref"]
        api.refadapt_ref_cache_update(kr, vr, self.cache_k[b], self.cache_v[b], self.modes[li, b], t, self.a_b[b],
                                      x_src=qr, x_cache=self.cache_x[b], stream=stream)

    def attend(self, t, b, x, out, log_index=None, stream=None):
        """Block b's joint attention of step t (after its gate, and after its
        cache update unless fused_cache), with the mass partials the next
        step's gate reads. With fused_cache, materialising samples read x[ref]
        and the kernel writes it into the cache slot and stamps a_b = t."""
        li = (t % self.log_steps) if log_index is None else log_index
        mode = self.modes[li, b]
        qt = x["tgt"][0]
        if self.attn_hook is not None:
            self.attn_hook("pre", t, b)
        with self._range("t%d b%d attention" % (t, b)):
            self._attend(t, b, x, out, mode, qt, stream)
        if self.attn_hook is not None:
            self.attn_hook("post", t, b)
        if self.diagnostics:
            self._diagnose(t, b, li, x, out, stream)

    def _attend(self, t, b, x, out, mode, qt, stream):
        api.refadapt_joint_attn(
            (x["text"][0], self.cache_x[b], qt),
            (x["text"][1], self.cache_k[b], x["tgt"][1]),
            (x["text"][2], self.cache_v[b], x["tgt"][2]),
            (out["text"], out["ref"], out["tgt"]),
            self.mass[b], mode=mode, softmax_scale=self.softmax_scale, ref_logit_bias=self.bias,
            mass_rows=self.mass_rows, err_word=self.err, mass_row_stride=self.sample_stride,
            ref_fresh=x["ref"] if self.fused_cache else None,
            a_b=self.a_b[b] if self.fused_cache else None, step=t, stream=stream)

    def _diagnose(self, t, b, li, x, out, stream):
        k = self.diag_row_stride
        ws, of = self.workspace_diag[b % 2], self._o_fresh[b % 2]
        qr, kr, vr = x["ref"]
        api.refadapt_q_delta(kr, self.cache_k[b], self.E_K[li, b], ws, self.eps, stream)
        api.refadapt_q_delta(vr, self.cache_v[b], self.E_V[li, b], ws, self.eps, stream)
        q_s = x["tgt"][0][:, :, ::k, :]
        api.refadapt_joint_attn(
            (x["text"][0], None, q_s), (x["text"][1], kr, x["tgt"][1]), (x["text"][2], vr, x["tgt"][2]),
            (of["text"], None, of["tgt"]), self.M_fresh_part[li, b],
            softmax_scale=self.softmax_scale, ref_logit_bias=self.bias, err_word=self.err, stream=stream)
        api.refadapt_q_delta(out["tgt"][:, :, ::k, :], of["tgt"], self.I_KV[li, b], ws, self.eps, stream)

    def step(self, t, inputs, outs=None, log_index=None, stream=None, after_block=None):
        """Enqueue one denoising step. inputs[b]: dict role -> (q, k, v);
        outs[b] (optional): dict role -> O. The caller keeps step t's target Q
        alive until step t + 1 has been enqueued (it is read as q_{t-1}).

        With overlap (the default) block b's decision (the Q change with the
        gate; the cache update too when it is not fused into the attention)
        runs on a side stream, ordered after the step's start and after the
        attention of block b - 2, and block b's attention waits for it: so it
        runs during the attention of block b - 1, whose last wave
        leaves SMs idle (the attentions run on higher-priority streams, so
        their pending CTAs go first). Consecutive attentions alternate between
        two streams: they share no data (inputs, cache slot, outputs and mass
        partials are the block's own), so block b + 1's first CTAs may start in
        block b's last wave. Every stream forks from the caller's stream at
        the step's start and joins it at the end. A gate reads only its
        block's target queries, the block's previous-step mass partials and
        the controller state of the
        blocks before it, never an attention of the same step, so the results
        are those of the one-stream order. Every event is recorded inside the
        step, which can be captured as a CUDA graph."""
        if not self.overlap:
            for b in range(self.n_blocks):
                out = outs[b] if outs is not None else self.scratch_outputs(b % 2)
                self.block(t, b, inputs[b], out, log_index, stream)
                if after_block is not None:
                    after_block(t, b)
            return
        caller = torch.cuda.current_stream() if stream is None else stream
        side = self._side
        self._fork.record(caller)
        for m in self._mains:
            m.wait_event(self._fork)
        side.wait_event(self._fork)  # everything enqueued before this step (the previous step's attentions)
        for b in range(self.n_blocks):
            main = self._mains[b % 2]
            out = outs[b] if outs is not None else self.scratch_outputs(b % 2)
            if b >= 2:
                side.wait_event(self._attn_done[b - 2])
            with torch.cuda.stream(side):
                self.gate_block(t, b, inputs[b]["tgt"][0], log_index)
                if not self.fused_cache:
                    self.update_cache(t, b, inputs[b], log_index)
                self._decided[b].record(side)
            with torch.cuda.stream(main):
                main.wait_event(self._decided[b])
                self.attend(t, b, inputs[b], out, log_index)
                self._attn_done[b].record(main)
            if after_block is not None:
                with torch.cuda.stream(main):
                    after_block(t, b)
        for m, j in zip(self._mains, self._join):  # the side stream's last work is behind a main wait
            j.record(m)
            caller.wait_event(j)

    def capture_step(self, t, inputs, outs=None, log_index=None):
        """Capture step t (every block's launches, on one stream) as a CUDA graph.

        Steps must be captured in trajectory order (the Q change of step t
        reads the target Q handed to step t-1). Capturing runs nothing;
        replaying the graph enqueues the step with the pointers and step index
        baked in. Make one eager call of each entry point first (first calls
        set kernel attributes and look up driver entry points)."""
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.step(t, inputs, outs, log_index)
        return g

    def exposure_summary(self, n_steps, fresh=False):
        """The exposure summaries of Sec. 3.2 over the logged steps
        0 .. n_steps - 1 of a trajectory (n_steps <= log_steps, read after the
        steps have run): the head-mean exposure of Eq. 5, Mbar [n_steps,
        blocks, B], and its mean adjacent-step change of Eq. 6 in percentage
        points, Delta [blocks, B] (fp64 numpy arrays).

        fresh=False takes the executed attention's exposure, the one the
        controller reads: step t's is what step t + 1's gate logged, the last
        step's comes from the current mass partials. fresh=True takes the
        fresh-reference pass of the diagnostics (A^fresh, the paper's
        summaries); it needs diagnostics=True. A summary of logged results
        for analysis, read back to the host; no part of a step."""
        import numpy as np
        T = int(n_steps)
        if T < 2 or T > self.log_steps:
            raise ValueError("exposure_summary: need 2 <= n_steps <= log_steps (%d)" % self.log_steps)
        if fresh:
            if not self.diagnostics:
                raise ValueError("exposure_summary(fresh=True) needs Executor(diagnostics=True)")
            M = self.M_fresh_part[:T].double().sum(-1).cpu().numpy() / float(self.n_tgt_sampled)
        else:
            M = np.empty((T, self.n_blocks, self.B, self.H))
            M[:T - 1] = self.M[1:T].double().cpu().numpy()
            M[T - 1] = self.mass.double().sum(-1).cpu().numpy() / float(self.mass_row_count)
        Mbar = M.mean(axis=-1)
        Delta = 100.0 * np.abs(np.diff(Mbar, axis=0)).sum(axis=0) / (T - 1)
        return Mbar, Delta

    # Cross-step state of Algorithm 1 (Eq. 11's block caches and a_b, the
    # controller state, the previous step's mass partials and Q change) and the
    # per-step logs; the Q-change workspace is zero between calls and is not
    # state.
    _STATE = ("cache_k", "cache_v", "cache_x", "a_b", "mass", "D", "state", "modes", "gbar", "M")
    _STATE_OPT = ("anchor", "E_K", "E_V", "I_KV", "M_fresh_part")

    def snapshot(self):
        """A host copy of everything a trajectory carries from one step to
        the next (after the enqueued work has finished): restore() on an
        executor of the same configuration continues the trajectory with the
        same results, bit for bit. The previous step's target queries are
        copied too (the next step's Q change reads them)."""
        torch.cuda.synchronize(self.cache_k.device)
        snap = {k: getattr(self, k).detach().cpu().clone() for k in self._STATE}
        for k in self._STATE_OPT:
            if getattr(self, k, None) is not None:
                snap[k] = getattr(self, k).detach().cpu().clone()
        snap["prev_qtgt"] = [None if q is None else q.detach().cpu().clone() for q in self._prev_qtgt]
        snap["config"] = self._config()
        return snap

    def restore(self, snap):
        """Load a snapshot() taken from an executor of the same configuration."""
        if snap["config"] != self._config():
            raise ValueError("restore: the snapshot's configuration differs: %r vs %r"
                             % (snap["config"], self._config()))
        for k in self._STATE + self._STATE_OPT:
            if k in snap:
                getattr(self, k).copy_(snap[k])
        dev = self.cache_k.device
        self._prev_qtgt = [None if q is None else q.to(dev) for q in snap["prev_qtgt"]]
        torch.cuda.synchronize(dev)

    def _config(self):
        return (self.n_blocks, self.B, self.H, self.d, self.n["text"], self.n["ref"], self.n["tgt"],
                self.log_steps, self.mpl, self.cue, self.sample_stride, self.mass_rows, self.diagnostics)

    def trace(self, n_steps):
        """The observation record of the logged steps 0 .. n_steps - 1 (read
        after they have run): per (step, block) the mode and gbar of every
        sample, the head-mean exposure the gate read (Eq. 5 on M_{t-1}; None at
        t = 0) and a_b now. A list of dicts, one per (step, block), for a JSONL
        log; one host read of the logs."""
        T = int(n_steps)
        if T < 1 or T > self.log_steps:
            raise ValueError("trace: need 1 <= n_steps <= log_steps (%d)" % self.log_steps)
        modes = self.modes[:T].cpu().tolist()
        gbar = self.gbar[:T].double().cpu().tolist()
        mbar = self.M[:T].double().mean(-1).cpu().tolist()
        a_b = self.a_b.cpu().tolist()
        out = []
        for t in range(T):
            for b in range(self.n_blocks):
                out.append({"t": t, "b": b, "mode": modes[t][b],
                            "gbar": [None if g != g else g for g in gbar[t][b]],
                            "m_bar_read": mbar[t][b] if t >= 1 else None, "a_b": a_b[b]})
        return out

    def check(self, stream=None):
        api.refadapt_check_error(self.err, stream)
