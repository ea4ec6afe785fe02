"""Algorithm 1 over a stack of DiT blocks, through the C ABI.

The block is a dual-stream MMDiT block (text rows use the text stream's
weights, reference and target rows the image stream's): modulated LayerNorm,
QKV projection with per-head RMS norm and RoPE, joint [text; reference;
target] attention, gated output projection, modulated LayerNorm, gated GELU
MLP. The paper's method decides per block and sample what happens to the
reference rows (Algorithm 1; App. A.3, A.4):

  REUSE     reference rows do nothing: no LayerNorm, projection, attention
            rows or MLP; text and target rows attend to the cached reference
            K/V of the block.
  BOUNDARY  the reference rows restore the block's cached input hidden state
            H_b, form their query (their K/V stay the cached ones), attend,
            finish the block and store the next block's cached hidden state
            H_{b+1}.
  COMPUTE / FULL  the reference rows form Q, K, V from H_b; K and V go
            straight into the block's cache slot (a_b = t); all rows attend;
            the reference output is stored as H_{b+1}.

D (Eq. 1) is taken on the post-RoPE target query the QKV projection of this
block just wrote, against the previous step's (kept per block); M comes from
the executed attention's mass partials. Every kernel reads the mode from
device memory (refadapt_gate writes it), so a step is enqueued without a host
synchronisation and can be captured as a CUDA graph.

Buffers: the caches (reference K/V per block, H_b for b = 0..n_blocks, the
previous target Q per block, mass partials) persist across steps; the
activations (LN outputs, Q/K/V, attention outputs, MLP hidden) are one
shared set reused by every block. The running text and target hidden states
are updated in place by the gated-residual epilogues.
"""
import torch

from . import api
from ._lib import RA_EPI_GELU, RA_EPI_QKV, RA_EPI_RESID

ROLES = ("text", "ref", "tgt")
STREAM_OF = {"text": "text", "ref": "image", "tgt": "image"}
CUES = {"product": 0, "change": 1, "exposure": 2}


class DiTExecutor:
    def __init__(self, n_blocks, B, H, d, n_text, n_ref, n_tgt, theta, delta_max, eps=1e-6, mlp_ratio=4,
                 forced_boundary=-1, mass_rows=0, ln_eps=1e-6, norm_eps=1e-6, rope_base=10000.0, log_steps=8,
                 cue="product", device="cuda"):
        if cue not in CUES:
            raise ValueError("unknown cue %r" % (cue,))
        dev = torch.device(device)
        self.n_blocks, self.B, self.H, self.d = n_blocks, B, H, d
        self.C = C = H * d
        self.F = F = mlp_ratio * C
        self.n = {"text": n_text, "ref": n_ref, "tgt": n_tgt}
        self.theta, self.delta_max, self.eps = float(theta), int(delta_max), float(eps)
        self.forced_boundary, self.mass_rows, self.cue = int(forced_boundary), int(mass_rows), cue
        self.ln_eps, self.norm_eps = float(ln_eps), float(norm_eps)
        bf = dict(dtype=torch.bfloat16, device=dev)
        # persistent state
        self.cache_k = torch.zeros((n_blocks, B, H, n_ref, d), **bf)
        self.cache_v = torch.zeros((n_blocks, B, H, n_ref, d), **bf)
        self.hbar = [None] + [torch.zeros((B, n_ref, C), **bf) for _ in range(n_blocks)]
        self.q_tgt = torch.zeros((2, n_blocks, B, H, n_tgt, d), **bf)   # ping-pong over steps
        self.a_b = torch.full((n_blocks, B), -1, dtype=torch.int32, device=dev)
        self.mpl = api.refadapt_mass_partial_len(n_text, n_tgt)
        self.mass = torch.zeros((n_blocks, B, H, self.mpl), dtype=torch.float32, device=dev)
        self.mass_row_count = n_tgt + (n_text if mass_rows == 1 else 0)
        self.D = torch.zeros((n_blocks, B, H), dtype=torch.float32, device=dev)
        self.log_steps = int(log_steps)
        self.modes = torch.full((self.log_steps, n_blocks, B), -1, dtype=torch.int32, device=dev)
        self.gbar = torch.zeros((self.log_steps, n_blocks, B), dtype=torch.float32, device=dev)
        self.M = torch.zeros((self.log_steps, n_blocks, B, H), dtype=torch.float32, device=dev)
        self.workspace = api.q_delta_workspace(B, H, dev)
        self.state = api.new_state(B, dev)
        self.err = torch.zeros(1, dtype=torch.int32, device=dev)
        self.rope = api.rope_table(n_text + n_ref + n_tgt, d, rope_base, dev)
        # activations shared by all blocks
        self.h = {r: torch.zeros((B, self.n[r], C), **bf) for r in ("text", "tgt")}   # running hidden state
        self.h1 = {r: torch.empty((B, self.n[r], C), **bf) for r in ROLES}
        self.x = {r: torch.empty((B, self.n[r], C), **bf) for r in ROLES}
        self.u = {r: torch.empty((B, self.n[r], F), **bf) for r in ROLES}
        self.o = {r: torch.empty((B, self.n[r], C), **bf) for r in ROLES}
        self.qkv = {r: [torch.empty((B, H, self.n[r], d), **bf) for _ in range(3)] for r in ("text", "tgt")}
        self.q_ref = torch.empty((B, H, n_ref, d), **bf)
        self.pos0 = {"text": 0, "ref": n_text, "tgt": n_text + n_ref}
        self.gemm_hook = None   # optional callable(phase, name, t, b), e.g. CUDA events
        self.attn_hook = None

    def _heads(self, t):
        """[B, n, C] token-major buffer viewed as [B, H, n, d]."""
        B, n, _ = t.shape
        return t.view(B, n, self.H, self.d).permute(0, 2, 1, 3)

    def _gemm(self, name, t, b, *args, **kw):
        if self.gemm_hook is not None:
            self.gemm_hook("pre", name, t, b)
        api.refadapt_gemm(*args, **kw)
        if self.gemm_hook is not None:
            self.gemm_hook("post", name, t, b)

    def block(self, t, b, h_in, mods, W, log_index=None, stream=None):
        """Enqueue block b of step t. h_in: dict text, tgt -> [B, n, C] bf16
        block inputs (the running state or the step's inputs); mods: dict
        stream -> six [B, C] fp32 vectors; W: dict stream -> weights."""
        li = (t % self.log_steps) if log_index is None else log_index
        mode = self.modes[li, b]
        n, C, F = self.n, self.C, self.F
        cur = self.q_tgt[t % 2, b]
        prev = self.q_tgt[(t + 1) % 2, b]
        ms = {r: mods[STREAM_OF[r]] for r in ROLES}
        Ws = {r: W[STREAM_OF[r]] for r in ROLES}
        hin = {"text": h_in["text"], "ref": self.hbar[b], "tgt": h_in["tgt"]}
        # 1. text and target rows: modulated LN, QKV (post-RoPE Q of the target kept for D)
        api.refadapt_ln_modulate(
            [{"h": hin[r], "x": self.x[r], "shift": ms[r]["shift_a"], "scale": ms[r]["scale_a"]}
             for r in ("text", "tgt")], C, self.ln_eps, stream=stream)
        q_out = {"text": self.qkv["text"][0], "tgt": cur}
        self._gemm("qkv", t, b, [
            {"a": self.x[r], "w": Ws[r]["w_qkv"], "bias": Ws[r]["b_qkv"], "q": q_out[r], "k": self.qkv[r][1],
             "v": self.qkv[r][2], "q_norm": Ws[r]["q_norm"], "k_norm": Ws[r]["k_norm"], "pos_offset": self.pos0[r]}
            for r in ("text", "tgt")], 3 * C, C, RA_EPI_QKV, rope=self.rope, H=self.H, d=self.d,
            norm_eps=self.norm_eps, err_word=self.err, stream=stream)
        # 2. Q change and the gate
        if t >= 1:
            api.refadapt_q_delta_gate(cur, prev, self.D[b], self.workspace, t, b, self.state, mode, self.theta,
                                      self.delta_max, self.mass[b], self.mass_row_count, eps=self.eps,
                                      forced_boundary=self.forced_boundary, gbar_out=self.gbar[li, b],
                                      m_out=self.M[li, b], cue=CUES[self.cue], stream=stream)
        else:
            api.refadapt_gate(t, b, self.state, mode, self.theta, self.delta_max, self.B, self.H,
                              mass_row_count=self.mass_row_count, forced_boundary=self.forced_boundary,
                              gbar_out=self.gbar[li, b], m_out=self.M[li, b], cue=CUES[self.cue], stream=stream)
        # 3. reference rows (gated on the mode): LN of H_b, QKV into the cache slot
        api.refadapt_ln_modulate(
            [{"h": hin["ref"], "x": self.x["ref"], "shift": ms["ref"]["shift_a"], "scale": ms["ref"]["scale_a"],
              "gated": True}], C, self.ln_eps, mode=mode, stream=stream)
        self._gemm("qkv_ref", t, b, [
            {"a": self.x["ref"], "w": Ws["ref"]["w_qkv"], "bias": Ws["ref"]["b_qkv"], "q": self.q_ref,
             "k": self.cache_k[b], "v": self.cache_v[b], "q_norm": Ws["ref"]["q_norm"],
             "k_norm": Ws["ref"]["k_norm"], "pos_offset": self.pos0["ref"], "gated": True}],
            3 * C, C, RA_EPI_QKV, mode=mode, rope=self.rope, H=self.H, d=self.d, norm_eps=self.norm_eps,
            err_word=self.err, stream=stream)
        # 4. joint attention (mass partials of the executed attention). The
        # reference K/V were written into the cache slot in place, so the fresh
        # reference rows are the slot itself: the kernel copies nothing and
        # stamps a_b = t for COMPUTE / FULL samples.
        if self.attn_hook is not None:
            self.attn_hook("pre", t, b)
        api.refadapt_joint_attn(
            (self.qkv["text"][0], self.q_ref, cur),
            (self.qkv["text"][1], self.cache_k[b], self.qkv["tgt"][1]),
            (self.qkv["text"][2], self.cache_v[b], self.qkv["tgt"][2]),
            tuple(self._heads(self.o[r]) for r in ROLES),
            self.mass[b], mode=mode, mass_rows=self.mass_rows, err_word=self.err,
            ref_fresh=(self.q_ref, self.cache_k[b], self.cache_v[b]), a_b=self.a_b[b], step=t, stream=stream)
        if self.attn_hook is not None:
            self.attn_hook("post", t, b)
        # 5. output projection with the gated residual (reference: H_b -> h1_ref)
        self._gemm("o_proj", t, b, [
            {"a": self.o[r], "w": Ws[r]["w_o"], "bias": Ws[r]["b_o"], "resid": hin[r], "gate": ms[r]["gate_a"],
             "out": self.h1[r], "gated": r == "ref"} for r in ROLES], C, C, RA_EPI_RESID, mode=mode,
            err_word=self.err, stream=stream)
        # 6. MLP branch
        api.refadapt_ln_modulate(
            [{"h": self.h1[r], "x": self.x[r], "shift": ms[r]["shift_m"], "scale": ms[r]["scale_m"],
              "gated": r == "ref"} for r in ROLES], C, self.ln_eps, mode=mode, stream=stream)
        self._gemm("mlp1", t, b, [
            {"a": self.x[r], "w": Ws[r]["w_1"], "bias": Ws[r]["b_1"], "out": self.u[r], "gated": r == "ref"}
            for r in ROLES], F, C, RA_EPI_GELU, mode=mode, err_word=self.err, stream=stream)
        out = {"text": self.h["text"], "ref": self.hbar[b + 1], "tgt": self.h["tgt"]}
        self._gemm("mlp2", t, b, [
            {"a": self.u[r], "w": Ws[r]["w_2"], "bias": Ws[r]["b_2"], "resid": self.h1[r], "gate": ms[r]["gate_m"],
             "out": out[r], "gated": r == "ref"} for r in ROLES], C, F, RA_EPI_RESID, mode=mode,
            err_word=self.err, stream=stream)

    def step(self, t, h_in, mods, weights, log_index=None, stream=None, after_block=None):
        """Enqueue one denoising step. h_in: dict role -> [B, n, C] bf16 stack
        inputs (the reference rows become H_0); mods(t, b), weights(b) give the
        block's AdaLN vectors and weights. The stack's output rows end in
        self.h['text'], self.h['tgt']; the reference hidden states in self.hbar."""
        self.hbar[0] = h_in["ref"]
        for b in range(self.n_blocks):
            src = {"text": h_in["text"], "tgt": h_in["tgt"]} if b == 0 else self.h
            self.block(t, b, src, mods(t, b), weights(b), log_index, stream)
            if after_block is not None:
                after_block(t, b)

    def check(self, stream=None):
        api.refadapt_check_error(self.err, stream)
