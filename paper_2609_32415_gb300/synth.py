"""Seeded synthetic inputs for the RefAdapt-DiT hot path.

This module is the one piece that both the CUDA path's tests/bench and the CPU
oracle's tests consume: it draws numbers and lays them out, and holds none of
the method's arithmetic (no attention, no drift metric, no gate).

Recipe (every workload):

* Each (step t, block b, role r, tensor z) with r in {text, ref, tgt} and
  z in {q, k, v} is a bf16 tensor [B, H, n_r, d].
* Step 0: X_0 = sigma0 * N(0, 1), sigma0 = 1/sqrt(d).
* Step t >= 1: X_t = bf16(X_{t-1} + delta_{r,b} * sigma0 * N(0, 1)), so the
  relative per-step change of a role is about delta_{r,b}.
* Every N(0, 1) draw comes from its own torch generator seeded by a hash of
  (seed, t, b, role, tensor), on the device the tensors are made on. The same
  bytes are handed to both sides of a parity check.
* Text rows drift like target rows (they are active-generation rows).
* Optional per-head bias beta_h (added by the kernel to target-row x
  reference-key logits) is drawn once from U(lo, hi).

Workloads (shapes follow the paper's image-edit and video settings; the
paper's datasets and checkpoints are not used): see ``WORKLOADS``.
"""
import math
from dataclasses import dataclass, field
from typing import Dict, List, Optional

import torch

ROLES = ("text", "ref", "tgt")
_ROLE_ID = {"text": 1, "ref": 2, "tgt": 3}
_TENSOR_ID = {"q": 1, "k": 2, "v": 3}


def _key(*parts) -> int:
    h = 0xCBF29CE484222325
    for p in parts:
        h ^= (int(p) & 0xFFFFFFFF)
        h = (h * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    return h & 0x7FFFFFFFFFFFFFFF


def _gen(device, *parts) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(_key(*parts))
    return g


@dataclass
class Workload:
    name: str
    B: int
    H: int
    d: int
    n_text: int
    n_ref: int
    n_tgt: int
    n_blocks: int
    n_steps: int
    ref_drift: List[float]            # per block
    tgt_drift: List[float]            # per block (text rows use the same)
    theta: float
    delta_max: int = 4
    eps: float = 1e-6
    mass_rows: int = 0
    bias: Optional[List[float]] = None  # per head, or None
    forced_boundary: int = -1
    seed: int = 0
    note: str = ""
    extra: Dict = field(default_factory=dict)

    @property
    def N(self) -> int:
        return self.n_text + self.n_ref + self.n_tgt

    @property
    def n(self) -> Dict[str, int]:
        return {"text": self.n_text, "ref": self.n_ref, "tgt": self.n_tgt}

    def offsets(self) -> Dict[str, int]:
        return {"text": 0, "ref": self.n_text, "tgt": self.n_text + self.n_ref}


def _expected_gbar(delta, t, m_est):
    # Closed-form expectation of the head-mean score under this recipe, used
    # only to place theta away from the realised scores: D_t ~ delta /
    # sqrt(1 + (t-1) delta^2) (the norm of X grows with every drift) and, with
    # near-uniform logits, M ~ the reference share of the keys.
    return delta / math.sqrt(1.0 + (t - 1) * delta * delta) * m_est


def _uniform_mass(n_ref, n_other, bias=None, H=1):
    if bias is None:
        return n_ref / float(n_ref + n_other)
    vals = [n_ref * math.exp(b) / (n_ref * math.exp(b) + n_other) for b in bias]
    return sum(vals) / len(vals)


def _profile_c2(n_blocks=60):
    # Reference drift decays linearly 0.05 -> 0.005 over blocks 0..44, then
    # rises linearly to 0.010 over the last 15 blocks.
    r = []
    for b in range(n_blocks):
        if b < 45:
            r.append(0.05 + (0.005 - 0.05) * b / 44.0)
        else:
            r.append(0.005 + (0.010 - 0.005) * (b - 44) / 15.0)
    return r


def _lognormal_profile(n_blocks, mu, sigma, seed):
    g = torch.Generator(device="cpu")
    g.manual_seed(_key(seed, 0xD81F7, n_blocks))
    z = torch.randn(n_blocks, generator=g, dtype=torch.float64)
    return [float(math.exp(mu + sigma * zz)) for zz in z.tolist()]


def _coupled_target(r, base):
    # Target-side drift follows the depth profile of the reference drift
    # (timing coupling), scaled to mean `base`.
    mean = sum(r) / len(r)
    return [base * x / mean for x in r]


def make_workload(name: str, **over) -> Workload:
    """Build one of the named workloads; keyword arguments override fields."""
    if name == "c1":
        wl = Workload("c1", B=1, H=8, d=64, n_text=32, n_ref=256, n_tgt=256, n_blocks=1,
                      n_steps=4, ref_drift=[0.02], tgt_drift=[0.2], theta=0.05,
                      note="single block, B=1, H=8, d=64, text 32 + ref 256 + tgt 256, 4 steps")
    elif name == "c2":
        r = _profile_c2(60)
        tgt = _coupled_target(r, 0.3)
        m_est = _uniform_mass(8192, 256 + 4096)
        # theta between the block-0 scores expected at steps 2 and 3.
        theta = 0.5 * (_expected_gbar(tgt[0], 2, m_est) + _expected_gbar(tgt[0], 3, m_est))
        wl = Workload("c2", B=1, H=24, d=128, n_text=256, n_ref=8192, n_tgt=4096, n_blocks=60,
                      n_steps=8, ref_drift=r, tgt_drift=tgt, theta=theta,
                      note="multi-reference image edit: 60 blocks, H=24, d=128, "
                           "text 256 + 2x4096 ref + 4096 tgt, 8 steps")
    elif name == "c3":
        seed = over.get("seed", 0)
        g = torch.Generator(device="cpu")
        g.manual_seed(_key(seed, 0xB1A5, 24))
        bias = (torch.rand(24, generator=g, dtype=torch.float64) * 3.0 - 3.0).tolist()
        m_est = _uniform_mass(16380, 512 + 16380, bias)
        theta = 0.5 * (_expected_gbar(0.4, 1, m_est) + _expected_gbar(0.4, 2, m_est))
        wl = Workload("c3", B=1, H=24, d=128, n_text=512, n_ref=16380, n_tgt=16380, n_blocks=40,
                      n_steps=4, ref_drift=[0.03] * 40, tgt_drift=[0.4] * 40, theta=theta,
                      bias=bias,
                      note="video: 40 blocks, H=24, d=128, text 512 + ref 21x30x26 + "
                           "tgt 21x30x26, 4 steps, per-head target->reference bias U(-3,0)")
    elif name == "c4":
        seed = over.get("seed", 0)
        r = _lognormal_profile(60, math.log(0.02), 0.5, seed)
        tgt = _coupled_target(r, 0.3)
        m_est = _uniform_mass(16384, 256 + 4096)
        gb = [_expected_gbar(x, 1, m_est) for x in tgt]
        head = max(gb[:51])
        later = sorted(x for x in gb[51:] if x > head)
        theta = 0.5 * (head + later[0]) if later else head * 1.05
        wl = Workload("c4", B=1, H=24, d=128, n_text=256, n_ref=16384, n_tgt=4096, n_blocks=60,
                      n_steps=8, ref_drift=r, tgt_drift=tgt, theta=theta,
                      note="heavy reference stream: 60 blocks, H=24, d=128, "
                           "text 256 + 4x4096 ref + 4096 tgt, 8 steps")
    elif name == "c5":
        total = int(over.pop("total", 8192))
        frac = float(over.pop("ref_frac", 0.5))
        reuse = float(over.pop("reuse_frac", 0.5))
        n_text = 256
        n_ref = int(round(frac * (total - n_text) / 128.0)) * 128
        n_tgt = total - n_text - n_ref
        nb = 8
        wl = Workload("c5", B=1, H=24, d=128, n_text=n_text, n_ref=n_ref, n_tgt=n_tgt,
                      n_blocks=nb, n_steps=8, ref_drift=[0.02] * nb, tgt_drift=[0.3] * nb,
                      theta=float("inf"), delta_max=8, forced_boundary=int(math.floor(reuse * nb)),
                      note="sweep point: total %d, ref %.0f%%, reuse %.0f%%"
                           % (total, 100 * frac, 100 * reuse))
    else:
        raise ValueError("unknown workload %r" % name)
    for k, v in over.items():
        if k == "seed" and name in ("c3", "c4"):
            wl.seed = v
            continue
        setattr(wl, k, v)
    return wl


def custom_workload(B, H, d, n_text, n_ref, n_tgt, n_blocks=1, n_steps=2, ref_drift=0.02,
                    tgt_drift=0.2, theta=0.05, delta_max=4, **kw) -> Workload:
    """A small workload for tests (drifts may be scalars or per-block lists)."""
    rd = ref_drift if isinstance(ref_drift, list) else [ref_drift] * n_blocks
    td = tgt_drift if isinstance(tgt_drift, list) else [tgt_drift] * n_blocks
    return Workload("custom", B=B, H=H, d=d, n_text=n_text, n_ref=n_ref, n_tgt=n_tgt,
                    n_blocks=n_blocks, n_steps=n_steps, ref_drift=rd, tgt_drift=td,
                    theta=theta, delta_max=delta_max, **kw)


class Trajectory:
    """Per-(step, block) joint Q/K/V tensors of a workload.

    ``get(t, b)`` returns a bf16 tensor X[3, B, H, N, d] (q, k, v stacked; the
    roles text, ref, tgt are consecutive slices along N, see
    ``Workload.offsets``). Steps are produced by the drift recurrence; access
    in increasing t per block is incremental, earlier t restarts from step 0.
    """

    def __init__(self, wl: Workload, device="cpu", base_scale: float = None):
        self.wl = wl
        self.device = torch.device(device)
        self.sigma0 = (1.0 / math.sqrt(wl.d)) if base_scale is None else float(base_scale)
        self._state = {}

    def _noise(self, t, b, role, z):
        wl = self.wl
        shape = (wl.B, wl.H, wl.n[role], wl.d)
        g = _gen(self.device, wl.seed, t, b, _ROLE_ID[role], _TENSOR_ID[z])
        return torch.randn(shape, generator=g, device=self.device, dtype=torch.float32)

    def _fresh(self, b):
        wl = self.wl
        X = torch.empty((3, wl.B, wl.H, wl.N, wl.d), dtype=torch.bfloat16, device=self.device)
        off = wl.offsets()
        for zi, z in enumerate("qkv"):
            for r in ROLES:
                if wl.n[r] == 0:
                    continue
                sl = X[zi, :, :, off[r]:off[r] + wl.n[r], :]
                sl.copy_((self._noise(0, b, r, z) * self.sigma0).to(torch.bfloat16))
        return X

    def _advance(self, X, t, b):
        wl = self.wl
        off = wl.offsets()
        Y = torch.empty_like(X)
        for zi, z in enumerate("qkv"):
            for r in ROLES:
                if wl.n[r] == 0:
                    continue
                delta = wl.ref_drift[b] if r == "ref" else wl.tgt_drift[b]
                src = X[zi, :, :, off[r]:off[r] + wl.n[r], :].float()
                src.add_(self._noise(t, b, r, z), alpha=delta * self.sigma0)
                Y[zi, :, :, off[r]:off[r] + wl.n[r], :].copy_(src.to(torch.bfloat16))
        return Y

    def get(self, t: int, b: int) -> torch.Tensor:
        st = self._state.get(b)
        if st is None or st[0] > t:
            st = (0, self._fresh(b))
        cur_t, X = st
        while cur_t < t:
            cur_t += 1
            X = self._advance(X, cur_t, b)
        self._state[b] = (cur_t, X)
        return X

    def forget(self):
        self._state.clear()

    def role_view(self, X: torch.Tensor, role: str) -> torch.Tensor:
        """The [3, B, H, n_role, d] slice of a joint tensor."""
        off = self.wl.offsets()[role]
        return X[:, :, :, off:off + self.wl.n[role], :]

    def bias_tensor(self):
        wl = self.wl
        if wl.bias is None:
            return None
        return torch.tensor(wl.bias, dtype=torch.float32).reshape(1, wl.H).repeat(wl.B, 1)


def sweep_points():
    """The c5 sweep grid: total tokens x reference fraction x reuse fraction."""
    pts = []
    for total in (8192, 16384, 32768, 65536):
        for frac in (0.5, 0.7, 0.9):
            for reuse in (0.0, 0.5, 0.9):
                pts.append((total, frac, reuse))
    return pts


# --------------------------------------------------------------------------- DiT block stack
# Inputs of the DiT-block stack around the attention (dual-stream MMDiT block:
# text rows use the text stream's weights, reference and target rows the image
# stream's). Random numbers only:
#
# * stack input rows [B, n_role, C], C = H d: text and reference rows
#   N(0, 1), the same at every step; target rows x_0 = N(0, 1),
#   x_t = bf16(x_{t-1} + tgt_drift * N(0, 1)) (the sampler's latent moving);
# * AdaLN modulation per (step, block, stream), six fp32 vectors [B, C]:
#   shift, scale ~ 0.1 N(0, 1), gate ~ 0.3 + 0.05 N(0, 1) drawn once per
#   (block, stream), plus mod_drift * N(0, 1) per step (the timestep
#   embedding moving);
# * weights per (block, stream): linear weights bf16 N(0, 1) / sqrt(fan_in),
#   biases fp32 0.02 N(0, 1), q/k norm weights fp32 1 + 0.1 N(0, 1).
MOD_NAMES = ("shift_a", "scale_a", "gate_a", "shift_m", "scale_m", "gate_m")
STREAMS = ("text", "image")


class DiTInputs:
    """Seeded inputs of a DiT-block stack over a workload's row partition."""

    def __init__(self, wl: Workload, device="cpu", mlp_ratio: int = 4, tgt_drift: float = 0.2,
                 mod_drift: float = 0.05, weight_cache: bool = True):
        self.wl = wl
        self.device = torch.device(device)
        self.C = wl.H * wl.d
        self.F = mlp_ratio * self.C
        self.tgt_drift = float(tgt_drift)
        self.mod_drift = float(mod_drift)
        self._x = None
        self._w = {} if weight_cache else None

    def _randn(self, shape, *parts):
        g = _gen(self.device, self.wl.seed, 0xD17, *parts)
        return torch.randn(shape, generator=g, device=self.device, dtype=torch.float32)

    def h_in(self, t: int) -> Dict[str, torch.Tensor]:
        """dict role -> bf16 [B, n_role, C] input rows of the stack at step t."""
        wl = self.wl
        out = {}
        for r in ("text", "ref"):
            out[r] = self._randn((wl.B, wl.n[r], self.C), 1, _ROLE_ID[r]).to(torch.bfloat16)
        if self._x is None or self._x[0] > t:
            self._x = (0, self._randn((wl.B, wl.n_tgt, self.C), 1, _ROLE_ID["tgt"]).to(torch.bfloat16))
        cur, x = self._x
        while cur < t:
            cur += 1
            x = (x.float() + self.tgt_drift * self._randn((wl.B, wl.n_tgt, self.C), 2, cur)).to(torch.bfloat16)
        self._x = (cur, x)
        out["tgt"] = x
        return out

    def mods(self, t: int, b: int) -> Dict[str, Dict[str, torch.Tensor]]:
        """dict stream -> dict name -> fp32 [B, C] modulation vectors."""
        wl = self.wl
        out = {}
        for si, st in enumerate(STREAMS):
            d = {}
            for j, name in enumerate(MOD_NAMES):
                base = self._randn((wl.B, self.C), 3, b, si, j)
                v = (0.3 + 0.05 * base) if name.startswith("gate") else 0.1 * base
                if t > 0 and self.mod_drift > 0:
                    v = v + self.mod_drift * self._randn((wl.B, self.C), 4, t, b, si, j)
                d[name] = v.contiguous()
            out[st] = d
        return out

    def weights(self, b: int) -> Dict[str, Dict[str, torch.Tensor]]:
        """dict stream -> w_qkv [3C, C], w_o [C, C], w_1 [F, C], w_2 [C, F]
        (bf16), b_qkv, b_o, b_1, b_2 (fp32), q_norm, k_norm [d] (fp32)."""
        if self._w is not None and b in self._w:
            return self._w[b]
        C, F, d = self.C, self.F, self.wl.d
        out = {}
        for si, st in enumerate(STREAMS):
            w = {}
            for j, (name, shape, fan) in enumerate((("w_qkv", (3 * C, C), C), ("w_o", (C, C), C),
                                                     ("w_1", (F, C), C), ("w_2", (C, F), F))):
                w[name] = (self._randn(shape, 5, b, si, j) / math.sqrt(fan)).to(torch.bfloat16)
            for j, (name, n) in enumerate((("b_qkv", 3 * C), ("b_o", C), ("b_1", F), ("b_2", C))):
                w[name] = 0.02 * self._randn((n,), 6, b, si, j)
            w["q_norm"] = 1.0 + 0.1 * self._randn((d,), 7, b, si, 0)
            w["k_norm"] = 1.0 + 0.1 * self._randn((d,), 7, b, si, 1)
            out[st] = w
        if self._w is not None:
            self._w[b] = out
        return out
