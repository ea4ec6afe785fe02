"""Thin Python binding of the C ABI (include/refadapt.h), same names.

Only argument marshalling happens here: torch tensors supply device memory and
streams; every step of the computation runs in librefadapt.so's kernels.
Tensors are [B, H, n, d] bf16 CUDA views with a contiguous last axis (any
other strides, 16-byte aligned).
"""
import ctypes

import torch

from . import _lib
from ._lib import RaAttnArgs, RaGateArgs, RaSeg, check

__all__ = ["seg", "refadapt_joint_attn", "refadapt_mass_partial_len", "refadapt_q_delta",
           "refadapt_q_delta_workspace_size", "refadapt_q_delta_noalloc", "refadapt_state_size", "refadapt_state_init",
           "refadapt_gate", "refadapt_ref_cache_update", "refadapt_set_wait_budget_ns",
           "refadapt_check_error", "refadapt_version", "refadapt_selftest_wait_timeout", "q_delta_workspace", "new_state",
           "alloc_mass_partial", "refadapt_rope_table", "rope_table", "refadapt_ln_modulate", "refadapt_gemm"]


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    if isinstance(stream, torch.cuda.Stream):
        return ctypes.c_void_p(stream.cuda_stream)
    return ctypes.c_void_p(int(stream))


def seg(t, n=None) -> RaSeg:
    """ra_seg of a [B, H, n, d] bf16 CUDA tensor (None -> empty/absent segment)."""
    if t is None:
        return RaSeg(None, 0, 0, 0, int(n or 0), 0)
    if t.dim() != 4 or t.dtype != torch.bfloat16 or not t.is_cuda or (t.shape[3] > 1 and t.stride(3) != 1):
        raise ValueError("expected a [B, H, n, d] bf16 CUDA tensor with contiguous last axis, got %s %s %s"
                         % (tuple(t.shape), t.dtype, t.device))
    ptr = t.data_ptr() if t.numel() > 0 else 0
    return RaSeg(ptr or None, t.stride(0), t.stride(1), t.stride(2), t.shape[2], 0)


def refadapt_mass_partial_len(n_text, n_tgt) -> int:
    return int(_lib.load().refadapt_mass_partial_len(int(n_text), int(n_tgt)))


def alloc_mass_partial(B, H, n_text, n_tgt, device="cuda"):
    return torch.zeros((B, H, refadapt_mass_partial_len(n_text, n_tgt)), dtype=torch.float32, device=device)


def refadapt_joint_attn(q, k, v, o, mass_partial, mode=None, softmax_scale=0.0, ref_logit_bias=None,
                        mass_rows=0, err_word=None, mass_row_stride=0, ref_fresh=None, a_b=None, step=0,
                        stream=None):
    """q, k, v, o: sequences (text, ref, tgt) of [B, H, n, d] tensors; q[1] / o[1] may be None.
    ref_fresh: optional (q, k, v) of this step's reference rows for the fused
    cache update (q may be None when q[1] is); a_b, step: the stamp it writes."""
    lib = _lib.load()
    B, H, _, d = k[2].shape
    a = RaAttnArgs()
    a.B, a.H, a.d, a.mass_rows = B, H, d, int(mass_rows)
    for r in range(3):
        n_q = q[r].shape[2] if q[r] is not None else k[r].shape[2]
        a.q[r] = seg(q[r], n_q)
        a.k[r] = seg(k[r])
        a.v[r] = seg(v[r])
        a.o[r] = seg(o[r], n_q)
    a.softmax_scale = float(softmax_scale)
    a.mass_row_stride = int(mass_row_stride)
    a.ref_logit_bias = _ptr(ref_logit_bias)
    a.mode = _ptr(mode)
    a.mass_partial = _ptr(mass_partial)
    a.err_word = _ptr(err_word)
    if ref_fresh is not None:
        fq, fk, fv = ref_fresh
        a.ref_fresh_q = seg(fq)
        a.ref_fresh_k = seg(fk)
        a.ref_fresh_v = seg(fv)
        a.a_b = _ptr(a_b)
        a.step = int(step)
    elif a_b is not None:
        raise ValueError("refadapt_joint_attn: a_b is written only with ref_fresh")
    return check("refadapt_joint_attn", lib.refadapt_joint_attn(ctypes.byref(a), _stream(stream)))


def refadapt_q_delta_workspace_size(B, H) -> int:
    return int(_lib.load().refadapt_q_delta_workspace_size(int(B), int(H)))


def q_delta_workspace(B, H, device="cuda"):
    """A zero-filled workspace for refadapt_q_delta (reusable across calls)."""
    return torch.zeros(refadapt_q_delta_workspace_size(B, H), dtype=torch.uint8, device=device)


def refadapt_q_delta(q_cur, q_prev, d_out, workspace, eps=1e-6, stream=None):
    lib = _lib.load()
    B, H, _, d = q_cur.shape
    sc, sp = seg(q_cur), seg(q_prev)
    return check("refadapt_q_delta", lib.refadapt_q_delta(
        ctypes.byref(sc), ctypes.byref(sp), B, H, d, float(eps), _ptr(d_out), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def refadapt_q_delta_noalloc(q_cur, q_prev, d_out, eps=1e-6, stream=None):
    """refadapt_q_delta without a workspace (static scratch inside the library;
    B * H <= RA_Q_DELTA_NOALLOC_MAX_BH; calls must not overlap on the GPU)."""
    lib = _lib.load()
    B, H, _, d = q_cur.shape
    sc, sp = seg(q_cur), seg(q_prev)
    return check("refadapt_q_delta_noalloc", lib.refadapt_q_delta_noalloc(
        ctypes.byref(sc), ctypes.byref(sp), B, H, d, float(eps), _ptr(d_out), _stream(stream)))


def refadapt_state_size(B) -> int:
    return int(_lib.load().refadapt_state_size(int(B)))


def refadapt_state_init(state, B, stream=None):
    return check("refadapt_state_init", _lib.load().refadapt_state_init(_ptr(state), int(B), _stream(stream)))


def new_state(B, device="cuda", stream=None):
    st = torch.empty(refadapt_state_size(B), dtype=torch.uint8, device=device)
    refadapt_state_init(st, B, stream)
    return st


def _gate_args(t, b, state, mode_out, theta, delta_max, B, H, q_delta, mass_partial_prev, mass_row_count,
               forced_boundary, gbar_out, m_out, cue):
    a = RaGateArgs()
    a.theta = float(theta)
    a.t, a.b, a.B, a.H = int(t), int(b), int(B), int(H)
    a.delta_max = int(delta_max)
    a.forced_boundary = int(forced_boundary)
    a.mass_partial_len = int(mass_partial_prev.shape[-1]) if mass_partial_prev is not None else 0
    a.mass_row_count = int(mass_row_count)
    a.cue = int(cue)
    a.q_delta = _ptr(q_delta)
    a.mass_partial_prev = _ptr(mass_partial_prev)
    a.state = _ptr(state)
    a.mode_out = _ptr(mode_out)
    a.gbar_out = _ptr(gbar_out)
    a.m_out = _ptr(m_out)
    return a


def refadapt_gate(t, b, state, mode_out, theta, delta_max, B, H, q_delta=None, mass_partial_prev=None,
                  mass_row_count=0, forced_boundary=-1, gbar_out=None, m_out=None, cue=0, stream=None):
    a = _gate_args(t, b, state, mode_out, theta, delta_max, B, H, q_delta, mass_partial_prev, mass_row_count,
                   forced_boundary, gbar_out, m_out, cue)
    return check("refadapt_gate", _lib.load().refadapt_gate(ctypes.byref(a), _stream(stream)))


def refadapt_q_delta_gate(q_cur, q_prev, d_out, workspace, t, b, state, mode_out, theta, delta_max,
                          mass_partial_prev, mass_row_count, eps=1e-6, forced_boundary=-1, gbar_out=None,
                          m_out=None, cue=0, stream=None):
    """refadapt_q_delta then refadapt_gate on its D (t >= 1), in one launch
    when the Q change takes its cluster path."""
    lib = _lib.load()
    B, H, _, d = q_cur.shape
    sc, sp = seg(q_cur), seg(q_prev)
    a = _gate_args(t, b, state, mode_out, theta, delta_max, B, H, d_out, mass_partial_prev, mass_row_count,
                   forced_boundary, gbar_out, m_out, cue)
    return check("refadapt_q_delta_gate", lib.refadapt_q_delta_gate(
        ctypes.byref(sc), ctypes.byref(sp), B, H, d, float(eps), _ptr(d_out), _ptr(workspace),
        workspace.numel() * workspace.element_size(), ctypes.byref(a), _stream(stream)))


def refadapt_ref_cache_update(k_src, v_src, k_cache, v_cache, mode, t, a_b=None, x_src=None, x_cache=None,
                              stream=None):
    lib = _lib.load()
    B, H, _, d = k_src.shape
    ks, vs, kc, vc = seg(k_src), seg(v_src), seg(k_cache), seg(v_cache)
    if x_src is not None:
        xs, xc = seg(x_src), seg(x_cache)
        xp, xcp = ctypes.byref(xs), ctypes.byref(xc)
        x_heads, x_width = x_src.shape[1], x_src.shape[3]
    else:
        xp = xcp = None
        x_heads = x_width = 0
    return check("refadapt_ref_cache_update", lib.refadapt_ref_cache_update(
        ctypes.byref(ks), ctypes.byref(vs), ctypes.byref(kc), ctypes.byref(vc), B, H, d, xp, xcp,
        x_heads, x_width, _ptr(mode), int(t), _ptr(a_b), _stream(stream)))


def refadapt_set_wait_budget_ns(ns):
    _lib.load().refadapt_set_wait_budget_ns(int(ns))


def refadapt_check_error(err_word, stream=None):
    return check("refadapt_check_error", _lib.load().refadapt_check_error(_ptr(err_word), _stream(stream)))


def refadapt_selftest_wait_timeout(err_word, budget_ns, stream=None):
    return check("refadapt_selftest_wait_timeout",
                 _lib.load().refadapt_selftest_wait_timeout(_ptr(err_word), int(budget_ns), _stream(stream)))


def refadapt_version() -> int:
    return int(_lib.load().refadapt_version())


# --------------------------------------------------------------------------- DiT block around the attention
def _rows(t, what):
    """(ptr, stride_s, stride_r, rows) of a [B, rows, F] CUDA tensor with contiguous last axis."""
    if t.dim() != 3 or not t.is_cuda or (t.shape[2] > 1 and t.stride(2) != 1):
        raise ValueError("%s: expected a [B, rows, F] CUDA tensor with contiguous last axis, got %s"
                         % (what, tuple(t.shape)))
    return (t.data_ptr() if t.numel() > 0 else None), t.stride(0), t.stride(1), t.shape[1]


def refadapt_rope_table(table, n_pos, d, base=10000.0, stream=None):
    return check("refadapt_rope_table", _lib.load().refadapt_rope_table(
        _ptr(table), int(n_pos), int(d), float(base), _stream(stream)))


def rope_table(n_pos, d, base=10000.0, device="cuda", stream=None):
    """[n_pos, d/2, 2] fp32 (cos, sin) table built by refadapt_rope_table."""
    t = torch.empty((int(n_pos), int(d) // 2, 2), dtype=torch.float32, device=device)
    refadapt_rope_table(t, n_pos, d, base, stream)
    return t


def refadapt_ln_modulate(segs, C, eps=1e-6, mode=None, stream=None):
    """segs: up to three dicts with h, x ([B, rows, C] bf16), shift, scale
    ([B, C] fp32) and optional gated (bool)."""
    a = _lib.RaLnmodArgs()
    B = None
    for i, sd in enumerate(segs):
        hp, hs, hr, rows = _rows(sd["h"], "h")
        xp, xs, xr, xrows = _rows(sd["x"], "x")
        if xrows != rows:
            raise ValueError("h and x rows differ")
        B = sd["h"].shape[0]
        s = a.seg[i]
        s.h, s.h_stride_s, s.h_stride_r = hp, hs, hr
        s.x, s.x_stride_s, s.x_stride_r = xp, xs, xr
        s.shift, s.scale = _ptr(sd["shift"]), _ptr(sd["scale"])
        s.mod_stride_s = sd["shift"].stride(0)
        if sd["scale"].stride(0) != s.mod_stride_s:
            raise ValueError("shift and scale must share a row stride")
        s.rows, s.gated = int(rows), int(bool(sd.get("gated", False)))
    a.B, a.C, a.n_seg = int(B), int(C), len(segs)
    a.eps = float(eps)
    a.mode = _ptr(mode)
    return check("refadapt_ln_modulate", _lib.load().refadapt_ln_modulate(ctypes.byref(a), _stream(stream)))


def refadapt_gemm(segs, N, K, epilogue, mode=None, rope=None, H=0, d=0, norm_eps=1e-6, err_word=None,
                  tile_mode=0, stream=None):
    """segs: up to three dicts with a ([B, rows, K] bf16), w ([N, K] bf16),
    optional bias ([N] fp32), gated; plus per epilogue out ([B, rows, N]),
    resid and gate ([B, N] fp32) for RESID, or q, k, v ([B, H, rows, d]),
    q_norm, k_norm ([d] fp32) and pos_offset for QKV."""
    a = _lib.RaGemmArgs()
    B = None
    for i, sd in enumerate(segs):
        ap, ass, asr, rows = _rows(sd["a"], "a")
        B = sd["a"].shape[0]
        s = a.seg[i]
        s.a, s.a_stride_s, s.a_stride_r, s.rows = ap, ass, asr, int(rows)
        s.gated = int(bool(sd.get("gated", False)))
        w = sd["w"]
        if tuple(w.shape) != (int(N), int(K)) or not w.is_contiguous() or w.dtype != torch.bfloat16:
            raise ValueError("w: expected a contiguous [N, K] = [%d, %d] bf16 tensor, got %s"
                             % (N, K, tuple(w.shape)))
        s.w = _ptr(w)
        s.bias = _ptr(sd.get("bias"))
        if sd.get("out") is not None:
            s.out, s.out_stride_s, s.out_stride_r, _ = _rows(sd["out"], "out")
        if sd.get("resid") is not None:
            s.resid, s.resid_stride_s, s.resid_stride_r, _ = _rows(sd["resid"], "resid")
        if sd.get("gate") is not None:
            s.gate, s.gate_stride_s = _ptr(sd["gate"]), sd["gate"].stride(0)
        if epilogue == _lib.RA_EPI_QKV:
            s.q_out, s.k_out, s.v_out = seg(sd["q"]), seg(sd["k"]), seg(sd["v"])
            s.q_norm, s.k_norm = _ptr(sd["q_norm"]), _ptr(sd["k_norm"])
            s.pos_offset = int(sd.get("pos_offset", 0))
    a.B, a.N, a.K, a.epilogue = int(B), int(N), int(K), int(epilogue)
    a.H, a.d, a.n_seg = int(H), int(d), len(segs)
    a.rope_len = int(rope.shape[0]) if rope is not None else 0
    a.mode = _ptr(mode)
    a.rope = _ptr(rope)
    a.norm_eps = float(norm_eps)
    a.tile_mode = int(tile_mode)
    a.err_word = _ptr(err_word)
    return check("refadapt_gemm", _lib.load().refadapt_gemm(ctypes.byref(a), _stream(stream)))
