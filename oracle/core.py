"""RefAdapt-DiT oracle: a plain, slow, fp64 restatement of the paper's hot path.

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's
cpu_baseline / reference legs may import this module. It shares no code with
the CUDA library or its Python binding and imports neither.

Each function names the passage of the paper it restates:

* ``bf16_to_f64``          exact widening of bf16 bit patterns (no rounding).
* ``joint_attention``      Sec. 3.3, Attn(Q,K,V) = Softmax(QK^T/sqrt(d_h))V, and
                           the inner sum of Eq. 4 (C part in attn_oracle.c).
* ``exposure``             Eq. 4: mean over target query rows of the softmax
                           mass on reference keys.
* ``head_mean_exposure``   Eq. 5: the mean of Eq. 4 over heads.
* ``adjacent_ref_mass_change``  Eq. 6: mean absolute change of Eq. 5 between
                           neighbouring steps of a block, in percentage points.
* ``q_change``             Eq. 1 applied to each post-RoPE target-query head
                           (Sec. 4, "Runtime cues observable under reuse").
* ``Gate``                 Eq. 12 (per-head product), the head mean of App. A.2,
                           Eq. 13 (first crossing) and the bounded-age refresh
                           of Sec. 4 / Algorithm 1.
* ``block_attention``      one block of Algorithm 1 for one sample: which query
                           rows run and which reference K/V they see.
* ``closed_loop``          Algorithm 1 end to end, with the block cache state of
                           Eq. 11.
* ``attention_flops``      App. A.4 compute accounting.

Readings of points the paper leaves open:
eps of Eq. 1 is a parameter (default 1e-6); all target rows are used unless
``sample_stride`` k > 1 takes D and M over the rows 0, k, 2k, ...; mass rows
default to the target-latent rows (``mass_rows=0``), with
``mass_rows=1`` for text + target; a score equal to theta reactivates; the
reference query rows at a boundary block are the ones cached at the block's
last materialisation (the stand-in for restoring the cached hidden state).
"""
import ctypes
import math
import os

import numpy as np

from . import build as _build

REUSE, BOUNDARY, COMPUTE, FULL = 0, 1, 2, 3
ROLES = ("text", "ref", "tgt")

_lib = None


def _load():
    global _lib
    if _lib is None:
        path = _build.build()
        lib = ctypes.CDLL(path)
        f = lib.oracle_joint_attn_f64
        f.restype = ctypes.c_int
        f.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                      ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_double,
                      ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64,
                      ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int]
        _lib = lib
    return _lib


def default_threads() -> int:
    return max(1, os.cpu_count() or 1)


def bf16_to_f64(bits) -> np.ndarray:
    """Widen bf16 bit patterns (uint16) to float64 exactly.

    A bf16 value is the upper half of an IEEE binary32 word, so placing the 16
    bits in the high half of a uint32 gives the same real number as a float32,
    which float64 represents exactly.
    """
    b = np.ascontiguousarray(np.asarray(bits, dtype=np.uint16))
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def joint_attention(q, k, v, scale, bias=None, row_biased=None, ref_range=(0, 0),
                    want_o=True, nthreads=None):
    """Softmax(scale * Q K^T [+ bias]) V per head, and each row's reference mass.

    q: [H, nq, d], k, v: [H, nk, d] (float64). ``bias`` [H] is added to the
    logits of rows flagged in ``row_biased`` [nq] against keys in
    ``ref_range`` = [r0, r1). Returns (o [H, nq, d] or None, mass [H, nq]) where
    mass[h, i] = sum over reference keys of the row's softmax probabilities
    (the inner sum of Eq. 4).
    """
    q = np.ascontiguousarray(q, dtype=np.float64)
    k = np.ascontiguousarray(k, dtype=np.float64)
    v = np.ascontiguousarray(v, dtype=np.float64)
    H, nq, d = q.shape
    nk = k.shape[1]
    assert k.shape == (H, nk, d) and v.shape == (H, nk, d)
    r0, r1 = int(ref_range[0]), int(ref_range[1])
    o = np.zeros((H, nq, d), dtype=np.float64) if want_o else None
    mass = np.zeros((H, nq), dtype=np.float64)
    if nq == 0 or H == 0:
        return o, mass
    bias_arr = None
    rb = None
    if bias is not None:
        bias_arr = np.ascontiguousarray(np.asarray(bias, dtype=np.float64).reshape(H))
        rb = np.ascontiguousarray(np.asarray(row_biased, dtype=np.uint8).reshape(nq))
    rc = _load().oracle_joint_attn_f64(
        H, nq, nk, d, q.ctypes.data, k.ctypes.data, v.ctypes.data, float(scale),
        bias_arr.ctypes.data if bias_arr is not None else None,
        rb.ctypes.data if rb is not None else None, r0, r1,
        o.ctypes.data if o is not None else None, mass.ctypes.data,
        int(nthreads or default_threads()))
    if rc != 0:
        raise RuntimeError("oracle_joint_attn_f64 failed")
    return o, mass


def q_change(q_cur, q_prev, eps=1e-6) -> np.ndarray:
    """Eq. 1, D = ||X_t - X_{t-1}||_F / (||X_{t-1}||_F + eps), per leading index.

    q_cur, q_prev: [..., n, d] float64 (the token scope is the last two axes).
    Returns one value per leading index (per head, or per sample and head).
    """
    qc = np.asarray(q_cur, dtype=np.float64)
    qp = np.asarray(q_prev, dtype=np.float64)
    num = np.sqrt(np.sum((qc - qp) ** 2, axis=(-2, -1)))
    den = np.sqrt(np.sum(qp ** 2, axis=(-2, -1))) + eps
    return num / den


def endpoint_drift(z_t, z_a, eps=1e-6) -> np.ndarray:
    """Eq. 7, D_{t|a}(Z) = ||Z_t - Z_a||_F / (||Z_a||_F + eps): anchor-to-current
    change of a reference tensor (per leading index)."""
    return q_change(z_t, z_a, eps)


def local_impact(o_stale, o_fresh, eps=1e-6) -> np.ndarray:
    """Eq. 10, I = ||O^staleKV - O^fresh||_F / (||O^fresh||_F + eps) over the
    target query rows (per leading index)."""
    return q_change(o_stale, o_fresh, eps)


def exposure(row_mass_tgt, row_mass_text=None) -> np.ndarray:
    """Eq. 4: mean over the chosen query rows of their reference mass, per head.

    row_mass_tgt [H, n_tgt]; with ``row_mass_text`` [H, n_text] the text rows
    are counted too (the literal reading of Y as every non-reference row).
    """
    parts = [np.asarray(row_mass_tgt, dtype=np.float64)]
    if row_mass_text is not None:
        parts.append(np.asarray(row_mass_text, dtype=np.float64))
    allm = np.concatenate(parts, axis=1)
    return allm.sum(axis=1) / allm.shape[1]


def head_mean_exposure(M) -> np.ndarray:
    """Eq. 5: (1/H) sum_h M_{t,b,h}; M [..., H] -> [...]."""
    M = np.asarray(M, dtype=np.float64)
    total = np.zeros(M.shape[:-1])
    for h in range(M.shape[-1]):
        total = total + M[..., h]
    return total / M.shape[-1]


def adjacent_ref_mass_change(Mbar) -> np.ndarray:
    """Eq. 6: (100 / (T - 1)) sum_{t=2}^{T} |Mbar_t - Mbar_{t-1}|, in
    percentage points. Mbar [T, ...] holds the head-mean exposure of steps
    1..T (first axis) of a block; T >= 2."""
    Mbar = np.asarray(Mbar, dtype=np.float64)
    T = Mbar.shape[0]
    if T < 2:
        raise ValueError("Eq. 6 needs at least two steps")
    total = np.zeros(Mbar.shape[1:])
    for t in range(1, T):
        total = total + np.abs(Mbar[t] - Mbar[t - 1])
    return 100.0 * total / (T - 1)


def attention_flops(n_q, n_k, H, d) -> int:
    """App. A.4: score and value products are 2*n_q*n_k*d multiply-adds each per head."""
    return 4 * int(d) * int(H) * int(n_q) * int(n_k)


def reuse_score_fraction(n_ref, n_y) -> float:
    """App. A.4: score work on a cached step over a full step,
    N_Y (N_R + N_Y) / (N_R + N_Y)^2."""
    return n_y * (n_ref + n_y) / float((n_ref + n_y) ** 2)


class Gate:
    """The controller of Algorithm 1 for one trajectory, per sample.

    Step 0 materialises every block (FULL). At the start of a later step t the
    bounded-age test t - a_full >= delta_max forces a full refresh from block 0
    (and sets a_full = t); otherwise the reactivated latch is cleared. Then,
    block by block: while not reactivated, the per-head score
    g_h = D_h * M_{t-1,h} (Eq. 12) is averaged over heads (App. A.2) and compared
    with theta (Eq. 13): below theta the block reuses, the first block at or
    above theta is the boundary and sets the latch; every later block computes.
    ``forced_boundary`` >= 0 replaces the comparison by "block index >= it".
    ``cue`` selects the per-head trigger of the controller ablation (Sec. 5.3,
    Tab. 4): "product" g_h = D_h M_h (the method), "change" g_h = D_h,
    "exposure" g_h = M_h. Only the trigger changes; the executor, stopping
    rule, bounded-age fallback and threshold stay.
    """

    CUES = ("product", "change", "exposure")

    def __init__(self, n_samples, theta, delta_max, forced_boundary=-1, cue="product"):
        if cue not in self.CUES:
            raise ValueError("unknown cue %r" % (cue,))
        self.cue = cue
        self.B = int(n_samples)
        self.theta = float(theta)
        self.delta_max = int(delta_max)
        self.forced_boundary = int(forced_boundary)
        self.a_full = 0
        self.full_step = True
        self.reactivated = [False] * self.B
        self.boundary = [-1] * self.B

    def begin_step(self, t):
        if t == 0:
            self.full_step = True
            self.a_full = 0
        elif t - self.a_full >= self.delta_max:
            self.full_step = True
            self.a_full = t
        else:
            self.full_step = False
        self.reactivated = [False] * self.B
        self.boundary = [-1] * self.B

    def decide(self, t, b, D=None, M_prev=None, tie=None, tie_band=1e-4):
        """Modes and head-mean scores for block b of step t.

        D, M_prev: [B, H]. ``tie(t, b, s)`` (optional) returns the crossing
        decision to adopt when |gbar - theta| < tie_band.
        """
        modes, gbars = [], []
        for s in range(self.B):
            if t >= 1 and D is not None and M_prev is not None:
                if self.cue == "change":
                    g = [float(D[s][h]) for h in range(len(D[s]))]
                elif self.cue == "exposure":
                    g = [float(M_prev[s][h]) for h in range(len(D[s]))]
                else:
                    g = [float(D[s][h]) * float(M_prev[s][h]) for h in range(len(D[s]))]
                gbar = sum(g) / len(g)
            else:
                gbar = float("nan")
            gbars.append(gbar)
            if self.full_step:
                modes.append(FULL)
            elif self.reactivated[s]:
                modes.append(COMPUTE)
            else:
                if self.forced_boundary >= 0:
                    cross = b >= self.forced_boundary
                else:
                    cross = gbar >= self.theta
                    if tie is not None and abs(gbar - self.theta) < tie_band:
                        cross = bool(tie(t, b, s))
                if cross:
                    modes.append(BOUNDARY)
                    self.reactivated[s] = True
                    self.boundary[s] = b
                else:
                    modes.append(REUSE)
        return modes, gbars


def block_attention(q, k, v, mode, scale, bias=None, mass_rows=0, o_rows=None,
                    want_o=True, nthreads=None, sample_stride=1):
    """One block's executed joint attention for one sample (Algorithm 1 body).

    q, k, v: dict role -> float64 [H, n_role, d] for roles text, ref, tgt.
    k['ref'], v['ref'] are the reference keys/values this block sees (the cache
    slot, or the fresh ones after a refresh); q['ref'] is the reference query
    the executor supplies. Query rows: text and target when ``mode`` is REUSE
    (reference rows skipped), every row otherwise. Keys: [text; ref; tgt].
    ``bias`` [H] is added to target-row x reference-key logits.
    ``o_rows``: optional dict role -> row indices at which to return O (all
    executed rows when None). Returns dict with O[role] (None when the role's
    rows are not executed), row_mass[role], and M [H] (Eq. 4) over the mass
    rows 0, k, 2k, ... of each counted role (k = ``sample_stride``, the
    "sampled target-query rows"; 1 = every row).
    """
    H = q["tgt"].shape[0]
    n = {r: q[r].shape[1] if r != "ref" else k["ref"].shape[1] for r in ROLES}
    keys = np.concatenate([k["text"], k["ref"], k["tgt"]], axis=1)
    vals = np.concatenate([v["text"], v["ref"], v["tgt"]], axis=1)
    r0, r1 = n["text"], n["text"] + n["ref"]
    run_roles = ("text", "tgt") if mode == REUSE else ROLES
    out = {"O": {r: None for r in ROLES}, "row_mass": {r: None for r in ROLES}}
    for r in run_roles:
        qr = q[r]
        if qr.shape[1] == 0:
            out["O"][r] = np.zeros((H, 0, qr.shape[2]))
            out["row_mass"][r] = np.zeros((H, 0))
            continue
        biased = np.full(qr.shape[1], 1 if r == "tgt" else 0, dtype=np.uint8)
        if o_rows is None or o_rows.get(r) is None:
            o, m = joint_attention(qr, keys, vals, scale, bias, biased if bias is not None else None,
                                   (r0, r1), want_o=want_o, nthreads=nthreads)
            out["O"][r] = o
            out["row_mass"][r] = m
        else:
            need_mass = (r == "tgt") or (r == "text" and mass_rows == 1)
            if need_mass:
                _, m = joint_attention(qr, keys, vals, scale, bias,
                                       biased if bias is not None else None, (r0, r1),
                                       want_o=False, nthreads=nthreads)
                out["row_mass"][r] = m
            idx = np.asarray(o_rows[r], dtype=np.int64)
            sub = qr[:, idx, :]
            o, _ = joint_attention(sub, keys, vals, scale, bias,
                                   biased[idx] if bias is not None else None, (r0, r1),
                                   want_o=want_o, nthreads=nthreads)
            out["O"][r] = o
    kk = max(1, int(sample_stride))
    out["M"] = exposure(out["row_mass"]["tgt"][:, ::kk],
                        out["row_mass"]["text"][:, ::kk] if mass_rows == 1 else None)
    return out


def closed_loop(get_inputs, n_steps, n_blocks, B, *, theta, delta_max, eps=1e-6,
                scale=None, bias=None, mass_rows=0, forced_boundary=-1, tie=None,
                o_rows=None, want_o=True, nthreads=None, cue="product", diagnostics=False,
                diag_row_stride=1, sample_stride=1):
    """Algorithm 1 over ``n_steps`` denoising steps and ``n_blocks`` blocks.

    ``get_inputs(t, b)`` returns dict role -> (q, k, v), each a uint16 array of
    bf16 bits shaped [B, H, n_role, d]: the fresh post-RoPE Q, K, V of block b
    at step t. ``bias`` [H] or None. ``o_rows(t, b, s)`` may return the
    per-role row indices at which to evaluate O.

    Block cache state (Eq. 11): per block and sample the cached reference K, V,
    the cached reference query (the stand-in for the cached hidden state) and
    the materialisation step a_b. REUSE: target and text rows attend to the
    cache, reference rows are skipped, the cache is untouched. BOUNDARY: every
    row runs against the cached reference K/V with the cached reference query;
    the cache is untouched. COMPUTE / FULL: the cache takes the fresh reference
    K/V/Q and a_b = t, then every row runs. D and M are recorded at every block
    for the next step.

    ``cue``: "product" (the method), "change", "exposure" (Tab. 4 variants),
    or "anchor_product": g_h = c^anchor_h M_h with c^anchor the change of the
    target query to its value at the block's last materialisation a_b
    (App. A.2), i.e. Eq. 1 against the anchor instead of the previous step.

    ``diagnostics``: also record, per block, the staleness diagnostics of
    Sec. 3.3 and App. A.2 on the target rows 0, k, 2k, ... (k =
    ``diag_row_stride``): E_K, E_V (Eq. 7: cache slot vs this step's fresh
    reference K, V), E_KV = (E_K + E_V) / 2, O_fresh (Eq. 8: target rows with
    fresh reference K/V), I_KV (Eq. 10: executed output vs O_fresh) and
    M_fresh (the exposure of Eq. 4 with fresh reference keys; the executed M
    is the same-step cached exposure when the block reuses).

    ``sample_stride`` k > 1: D (Eq. 1) and M (Eq. 4) over the sampled target
    query rows 0, k, 2k, ... only (Algorithm 1 stores sampled target queries
    and masses); 1 = every row.

    Returns records[t][b] = dict(mode [B], gbar [B], D [B,H], M [B,H],
    O [B] of dict role -> array or None, a_b [B]) (+ the diagnostics).
    """
    gate = Gate(B, theta, delta_max, forced_boundary, "product" if cue == "anchor_product" else cue)
    anchor_q = [None] * n_blocks                       # target Q at the last materialisation
    cache = [[None] * B for _ in range(n_blocks)]      # dict(k, v, q) per block/sample
    a_b = [[-1] * B for _ in range(n_blocks)]
    prev_q = [None] * n_blocks                         # target Q, float64 [B,H,n,d]
    prev_M = [None] * n_blocks                         # [B,H]
    records = []
    for t in range(n_steps):
        gate.begin_step(t)
        step_rec = []
        for b in range(n_blocks):
            raw = get_inputs(t, b)
            f = {r: tuple(bf16_to_f64(x) for x in raw[r]) for r in ROLES}
            q_tgt = f["tgt"][0]
            H, d = q_tgt.shape[1], q_tgt.shape[3]
            sc = (1.0 / math.sqrt(d)) if scale is None else float(scale)
            ks = max(1, int(sample_stride))
            if cue == "anchor_product":
                D = q_change(q_tgt[:, :, ::ks], anchor_q[b][:, :, ::ks], eps) \
                    if (t >= 1 and anchor_q[b] is not None) else None
            else:
                D = q_change(q_tgt[:, :, ::ks], prev_q[b][:, :, ::ks], eps) \
                    if (t >= 1 and prev_q[b] is not None) else None
            modes, gbars = gate.decide(t, b, D, prev_M[b], tie=tie)
            if anchor_q[b] is None:
                anchor_q[b] = np.array(q_tgt)
            for s in range(B):
                if modes[s] in (COMPUTE, FULL):
                    anchor_q[b][s] = q_tgt[s]
            M = np.zeros((B, H))
            O = []
            diag = {}
            for s in range(B):
                mode = modes[s]
                if mode in (COMPUTE, FULL):
                    cache[b][s] = {"k": f["ref"][1][s], "v": f["ref"][2][s], "q": f["ref"][0][s]}
                    a_b[b][s] = t
                if mode == REUSE or mode == BOUNDARY:
                    kref, vref, qref = cache[b][s]["k"], cache[b][s]["v"], cache[b][s]["q"]
                else:
                    kref, vref, qref = f["ref"][1][s], f["ref"][2][s], f["ref"][0][s]
                qd = {"text": f["text"][0][s], "ref": qref, "tgt": f["tgt"][0][s]}
                kd = {"text": f["text"][1][s], "ref": kref, "tgt": f["tgt"][1][s]}
                vd = {"text": f["text"][2][s], "ref": vref, "tgt": f["tgt"][2][s]}
                rows = o_rows(t, b, s) if o_rows is not None else None
                res = block_attention(qd, kd, vd, mode, sc,
                                      None if bias is None else np.asarray(bias),
                                      mass_rows, rows, want_o, nthreads, sample_stride)
                M[s] = res["M"]
                O.append(res["O"])
                if diagnostics:
                    k = int(diag_row_stride)
                    qf = {"text": f["text"][0][s], "ref": f["ref"][0][s], "tgt": f["tgt"][0][s][:, ::k]}
                    kf = {"text": f["text"][1][s], "ref": f["ref"][1][s], "tgt": f["tgt"][1][s]}
                    vf = {"text": f["text"][2][s], "ref": f["ref"][2][s], "tgt": f["tgt"][2][s]}
                    fresh = block_attention(qf, kf, vf, REUSE, sc, None if bias is None else np.asarray(bias),
                                            0, None, True, nthreads)
                    # target rows of the executed pass, same sampling
                    qs = {"text": f["text"][0][s], "ref": qref, "tgt": f["tgt"][0][s][:, ::k]}
                    stale = block_attention(qs, kd, vd, REUSE, sc, None if bias is None else np.asarray(bias),
                                            0, None, True, nthreads)
                    diag.setdefault("E_K", np.zeros((B, H)))[s] = endpoint_drift(f["ref"][1][s], kref, eps)
                    diag.setdefault("E_V", np.zeros((B, H)))[s] = endpoint_drift(f["ref"][2][s], vref, eps)
                    diag.setdefault("I_KV", np.zeros((B, H)))[s] = local_impact(stale["O"]["tgt"],
                                                                               fresh["O"]["tgt"], eps)
                    diag.setdefault("M_fresh", np.zeros((B, H)))[s] = fresh["M"]
                    diag.setdefault("M_cached", np.zeros((B, H)))[s] = stale["M"]
            rec = {"mode": modes, "gbar": gbars, "D": None if D is None else np.asarray(D),
                   "M": M, "O": O, "a_b": list(a_b[b])}
            if diagnostics:
                diag["E_KV"] = 0.5 * (diag["E_K"] + diag["E_V"])
                rec.update(diag)
            step_rec.append(rec)
            prev_q[b] = q_tgt
            prev_M[b] = M
        records.append(step_rec)
    return records
