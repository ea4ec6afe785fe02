"""The C-ABI library builds, loads and exports every entry point its header
declares; struct layouts agree between C and the Python binding; host-side
argument checks reject bad calls before touching the GPU (no GPU needed)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "refadapt.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2609_32415_gb300 import _lib, build
    build.build()
    return _lib.load()


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(refadapt_\w+)\s*\(", text)))


def test_header_declares_the_entry_points():
    names = _declared()
    for must in ("refadapt_joint_attn", "refadapt_q_delta", "refadapt_gate", "refadapt_ref_cache_update"):
        assert must in names


def test_library_exports_every_declared_symbol(lib):
    from paper_2609_32415_gb300 import _lib
    for name in _declared():
        assert hasattr(lib, name), name
    assert set(_lib.EXPORTED) == set(_declared())


def test_struct_layouts_match_c(tmp_path):
    from paper_2609_32415_gb300._lib import RaAttnArgs, RaGateArgs, RaSeg
    src = tmp_path / "layout.c"
    src.write_text(r'''
#include <stdio.h>
#include <stddef.h>
#include "refadapt.h"
int main(void) {
  printf("%zu %zu %zu\n", sizeof(ra_seg), sizeof(ra_attn_args), sizeof(ra_gate_args));
  printf("%zu %zu %zu %zu\n", offsetof(ra_attn_args, q), offsetof(ra_attn_args, softmax_scale),
         offsetof(ra_attn_args, mode), offsetof(ra_attn_args, err_word));
  printf("%zu %zu %zu %zu\n", offsetof(ra_attn_args, ref_fresh_q), offsetof(ra_attn_args, ref_fresh_v),
         offsetof(ra_attn_args, a_b), offsetof(ra_attn_args, step));
  printf("%zu %zu %zu\n", offsetof(ra_gate_args, t), offsetof(ra_gate_args, q_delta),
         offsetof(ra_gate_args, m_out));
  return 0;
}
''')
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c99", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)],
                   check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()
    got = [int(x) for x in out]
    want = [ctypes.sizeof(RaSeg), ctypes.sizeof(RaAttnArgs), ctypes.sizeof(RaGateArgs),
            RaAttnArgs.q.offset, RaAttnArgs.softmax_scale.offset, RaAttnArgs.mode.offset,
            RaAttnArgs.err_word.offset, RaAttnArgs.ref_fresh_q.offset, RaAttnArgs.ref_fresh_v.offset,
            RaAttnArgs.a_b.offset, RaAttnArgs.step.offset, RaGateArgs.t.offset, RaGateArgs.q_delta.offset,
            RaGateArgs.m_out.offset]
    assert got == want


def test_constants_match_c(tmp_path):
    """Every constant the binding copies from the header has the header's value."""
    from paper_2609_32415_gb300 import _lib
    src = tmp_path / "consts.c"
    src.write_text(r'''
#include <stdio.h>
#include "refadapt.h"
int main(void) {
  printf("%d %d\n", (int)RA_Q_DELTA_NOALLOC_MAX_BH, (int)RA_MASS_TILE_ROWS);
  printf("%d %d %d %d %d\n", (int)RA_OK, (int)RA_EINVAL, (int)RA_EUNSUPPORTED, (int)RA_ECUDA, (int)RA_ETIMEOUT);
  printf("%d %d %d %d\n", (int)RA_MODE_REUSE, (int)RA_MODE_BOUNDARY, (int)RA_MODE_COMPUTE, (int)RA_MODE_FULL);
  printf("%d %d %d %d %d %d\n", (int)RA_TEXT, (int)RA_REF, (int)RA_TGT, (int)RA_CUE_PRODUCT, (int)RA_CUE_CHANGE,
         (int)RA_CUE_EXPOSURE);
  printf("%d %d %d %d\n", (int)RA_EPI_STORE, (int)RA_EPI_GELU, (int)RA_EPI_RESID, (int)RA_EPI_QKV);
  return 0;
}
''')
    exe = tmp_path / "consts"
    subprocess.run(["gcc", "-std=c99", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)],
                   check=True)
    got = [int(x) for x in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()]
    want = [_lib.RA_Q_DELTA_NOALLOC_MAX_BH, _lib.RA_MASS_TILE_ROWS,
            _lib.RA_OK, _lib.RA_EINVAL, _lib.RA_EUNSUPPORTED, _lib.RA_ECUDA, _lib.RA_ETIMEOUT,
            _lib.RA_MODE_REUSE, _lib.RA_MODE_BOUNDARY, _lib.RA_MODE_COMPUTE, _lib.RA_MODE_FULL,
            _lib.RA_TEXT, _lib.RA_REF, _lib.RA_TGT, _lib.RA_CUE_PRODUCT, _lib.RA_CUE_CHANGE, _lib.RA_CUE_EXPOSURE,
            _lib.RA_EPI_STORE, _lib.RA_EPI_GELU, _lib.RA_EPI_RESID, _lib.RA_EPI_QKV]
    assert got == want


def test_dit_struct_layouts_match_c(tmp_path):
    """The GEMM and modulated-LayerNorm argument structs agree between the C
    header and the ctypes binding."""
    from paper_2609_32415_gb300._lib import RaGemmArgs, RaGemmSeg, RaLnmodArgs, RaLnmodSeg
    src = tmp_path / "layout_dit.c"
    src.write_text(r'''
#include <stdio.h>
#include <stddef.h>
#include "refadapt.h"
int main(void) {
  printf("%zu %zu %zu %zu\n", sizeof(ra_lnmod_seg), sizeof(ra_lnmod_args), sizeof(ra_gemm_seg),
         sizeof(ra_gemm_args));
  printf("%zu %zu %zu\n", offsetof(ra_lnmod_seg, rows), offsetof(ra_lnmod_args, seg),
         offsetof(ra_lnmod_args, mode));
  printf("%zu %zu %zu\n", offsetof(ra_gemm_seg, gate), offsetof(ra_gemm_seg, q_out),
         offsetof(ra_gemm_seg, pos_offset));
  printf("%zu %zu %zu %zu\n", offsetof(ra_gemm_args, seg), offsetof(ra_gemm_args, mode),
         offsetof(ra_gemm_args, tile_mode), offsetof(ra_gemm_args, err_word));
  return 0;
}
''')
    exe = tmp_path / "layout_dit"
    subprocess.run(["gcc", "-std=c99", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)],
                   check=True)
    got = [int(x) for x in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()]
    want = [ctypes.sizeof(RaLnmodSeg), ctypes.sizeof(RaLnmodArgs), ctypes.sizeof(RaGemmSeg),
            ctypes.sizeof(RaGemmArgs), RaLnmodSeg.rows.offset, RaLnmodArgs.seg.offset, RaLnmodArgs.mode.offset,
            RaGemmSeg.gate.offset, RaGemmSeg.q_out.offset, RaGemmSeg.pos_offset.offset,
            RaGemmArgs.seg.offset, RaGemmArgs.mode.offset, RaGemmArgs.tile_mode.offset,
            RaGemmArgs.err_word.offset]
    assert got == want


def test_plain_c_program_links_and_calls_the_library(lib, tmp_path):
    """A C99 program links librefadapt.so through the header alone and gets the
    same answers from the host-side entry points as the Python binding
    (nothing here launches a kernel)."""
    from paper_2609_32415_gb300 import _lib
    src = tmp_path / "client.c"
    src.write_text(r'''
#include <stdio.h>
#include <string.h>
#include "refadapt.h"
int main(void) {
  ra_attn_args a;
  memset(&a, 0, sizeof(a));
  a.B = 1; a.H = 2; a.d = 96;
  ra_status st = refadapt_joint_attn(&a, NULL);
  printf("%d %d %zu %zu %d %d\n", (int)refadapt_version(), (int)refadapt_mass_partial_len(130, 4096),
         refadapt_q_delta_workspace_size(2, 24), refadapt_state_size(3), (int)st,
         strstr(refadapt_last_error(), "d = 96") != NULL);
  printf("%s\n", refadapt_status_string(RA_EINVAL));
  return 0;
}
''')
    exe = tmp_path / "client"
    pkg = os.path.dirname(_lib.LIB_PATH)
    subprocess.run(["gcc", "-std=c99", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe),
                    "-L", pkg, "-lrefadapt", "-Wl,-rpath," + pkg], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.splitlines()
    got = [int(x) for x in out[0].split()]
    want = [lib.refadapt_version(), lib.refadapt_mass_partial_len(130, 4096),
            lib.refadapt_q_delta_workspace_size(2, 24), lib.refadapt_state_size(3), _lib.RA_EINVAL, 1]
    assert got == want
    assert out[1] == lib.refadapt_status_string(_lib.RA_EINVAL).decode()


def test_sizes_and_lengths(lib):
    assert lib.refadapt_mass_partial_len(32, 256) == 1 + 2
    assert lib.refadapt_mass_partial_len(0, 129) == 2
    assert lib.refadapt_mass_partial_len(256, 4096) == 2 + 32
    assert lib.refadapt_state_size(1) > 0
    assert lib.refadapt_state_size(4) == lib.refadapt_state_size(1) + 24
    assert lib.refadapt_q_delta_workspace_size(1, 24) >= 24 * 4 + 24 * 2 * 8
    assert lib.refadapt_q_delta_workspace_size(0, 24) == 0
    assert lib.refadapt_version() == 1
    assert lib.refadapt_status_string(4).startswith(b"RA_ETIMEOUT")


def _seg(ptr, n, sb=0, sh=0, sn=128):
    from paper_2609_32415_gb300._lib import RaSeg
    return RaSeg(ptr, sb, sh, sn, n, 0)


def test_host_validation_rejects_before_launch(lib):
    """Fake (never dereferenced) device pointers: every call must fail in the
    host-side checks with RA_EINVAL and a reason."""
    from paper_2609_32415_gb300._lib import RA_EINVAL, RaAttnArgs, RaGateArgs
    a = RaAttnArgs()
    a.B, a.H, a.d = 1, 2, 96
    assert lib.refadapt_joint_attn(ctypes.byref(a), None) == RA_EINVAL
    assert b"d = 96" in lib.refadapt_last_error()
    a.d = 128
    for r in range(3):
        for arr in (a.q, a.k, a.v, a.o):
            arr[r] = _seg(0x10000 + 0x1000 * r, 64)
    a.mass_partial = 0x90000
    a.q[2] = _seg(0x10002, 64)   # misaligned
    assert lib.refadapt_joint_attn(ctypes.byref(a), None) == RA_EINVAL
    assert b"aligned" in lib.refadapt_last_error()
    a.q[2] = _seg(0x12000, 63)   # n disagrees with k/v/o
    assert lib.refadapt_joint_attn(ctypes.byref(a), None) == RA_EINVAL
    a.q[2] = _seg(0x12000, 64, sn=100)   # stride not a multiple of 8 elements
    assert lib.refadapt_joint_attn(ctypes.byref(a), None) == RA_EINVAL
    a.q[2] = _seg(0x12000, 64)
    a.k[2] = a.v[2] = _seg(0x12000, 0)   # no target keys
    assert lib.refadapt_joint_attn(ctypes.byref(a), None) == RA_EINVAL
    assert b"at least one key row" in lib.refadapt_last_error()
    q0 = _seg(0x10000, 0)
    assert lib.refadapt_q_delta(ctypes.byref(q0), ctypes.byref(q0), 1, 1, 128, 1e-6, 0x30000, 0x40000,
                                1 << 20, None) == RA_EINVAL   # empty slab: D undefined
    assert b">= 1" in lib.refadapt_last_error()
    q1, q2 = _seg(0x10000, 10), _seg(0x20000, 11)
    assert lib.refadapt_q_delta(ctypes.byref(q1), ctypes.byref(q2), 1, 1, 128, 1e-6, 0x30000, 0x40000,
                                1 << 20, None) == RA_EINVAL
    q2 = _seg(0x20000, 10)
    assert lib.refadapt_q_delta(ctypes.byref(q1), ctypes.byref(q2), 1, 1, 128, 1e-6, 0x30000, 0x40000,
                                16, None) == RA_EINVAL   # workspace too small
    g = RaGateArgs()
    g.B, g.H, g.t, g.delta_max = 1, 2, 3, 4
    g.state, g.mode_out = 0x50000, 0x60000
    assert lib.refadapt_gate(ctypes.byref(g), None) == RA_EINVAL   # t >= 1 without cues
    g.t, g.delta_max = 0, 0
    assert lib.refadapt_gate(ctypes.byref(g), None) == RA_EINVAL
    k = _seg(0x10000, 10)
    assert lib.refadapt_ref_cache_update(ctypes.byref(k), ctypes.byref(k), ctypes.byref(k), ctypes.byref(k),
                                         1, 1, 80, None, None, 0, 0, 0x70000, 0, None, None) == RA_EINVAL
    assert lib.refadapt_selftest_wait_timeout(None, 1000, None) == RA_EINVAL


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    """With librefadapt.so absent every entry point raises; nothing falls back to
    a CPU implementation."""
    from paper_2609_32415_gb300 import _lib, api
    monkeypatch.setattr(_lib, "LIB_PATH", str(tmp_path / "librefadapt.so"))
    monkeypatch.setattr(_lib, "_lib", None)
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        _lib.load()
    with pytest.raises(RuntimeError, match="missing"):
        api.refadapt_mass_partial_len(256, 4096)
    with pytest.raises(RuntimeError, match="missing"):
        api.refadapt_state_size(1)
