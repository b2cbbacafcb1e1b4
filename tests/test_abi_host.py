"""Host-only checks of the C ABI: the library builds for sm_103a, loads, exports
every entry point include/ebd.h declares, lays out ebd_design as C does, and
rejects bad arguments synchronously (no kernel is launched; no GPU needed)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "ebd.h")


@pytest.fixture(scope="module")
def E():
    from paper_2607_21475_gb300.build import build
    build()
    from paper_2607_21475_gb300 import ebd
    return ebd


def _declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(ebd_[a-z_0-9]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared_functions()
    for must in ("ebd_compute_pi", "ebd_evict", "ebd_certified_decode"):
        assert must in names


def test_library_exports_every_declared_symbol(E):
    L = E.lib()
    for name in _declared_functions():
        assert hasattr(L, name), name
    assert sorted(E.ABI_FUNCTIONS) == _declared_functions()
    out = subprocess.run(["nm", "-D", "--defined-only", E.lib_path()], capture_output=True,
                         text=True).stdout
    exported = set(re.findall(r" T (ebd_[a-z_0-9]+)", out))
    assert set(_declared_functions()) <= exported


def test_library_has_no_cuda_runtime_dependency(E):
    out = subprocess.run(["ldd", E.lib_path()], capture_output=True, text=True).stdout
    assert "libcudart" not in out  # static runtime: loads without a GPU stack


def test_design_struct_layout_matches_c(tmp_path, E):
    prog = tmp_path / "layout.c"
    prog.write_text(
        '#include <stdio.h>\n#include <stddef.h>\n#include "ebd.h"\n'
        "int main(void){printf(\"%zu %zu %zu %zu\\n\", sizeof(ebd_design),"
        " offsetof(ebd_design, seed), offsetof(ebd_design, bisect_iters),"
        " offsetof(ebd_design, eps)); return 0;}\n")
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), str(prog), "-o", str(exe)],
                   check=True)
    size, seed, iters, eps = map(int, subprocess.run([str(exe)], capture_output=True, text=True,
                                                     check=True).stdout.split())
    D = E.EbdDesign
    assert ctypes.sizeof(D) == size
    assert D.seed.offset == seed and D.bisect_iters.offset == iters and D.eps.offset == eps


def test_status_strings_and_version(E):
    L = E.lib()
    for code in range(6):
        assert L.ebd_status_string(code).startswith(b"EBD_")
    assert E.ebd_abi_version() == 3


def test_bad_arguments_are_rejected_synchronously(E):
    L = E.lib()
    null = ctypes.c_void_p(0)
    fake = ctypes.c_void_p(0x1000)  # never dereferenced: validation fails first
    d = E.design_for(batch=1, n_kv_heads=1, group=1, head_dim=64, n_ctx=100, k_head=5,
                     budget_tokens=20)
    byref = ctypes.byref
    # null design / scores / pi
    assert L.ebd_compute_pi(None, fake, fake, null, null, null) == 1
    assert L.ebd_compute_pi(byref(d), null, fake, null, null, null) == 1
    assert L.ebd_compute_pi(byref(d), fake, null, null, null, null) == 1
    # invalid design fields
    for field, val in [("n_ctx", 0), ("n_ctx", (1 << 20) + 1), ("batch", 0), ("bisect_iters", 0),
                       ("bisect_iters", 201), ("eps", 0.0), ("k_head", -1), ("n_sink", -2)]:
        bad = E.design_for(batch=1, n_kv_heads=1, group=1, head_dim=64, n_ctx=100, k_head=5,
                           budget_tokens=20)
        setattr(bad, field, val)
        assert L.ebd_compute_pi(byref(bad), fake, fake, null, null, null) == 1, field
    # evict: missing outputs, zero capacity, head_dim not a 16-byte row, scores and q_obs both null
    args = [byref(d), 0, fake, fake, fake, null, 0, fake, fake, fake, fake, fake, 64, fake, null, 0,
            null]
    assert L.ebd_evict(*args[:7], null, *args[8:]) == 1
    a2 = list(args)
    a2[12] = 0
    assert L.ebd_evict(*a2) == 1
    a3 = list(args)
    a3[4] = null
    assert L.ebd_evict(*a3) == 1
    d_odd = E.design_for(batch=1, n_kv_heads=1, group=1, head_dim=3, n_ctx=100, k_head=5,
                         budget_tokens=20)
    a4 = list(args)
    a4[0] = byref(d_odd)
    assert L.ebd_evict(*a4) == 4
    # decode: head_dim outside {64,128}, group > 16, delta outside (0,1), null outputs
    # (each refused before anything is enqueued)
    dec = [0, 1, 1, 1, 64, fake, fake, fake, fake, fake, 64, ctypes.c_float(0.1),
           ctypes.c_float(1e-9), 0, fake, fake, fake, fake, fake, null, fake, 1 << 20, null]
    x = list(dec)
    x[4] = 96
    assert L.ebd_certified_decode(*x) == 4
    x = list(dec)
    x[3] = 17
    assert L.ebd_certified_decode(*x) == 4
    x = list(dec)
    x[11] = ctypes.c_float(1.0)
    assert L.ebd_certified_decode(*x) == 1
    x = list(dec)
    x[16] = null
    assert L.ebd_certified_decode(*x) == 1
    x = list(dec)
    x[13] = 7
    assert L.ebd_certified_decode(*x) == 1
    # philox: null output
    assert L.ebd_philox_uniforms(0, 0, 1, 1, 10, null, null) == 1


def test_workspace_queries(E):
    d = E.design_for(batch=8, n_kv_heads=4, group=7, head_dim=128, n_ctx=6144, k_head=307,
                     budget_tokens=1536)
    assert E.ebd_evict_workspace_bytes(d, 0) == 0
    assert E.ebd_evict_workspace_bytes(d, 448) >= 8 * 4 * (6144 + 448) * 4
    assert E.ebd_score_workspace_bytes(8, 4, 448) >= 8 * 4 * 448 * 4


def test_one_workspace_size_serves_every_call_of_a_layer(E):
    """ebd_workspace_bytes(design, capacity) is the largest per-call need:
    eviction with given scores, with scoring from 64 observation positions
    per query head, and the decode in either dtype -- including a group of
    16 query heads, decoded in slices of 8."""
    for G, N, cap in ((7, 6144, 1728), (4, 32768, 3520), (16, 8192, 1024)):
        d = E.design_for(batch=8, n_kv_heads=4, group=G, head_dim=128, n_ctx=N,
                         k_head=cap // 8, budget_tokens=cap // 2)
        need = E.ebd_workspace_bytes(d, cap)
        parts = [E.ebd_evict_workspace_bytes(d, 0), E.ebd_evict_workspace_bytes(d, 64 * G)]
        parts += [E.ebd_decode_workspace_bytes(t, 8, 4, G, 128, cap)
                  for t in (E.EBD_F32, E.EBD_BF16)]
        assert need == max(parts) > 0
    assert E.lib().ebd_workspace_bytes(None, 64) == 0
    # a group of 16 heads needs the workspace of one slice of 8
    assert (E.ebd_decode_workspace_bytes(E.EBD_BF16, 8, 4, 16, 128, 1024)
            == E.ebd_decode_workspace_bytes(E.EBD_BF16, 8, 4, 8, 128, 1024))
