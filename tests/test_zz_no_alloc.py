"""ebd_certified_decode_static against ebd_certified_decode.

The static variant exists for callers that cannot allocate device memory
(serving stacks that fix all device memory at start-up, plugin hosts that give
an operator no allocator): its split-K scratch is a fixed 16 MiB array inside
the library, shared by every call and keeping its contents between calls.  So
it is checked on consecutive calls -- including a call of a different shape in
between -- against the workspace entry point, within the parity tolerances.

This file is named to be collected last: if it fails, a run that stops at the
first failure has already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

DEV = "cuda"
STATIC_SCRATCH_BYTES = 16 << 20


@pytest.fixture(scope="module")
def E():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_21475_gb300.build import build
    build()
    from paper_2607_21475_gb300 import ebd
    return ebd


def _case(B, H, G, d, cap, dtype, seed):
    g = torch.Generator().manual_seed(seed)
    Kc = torch.randn((B, H, cap, d), generator=g).to(dtype)
    Vc = (torch.randn((B, H, cap, d), generator=g) + 0.2).to(dtype)
    pi = torch.rand((B, H, cap), generator=g) * 0.99 + 0.01
    pi[torch.rand((B, H, cap), generator=g) < 0.25] = 1.0
    logw = (-torch.log(pi.double())).float()
    n = torch.randint(cap // 3, cap + 1, (B, H), generator=g).int()
    n[0, 0] = 0  # an empty unit
    Q = torch.randn((B, H * G, d), generator=g).to(dtype)
    return [t.to(DEV) for t in (Q, Kc, Vc, logw, n)]


def _outputs(B, Hq, d):
    y = torch.full((B, Hq, d), float("nan"), device=DEV)
    rest = [torch.full((B, Hq), float("nan"), device=DEV) for _ in range(4)]
    return [y] + rest


def _assert_close(got, ref):
    y, lse, var, bt, r = (t.double().cpu().numpy() for t in got)
    y0, lse0, var0, bt0, r0 = (t.double().cpu().numpy() for t in ref)
    ymax = np.abs(y0).max(axis=-1, keepdims=True)
    ok = ymax[..., 0] > 0
    assert np.all(np.abs(y - y0)[ok] <= 2e-3 * ymax[ok])
    assert np.all(y[~ok] == 0)
    assert np.array_equal(np.isneginf(lse), np.isneginf(lse0))
    fin = np.isfinite(lse0)
    assert np.all(np.abs(lse[fin] - lse0[fin]) <= 1e-4 * np.maximum(1, np.abs(lse0[fin])))
    for a, b in ((var, var0), (bt, bt0), (r, r0)):
        assert np.all(np.abs(a - b) <= 1e-3 * np.abs(b) + 1e-9)


@pytest.mark.parametrize("range_mode", [0, 1])
def test_static_decode_matches_workspace_decode_on_consecutive_calls(E, range_mode):
    shapes = [(4, 4, 4, 128, 1024, torch.bfloat16, 11), (2, 3, 7, 64, 320, torch.float32, 12)]
    cases = [_case(*s) for s in shapes]
    refs = []
    for (B, H, G, d, cap, dt, _), (Q, Kc, Vc, lw, n) in zip(shapes, cases):
        out = _outputs(B, H * G, d)
        E.ebd_certified_decode(Q, Kc, Vc, lw, n, *out, range_mode=range_mode)
        refs.append(out)
    torch.cuda.synchronize()
    # first shape twice, the second shape, then the first shape again
    for k in (0, 0, 1, 0):
        B, H, G, d, cap, dt, _ = shapes[k]
        Q, Kc, Vc, lw, n = cases[k]
        out = _outputs(B, H * G, d)
        st = torch.zeros(1, dtype=torch.int32, device=DEV)
        E.ebd_certified_decode_static(Q, Kc, Vc, lw, n, *out, range_mode=range_mode,
                                      dev_status=st)
        torch.cuda.synchronize()
        assert st.item() == 0
        _assert_close(out, refs[k])


def test_static_decode_refuses_requests_beyond_its_scratch(E):
    B, H, G, d, cap = 256, 8, 8, 128, 4096
    need = E.ebd_decode_workspace_bytes(E.EBD_BF16, B, H, G, d, cap)
    assert need > STATIC_SCRATCH_BYTES
    fake = ctypes.c_void_p(0x1000)  # refused before anything is enqueued
    L = E.lib()
    rc = L.ebd_certified_decode_static(E.EBD_BF16, B, H, G, d, fake, fake, fake, fake, fake, cap,
                                       ctypes.c_float(0.1), ctypes.c_float(1e-9), 0, fake, fake,
                                       fake, fake, fake, None, None)
    assert rc == 2  # EBD_ERR_CAPACITY
    assert "capacity" in E.ebd_status_string(rc).lower()
