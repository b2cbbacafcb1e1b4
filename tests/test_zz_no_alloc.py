"""ebd_certified_decode_static against ebd_certified_decode.

The static variant exists for callers that cannot allocate device memory
(serving stacks that fix all device memory at start-up, plugin hosts that give
an operator no allocator): its split-K scratch is a fixed 16 MiB array inside
the library, shared by every call and keeping its contents between calls.

The shapes below take every decode path on a GB300 (152 SMs): two that run
the split-K kernels and so keep their tile prefix and partial records in the
array -- 160 units (a thin second wave), and 4160 units, beyond the 4096 whose
tile prefix fits in shared memory, so the separate prefix kernel writes it
into the array too -- plus the on-chip cluster path and the float32 CUDA-core
path.  The calls are issued back to back on one stream (the same shape twice,
other shapes in between, then the first again) with a single synchronisation
at the end, so each call reuses the array right after the previous one; each
output is then checked against the workspace entry point's, in both range
modes, within the parity tolerances.

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
EBD_ERR_INVALID, EBD_ERR_CAPACITY, EBD_ERR_UNSUPPORTED = 1, 2, 4

# B, H, G, d, capacity, dtype, seed
SHAPES = [
    (20, 8, 4, 128, 256, torch.bfloat16, 11),   # split-K: 160 units, 2nd wave too thin
    (1040, 4, 2, 64, 64, torch.bfloat16, 12),   # split-K, 4160 units: prefix kernel
    (4, 4, 4, 128, 1024, torch.bfloat16, 13),   # clusters of CTAs, combined on chip
    (2, 3, 7, 64, 320, torch.float32, 14),      # CUDA-core kernels
]
ORDER = (0, 0, 1, 2, 0, 3, 1, 0)


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
    yn2 = np.sum(y0 * y0, axis=-1)
    for a, b, floor in ((var, var0, 1e-12 * yn2), (bt, bt0, 1e-6 * np.sqrt(yn2)),
                        (r, r0, 1e-6)):
        assert np.all(np.abs(a - b) <= 1e-3 * np.abs(b) + floor)


@pytest.mark.parametrize("range_mode", [0, 1])
def test_static_decode_matches_workspace_decode_on_back_to_back_calls(E, range_mode):
    for B, H, G, d, cap, dt, _ in SHAPES:
        code = E.EBD_BF16 if dt == torch.bfloat16 else E.EBD_F32
        assert E.ebd_decode_workspace_bytes(code, B, H, G, d, cap) <= STATIC_SCRATCH_BYTES
    cases = [_case(*s) for s in SHAPES]
    refs = []
    for (B, H, G, d, cap, dt, _), (Q, Kc, Vc, lw, n) in zip(SHAPES, cases):
        out = _outputs(B, H * G, d)
        E.ebd_certified_decode(Q, Kc, Vc, lw, n, *out, range_mode=range_mode)
        refs.append(out)
    torch.cuda.synchronize()
    outs, stats = [], []
    for k in ORDER:  # all enqueued on one stream, no synchronisation in between
        B, H, G, d, cap, dt, _ = SHAPES[k]
        Q, Kc, Vc, lw, n = cases[k]
        out = _outputs(B, H * G, d)
        st = torch.zeros(1, dtype=torch.int32, device=DEV)
        E.ebd_certified_decode_static(Q, Kc, Vc, lw, n, *out, range_mode=range_mode,
                                      dev_status=st)
        outs.append(out)
        stats.append(st)
    torch.cuda.synchronize()
    for k, out, st in zip(ORDER, outs, stats):
        assert st.item() == 0
        _assert_close(out, refs[k])


def _call(E, dt, B, H, G, d, cap, t, workspace_entry=False):
    """ctypes call of an entry point with the pointers in t (None: NULL)."""
    L = E.lib()
    ins = [t[k] for k in ("Q", "K", "V", "lw", "n")]
    outs = [t[k] for k in ("y", "lse", "var", "b", "r")]
    args = (ctypes.c_float(0.1), ctypes.c_float(1e-9), 0)
    if workspace_entry:
        return L.ebd_certified_decode(dt, B, H, G, d, *ins, cap, *args, *outs, None, None,
                                      ctypes.c_size_t(0), None)
    return L.ebd_certified_decode_static(dt, B, H, G, d, *ins, cap, *args, *outs, None, None)


def _full_size_buffers(B, H, G, d, cap):
    """Real device buffers of a request's full size, n_kept = 0 (so that even
    a launch would read no cache row and write only these outputs)."""
    bufs = {"Q": torch.zeros((B, H * G, d), dtype=torch.bfloat16, device=DEV),
            "K": torch.empty((B, H, cap, d), dtype=torch.bfloat16, device=DEV),
            "V": torch.empty((B, H, cap, d), dtype=torch.bfloat16, device=DEV),
            "lw": torch.zeros((B, H, cap), dtype=torch.float32, device=DEV),
            "n": torch.zeros((B, H), dtype=torch.int32, device=DEV),
            "y": torch.empty((B, H * G, d), dtype=torch.float32, device=DEV)}
    for k in ("lse", "var", "b", "r"):
        bufs[k] = torch.empty((B, H * G), dtype=torch.float32, device=DEV)
    return bufs, {k: ctypes.c_void_p(v.data_ptr()) for k, v in bufs.items()}


def test_static_decode_refuses_requests_beyond_its_scratch(E):
    """A valid request that needs more scratch than the array is refused with
    EBD_ERR_CAPACITY before anything is enqueued."""
    B, H, G, d, cap = 256, 8, 8, 128, 4096
    need = E.ebd_decode_workspace_bytes(E.EBD_BF16, B, H, G, d, cap)
    assert need > STATIC_SCRATCH_BYTES
    bufs, ptrs = _full_size_buffers(B, H, G, d, cap)
    rc = _call(E, E.EBD_BF16, B, H, G, d, cap, ptrs)
    torch.cuda.synchronize()
    assert rc == EBD_ERR_CAPACITY
    assert "capacity" in E.ebd_status_string(rc).lower()
    del bufs, ptrs
    torch.cuda.empty_cache()


def test_static_decode_answers_bad_requests_like_the_workspace_entry(E):
    """Argument errors come back with the workspace entry point's status,
    before the size check, even for a shape whose scratch would not fit: null
    pointers are EBD_ERR_INVALID, an unsupported head_dim EBD_ERR_UNSUPPORTED."""
    B, H, G, cap = 256, 8, 8, 4096
    null = {k: None for k in ("Q", "K", "V", "lw", "n", "y", "lse", "var", "b", "r")}
    for ws in (False, True):
        assert _call(E, E.EBD_BF16, B, H, G, 128, cap, null, ws) == EBD_ERR_INVALID
    bufs, ptrs = _full_size_buffers(B, H, G, 96, cap)
    for ws in (False, True):
        assert _call(E, E.EBD_BF16, B, H, G, 96, cap, ptrs, ws) == EBD_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    del bufs, ptrs
    torch.cuda.empty_cache()
