"""Failure detection on the GPU without a fault: a pipeline wait that never
completes gives up after its bound, reports EBD_DEV_TIMEOUT through the
device status word, and leaves the CUDA context usable for the next call.

The wait is the library's own bounded mbarrier wait (the one every
tensor-core pipeline role uses) on a barrier phase that nothing completes;
no trap, assert or unbounded loop is involved."""
import time

import pytest
import torch

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def E():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_21475_gb300.build import build
    build()
    from paper_2607_21475_gb300 import ebd
    return ebd


def test_stalled_wait_reports_timeout_and_the_context_survives(E):
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    E.ebd_check_stalled_wait(st)
    torch.cuda.synchronize()
    waited = time.perf_counter() - t0
    assert st.item() & E.EBD_DEV_TIMEOUT
    assert 1.0 < waited < 30.0           # the bound (~2 s), not a hang
    # the context still runs the path: a small certified decode right after
    B, H, G, d, cap = 2, 2, 4, 128, 64
    g = torch.Generator().manual_seed(3)
    Kc = torch.randn((B, H, cap, d), generator=g).to(torch.bfloat16).to(DEV)
    Vc = torch.randn((B, H, cap, d), generator=g).to(torch.bfloat16).to(DEV)
    logw = torch.zeros((B, H, cap), device=DEV)
    n = torch.full((B, H), cap, dtype=torch.int32, device=DEV)
    Q = torch.randn((B, H * G, d), generator=g).to(torch.bfloat16).to(DEV)
    y = torch.empty((B, H * G, d), device=DEV)
    out = [torch.empty((B, H * G), device=DEV) for _ in range(4)]
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    E.ebd_certified_decode(Q, Kc, Vc, logw, n, y, *out, dev_status=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    ref = torch.softmax(Q.double().view(B, H, G, d) @ Kc.double().transpose(-1, -2) / d ** 0.5,
                        dim=-1) @ Vc.double()
    got = y.double().view(B, H, G, d)
    assert torch.allclose(got, ref, rtol=0, atol=2e-3 * ref.abs().max().item())
    assert torch.equal(out[1].cpu(), torch.zeros_like(out[1].cpu()))   # pi = 1: V_hat = 0


def test_stalled_wait_needs_a_status_word(E):
    import ctypes
    rc = E.lib().ebd_check_stalled_wait(None, None)
    assert rc == 1  # EBD_ERR_INVALID
