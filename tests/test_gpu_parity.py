"""GPU parity: the CUDA path through the C ABI against the float64 oracle on
the same seeded inputs.  Small cases span several tiles and ragged tails;
edge cases cover empty and tiny contexts, degenerate budgets and overflow."""
import math

import numpy as np
import pytest
import torch

from oracle import ebd_oracle as O
from tests.parity import (E0_RTOL, TIE_BAND, compare_decode_heads, compare_evict_unit,
                          oracle_unit)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def E():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_21475_gb300.build import build
    build()
    from paper_2607_21475_gb300 import ebd
    return ebd


DEV = "cuda"


def bits(t):
    t = t.detach().cpu()
    return t.view(torch.int16).numpy() if t.dtype == torch.bfloat16 else t.numpy()


def f64(t):
    return t.detach().cpu().double().numpy()


def _design(E, B, H, G, d, N, layer, seed, k_head, budget, n_sink=4, n_recent=32, iters=40,
            eps=1e-6):
    return E.design_for(batch=B, n_kv_heads=H, group=G, head_dim=d, n_ctx=N, layer=layer,
                        seed=seed, n_sink=n_sink, n_recent=n_recent, k_head=k_head,
                        budget_tokens=budget, bisect_iters=iters, eps=eps)


# ------------------------------------------------------------------ Philox
def test_philox_words_bit_exact(E):
    B, H, N = 2, 3, 1537
    seed, layer = 0x0123456789ABCDEF, 5
    x0 = torch.empty((B, H, N), dtype=torch.int32, device=DEV)
    E.ebd_philox_uniforms(seed, layer, x0)
    got = x0.cpu().numpy().view(np.uint32)
    for b in range(B):
        for h in range(H):
            _, ref = O.philox_uniforms(seed, layer, b, h, N)
            assert np.array_equal(got[b, h], ref)


# ------------------------------------------------------------- certainty + pi
PI_CASES = [
    # N, k_head, budget, score kind
    (1, 2, 1, "lognormal"),
    (17, 3, 8, "lognormal"),
    (37, 5, 30, "ties"),
    (100, 0, 50, "lognormal"),
    (100, 200, 50, "lognormal"),
    (512, 10, 51, "lognormal"),
    (512, 10, 20, "lognormal"),       # budget below the certainty set: floor everywhere
    (512, 10, 600, "lognormal"),      # budget above N: all ones
    (4097, 80, 410, "pareto"),
    (6144, 307, 1536, "signed"),      # zero / negative scores sit at the floor
    (32768, 655, 3277, "segments"),
    (70001, 1400, 7000, "lognormal"),  # ragged, beyond one smem tile of bits
    (50000, 1000, 5000, "ties"),       # large context: ordered scan of the tied top keys
    (40000, 0, 12000, "pareto"),       # large context, no top slice, clipped tail
    (250000, 5000, 25000, "lognormal"),  # a cluster of eight CTAs per unit
    (131072, 2600, 13000, "ties"),     # ties ordered across the CTAs of a cluster
]


def _scores(kind, B, H, N, seed):
    g = torch.Generator().manual_seed(seed)
    if kind == "lognormal":
        return torch.exp(1.5 * torch.randn((B, H, N), generator=g))
    if kind == "ties":
        return torch.randint(0, 5, (B, H, N), generator=g).float()
    if kind == "pareto":
        return torch.pow(1 - torch.rand((B, H, N), generator=g), -1 / 1.2)
    if kind == "signed":
        s = torch.randn((B, H, N), generator=g)
        s[s.abs() < 0.2] = 0.0
        return s
    if kind == "segments":
        pos = torch.arange(N)
        seg = torch.clamp(pos // 1092, max=29).double()
        return (torch.exp(1.5 * torch.randn((B, H, N), generator=g)) *
                torch.pow(0.5, (29 - seg) / 10).float())
    raise ValueError(kind)


@pytest.mark.parametrize("N,k_head,budget,kind", PI_CASES)
def test_compute_pi_matches_oracle(E, N, k_head, budget, kind):
    B, H = 2, 2
    s = _scores(kind, B, H, N, N + k_head).float()
    d = _design(E, B, H, 1, 64, N, 0, 0, k_head, budget)
    pi = torch.empty((B, H, N), dtype=torch.float32, device=DEV)
    mask = torch.empty((B, H, N), dtype=torch.uint8, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    E.ebd_compute_pi(d, s.to(DEV), pi, mask, st)
    torch.cuda.synchronize()
    assert st.item() == 0
    sn = s.numpy()
    for b in range(B):
        for h in range(H):
            cert, _ = O.certainty_set(sn[b, h], 4, 32, k_head)
            assert np.array_equal(mask[b, h].cpu().numpy().astype(bool), cert)
            ref, c, m = O.inclusion_probabilities(sn[b, h], cert, budget, 1e-6)
            got = pi[b, h].cpu().double().numpy()
            np.testing.assert_allclose(got, ref, rtol=2e-5, atol=0)
            if m > 0 and (~cert).any():
                assert abs(got[~cert].sum() - ref[~cert].sum()) <= 1e-4 * m + 1e-3


def test_compute_pi_flags_nonfinite(E):
    B, H, N = 1, 2, 300
    s = torch.exp(torch.randn((B, H, N)))
    s[0, 1, 100] = float("nan")
    d = _design(E, B, H, 1, 64, N, 0, 0, 10, 60)
    pi = torch.empty((B, H, N), dtype=torch.float32, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    E.ebd_compute_pi(d, s.to(DEV), pi, None, st)
    torch.cuda.synchronize()
    assert st.item() & E.EBD_DEV_NONFINITE
    assert torch.isfinite(pi).all()


# ------------------------------------------------------------------ eviction
EVICT_CASES = [
    # B, H, N, d, dtype, k_head, budget, cap
    (1, 4, 512, 64, torch.float32, 10, 51, 128),       # the tiny case
    (2, 3, 1000, 128, torch.bfloat16, 40, 250, 384),
    (1, 2, 37, 64, torch.float32, 2, 20, 64),
    (2, 2, 4097, 128, torch.bfloat16, 80, 410, 576),
    (1, 1, 1, 64, torch.float32, 2, 1, 64),
    (1, 2, 40000, 64, torch.float32, 800, 4000, 4480),      # large context (global scores)
    (2, 1, 65537, 128, torch.bfloat16, 1300, 6500, 7104),   # large, ragged (scalar loads)
    (1, 1, 100003, 64, torch.float32, 2000, 10000, 10496),  # cluster with a ragged and an empty CTA
    (1, 1, 300007, 64, torch.float32, 6000, 30000, 31232),  # beyond a cluster: global scores
]


def _run_evict(E, B, H, N, d, dtype, k_head, budget, cap, seed=0, layer=0, gen_seed=1):
    g = torch.Generator().manual_seed(gen_seed)
    K = torch.randn((B, H, N, d), generator=g).to(dtype)
    V = torch.randn((B, H, N, d), generator=g).to(dtype)
    s = torch.exp(1.5 * torch.randn((B, H, N), generator=g))
    des = _design(E, B, H, 1, d, N, layer, seed, k_head, budget)
    cc = E.alloc_compact(B, H, cap, d, dtype, DEV)
    E.ebd_evict(des, K.to(DEV), V.to(DEV), s.to(DEV), None, cc)
    torch.cuda.synchronize()
    return K, V, s, cc


@pytest.mark.parametrize("B,H,N,d,dtype,k_head,budget,cap", EVICT_CASES)
def test_evict_matches_oracle(E, B, H, N, d, dtype, k_head, budget, cap):
    K, V, s, cc = _run_evict(E, B, H, N, d, dtype, k_head, budget, cap, seed=12345, layer=3)
    assert cc.dev_status.item() == 0
    Kb, Vb = bits(K), bits(V)
    Kd, Vd, sn = K.double().numpy(), V.double().numpy(), s.numpy()
    ties = 0
    for b in range(B):
        for h in range(H):
            ref = O.evict_unit(Kd[b, h], Vd[b, h], sn[b, h], n_sink=4, n_recent=32, k_head=k_head,
                               budget_tokens=budget, eps=1e-6, seed=12345, layer=3, b=b, kvh=h,
                               capacity=cap)
            n = int(cc.n_kept[b, h])
            kg = min(n, cap)
            ties += compare_evict_unit(ref, n, cc.idx_c[b, h, :kg].cpu().numpy(),
                                       cc.logw_c[b, h, :kg].cpu().double().numpy(),
                                       bits(cc.K_c[b, h, :kg]), bits(cc.V_c[b, h, :kg]),
                                       Kb[b, h], Vb[b, h], cap)
    print(f"near ties: {ties}")


@pytest.mark.parametrize("B,H,N,d,dtype,cap", [
    (41, 8, 1000, 64, torch.bfloat16, 256),   # 328 units: three chunks of one SM count
    (100, 8, 300, 128, torch.float32, 128),   # 800 units: more chunks than side streams
])
def test_evict_pipelined_chunks_match_single_stream_and_oracle(E, B, H, N, d, dtype, cap):
    """With more units than SMs ebd_evict pipelines unit chunks over side
    streams; the outputs equal select then gather on one stream, eagerly and
    replayed from a captured graph, and sampled units (chunk edges) match the
    oracle."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    assert B * H > sms
    k_head, budget = N // 50, N // 10
    g = torch.Generator().manual_seed(21)
    K = torch.randn((B, H, N, d), generator=g).to(dtype)
    V = torch.randn((B, H, N, d), generator=g).to(dtype)
    s = torch.exp(1.5 * torch.randn((B, H, N), generator=g))
    Kg, Vg, sg = K.to(DEV), V.to(DEV), s.to(DEV)
    des = _design(E, B, H, 1, d, N, 2, 77, k_head, budget)
    ref = E.alloc_compact(B, H, cap, d, dtype, DEV)
    E.ebd_select(des, sg, ref)
    E.ebd_gather(des, Kg, Vg, ref)
    piped = E.alloc_compact(B, H, cap, d, dtype, DEV)
    E.ebd_evict(des, Kg, Vg, sg, None, piped)
    graphed = E.alloc_compact(B, H, cap, d, dtype, DEV)
    torch.cuda.synchronize()
    gr = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gr):
        E.ebd_evict(des, Kg, Vg, sg, None, graphed)
    gr.replay()
    torch.cuda.synchronize()
    for cc in (piped, graphed):
        assert cc.dev_status.item() == 0
        assert torch.equal(cc.n_kept, ref.n_kept)
        for b in range(B):
            for h in range(H):
                n = min(int(ref.n_kept[b, h]), cap)
                assert torch.equal(cc.idx_c[b, h, :n], ref.idx_c[b, h, :n])
                assert torch.equal(cc.logw_c[b, h, :n], ref.logw_c[b, h, :n])
                assert torch.equal(cc.K_c[b, h, :n], ref.K_c[b, h, :n])
                assert torch.equal(cc.V_c[b, h, :n], ref.V_c[b, h, :n])
    Kb, Vb = bits(K), bits(V)
    Kd, Vd, sn = K.double().numpy(), V.double().numpy(), s.numpy()
    for u in sorted({0, sms - 1, sms, min(2 * sms, B * H - 1), B * H - 1}):
        b, h = divmod(u, H)
        r = O.evict_unit(Kd[b, h], Vd[b, h], sn[b, h], n_sink=4, n_recent=32, k_head=k_head,
                         budget_tokens=budget, eps=1e-6, seed=77, layer=2, b=b, kvh=h,
                         capacity=cap)
        n = int(piped.n_kept[b, h])
        kg = min(n, cap)
        compare_evict_unit(r, n, piped.idx_c[b, h, :kg].cpu().numpy(),
                           piped.logw_c[b, h, :kg].cpu().double().numpy(),
                           bits(piped.K_c[b, h, :kg]), bits(piped.V_c[b, h, :kg]),
                           Kb[b, h], Vb[b, h], cap)


def test_evict_cluster_chunks_match_single_launch_and_oracle(E):
    """Contexts over 32768 tokens split each unit over a cluster of CTAs (two
    here); with more units than one wave of clusters holds, ebd_evict also
    pipelines chunks of units.  The outputs equal one select and one gather
    launch, eagerly and replayed from a captured graph, and sampled units
    (chunk edges) match the oracle."""
    B, H, N, d, dtype = 20, 8, 33000, 64, torch.bfloat16
    k_head, budget, cap = N // 50, N // 10, 3712
    g = torch.Generator(device=DEV).manual_seed(5)
    Kg = torch.randn((B, H, N, d), generator=g, device=DEV).to(dtype)
    Vg = torch.randn((B, H, N, d), generator=g, device=DEV).to(dtype)
    sg = torch.exp(1.5 * torch.randn((B, H, N), generator=g, device=DEV))
    des = _design(E, B, H, 1, d, N, 5, 99, k_head, budget)
    ref = E.alloc_compact(B, H, cap, d, dtype, DEV)
    E.ebd_select(des, sg, ref)
    E.ebd_gather(des, Kg, Vg, ref)
    piped = E.alloc_compact(B, H, cap, d, dtype, DEV)
    E.ebd_evict(des, Kg, Vg, sg, None, piped)
    graphed = E.alloc_compact(B, H, cap, d, dtype, DEV)
    torch.cuda.synchronize()
    gr = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gr):
        E.ebd_evict(des, Kg, Vg, sg, None, graphed)
    gr.replay()
    torch.cuda.synchronize()
    assert ref.dev_status.item() == 0
    for cc in (piped, graphed):
        assert cc.dev_status.item() == 0
        assert torch.equal(cc.n_kept, ref.n_kept)
        for b in range(B):
            for h in range(H):
                n = min(int(ref.n_kept[b, h]), cap)
                assert torch.equal(cc.idx_c[b, h, :n], ref.idx_c[b, h, :n])
                assert torch.equal(cc.logw_c[b, h, :n], ref.logw_c[b, h, :n])
                assert torch.equal(cc.K_c[b, h, :n], ref.K_c[b, h, :n])
                assert torch.equal(cc.V_c[b, h, :n], ref.V_c[b, h, :n])
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    wave = sms // 2
    for u in sorted({0, wave - 1, wave, min(2 * wave, B * H - 1), B * H - 1}):
        b, h = divmod(u, H)
        Ku, Vu = Kg[b, h].cpu(), Vg[b, h].cpu()
        su = sg[b, h].cpu()
        r = O.evict_unit(Ku.double().numpy(), Vu.double().numpy(), su.numpy(), n_sink=4,
                         n_recent=32, k_head=k_head, budget_tokens=budget, eps=1e-6, seed=99,
                         layer=5, b=b, kvh=h, capacity=cap)
        n = int(piped.n_kept[b, h])
        kg = min(n, cap)
        compare_evict_unit(r, n, piped.idx_c[b, h, :kg].cpu().numpy(),
                           piped.logw_c[b, h, :kg].cpu().double().numpy(),
                           bits(piped.K_c[b, h, :kg]), bits(piped.V_c[b, h, :kg]),
                           bits(Ku), bits(Vu), cap)


def test_evict_from_page_locked_host_memory_matches_device(E):
    """K, V and the scores left in page-locked host memory: the select reads the
    scores and the gather only the kept rows over the host link; the outputs
    equal those of the same call on device copies.  Pageable host memory is
    refused before any launch."""
    import ctypes
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    B, H, N, d, cap = 24, 8, 2048, 128, 384   # more units than SMs: pipelined chunks
    assert B * H > sms
    g = torch.Generator().manual_seed(5)
    K = torch.randn((B, H, N, d), generator=g).to(torch.bfloat16)
    V = torch.randn((B, H, N, d), generator=g).to(torch.bfloat16)
    s = torch.exp(1.5 * torch.randn((B, H, N), generator=g))
    des = _design(E, B, H, 4, d, N, 1, 9, N // 50, N // 10)
    dev = E.alloc_compact(B, H, cap, d, torch.bfloat16, DEV)
    E.ebd_evict(des, K.to(DEV), V.to(DEV), s.to(DEV), None, dev)
    host = E.alloc_compact(B, H, cap, d, torch.bfloat16, DEV)
    Kp, Vp, sp = K.pin_memory(), V.pin_memory(), s.pin_memory()
    E.ebd_evict(des, Kp, Vp, sp, None, host)
    sel = E.alloc_compact(B, H, cap, d, torch.bfloat16, DEV)   # the two halves alone
    E.ebd_select(des, sp, sel)
    E.ebd_gather(des, Kp, Vp, sel)
    torch.cuda.synchronize()
    for cc in (host, sel):
        assert cc.dev_status.item() == 0
        assert torch.equal(cc.n_kept, dev.n_kept)
        for b in range(B):
            for h in range(H):
                n = min(int(dev.n_kept[b, h]), cap)
                for f in ("idx_c", "logw_c", "K_c", "V_c"):
                    assert torch.equal(getattr(cc, f)[b, h, :n], getattr(dev, f)[b, h, :n]), f
    # pageable memory: the binding refuses it, and so does the C entry point
    with pytest.raises(ValueError):
        E.ebd_gather(des, K, V, sel)
    st = E.lib().ebd_gather(ctypes.byref(des), E.EBD_BF16, ctypes.c_void_p(K.data_ptr()),
                            ctypes.c_void_p(V.data_ptr()), ctypes.c_void_p(sel.idx_c.data_ptr()),
                            ctypes.c_void_p(sel.n_kept.data_ptr()), cap,
                            ctypes.c_void_p(sel.K_c.data_ptr()), ctypes.c_void_p(sel.V_c.data_ptr()),
                            ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 1  # EBD_ERR_INVALID


def test_scored_eviction_with_host_resident_values_matches_device(E):
    """Attention scoring reads every key, so K and the observation queries
    stay in device memory, but V may be page-locked host memory (only the kept
    rows are read); the outputs equal the all-device call.  A host-resident K
    is refused on this path."""
    B, H, G, N, d, R, cap = 2, 2, 4, 2048, 128, 256, 576
    g = torch.Generator().manual_seed(8)
    K = torch.randn((B, H, N, d), generator=g).to(torch.bfloat16)
    V = torch.randn((B, H, N, d), generator=g).to(torch.bfloat16)
    q = torch.randn((B, H, R, d), generator=g).to(torch.bfloat16)
    des = _design(E, B, H, G, d, N, 0, 3, N // 50, N // 5)
    ref = E.alloc_compact(B, H, cap, d, torch.bfloat16, DEV)
    E.ebd_evict(des, K.to(DEV), V.to(DEV), None, q.to(DEV), ref)
    out = E.alloc_compact(B, H, cap, d, torch.bfloat16, DEV)
    E.ebd_evict(des, K.to(DEV), V.pin_memory(), None, q.to(DEV), out)
    torch.cuda.synchronize()
    assert out.dev_status.item() == 0 and torch.equal(out.n_kept, ref.n_kept)
    for b in range(B):
        for h in range(H):
            n = min(int(ref.n_kept[b, h]), cap)
            for f in ("idx_c", "logw_c", "K_c", "V_c"):
                assert torch.equal(getattr(out, f)[b, h, :n], getattr(ref, f)[b, h, :n]), f
    with pytest.raises(ValueError):
        E.ebd_evict(des, K.pin_memory(), V.pin_memory(), None, q.to(DEV), out)


def test_evict_capacity_overflow_is_flagged_and_bounded(E):
    B, H, N, d = 1, 2, 2000, 64
    cap = 64  # far below the ~400 kept tokens
    g = torch.Generator().manual_seed(3)
    K = torch.randn((B, H, N, d), generator=g)
    V = torch.randn((B, H, N, d), generator=g)
    s = torch.exp(torch.randn((B, H, N), generator=g))
    des = _design(E, B, H, 1, d, N, 0, 0, 40, 400)
    # compact buffers carved out of larger ones, with a canary band behind them
    rows = B * H * cap
    flat_k = torch.full(((rows + 64) * d,), 7.0, device=DEV)
    flat_v = torch.full(((rows + 64) * d,), 7.0, device=DEV)
    flat_l = torch.full((rows + 64,), 7.0, device=DEV)
    flat_i = torch.full((rows + 64,), 7, dtype=torch.int32, device=DEV)
    cc = E.CompactCache(flat_k[: rows * d].view(B, H, cap, d), flat_v[: rows * d].view(B, H, cap, d),
                        flat_l[:rows].view(B, H, cap), flat_i[:rows].view(B, H, cap),
                        torch.empty((B, H), dtype=torch.int32, device=DEV),
                        torch.zeros(1, dtype=torch.int32, device=DEV))
    E.ebd_evict(des, K.to(DEV), V.to(DEV), s.to(DEV), None, cc)
    torch.cuda.synchronize()
    assert cc.dev_status.item() & E.EBD_DEV_CAPACITY
    assert torch.all(cc.n_kept.cpu() > cap)
    assert torch.all(torch.diff(cc.idx_c.cpu().long(), dim=-1) > 0)
    assert torch.all(flat_k[rows * d:] == 7.0) and torch.all(flat_v[rows * d:] == 7.0)
    assert torch.all(flat_l[rows:] == 7.0) and torch.all(flat_i[rows:] == 7)
    # decode reads min(n_kept, capacity) rows
    Q = torch.randn((B, H, d), generator=g).to(DEV)
    out = _decode(E, Q, cc.K_c, cc.V_c, cc.logw_c, cc.n_kept)
    assert np.all(np.isfinite(out[0]))


# ------------------------------------------------------------------ decode
def _decode(E, Q, cc_K, cc_V, cc_l, n_kept, exact=False):
    B, Hq, d = Q.shape
    y = torch.empty((B, Hq, d), dtype=torch.float32, device=DEV)
    lse, var, bt, r = (torch.empty((B, Hq), dtype=torch.float32, device=DEV) for _ in range(4))
    E.ebd_certified_decode(Q, cc_K, cc_V, cc_l, n_kept, y, lse, var, bt, r,
                           range_mode=E.EBD_RANGE_EXACT if exact else E.EBD_RANGE_BOUND)
    torch.cuda.synchronize()
    return (f64(y), f64(lse), f64(var), f64(bt), f64(r))


DECODE_CASES = [
    # B, H, G, d, cap, dtype, n_kept pattern
    (1, 4, 1, 64, 128, torch.float32, "random"),
    (2, 4, 7, 128, 1600, torch.bfloat16, "random"),
    (3, 2, 4, 128, 704, torch.bfloat16, "edges"),   # 0, 1, cap, ragged
    (2, 2, 8, 64, 320, torch.float32, "edges"),
    (1, 3, 2, 128, 64, torch.bfloat16, "full"),
    (2, 2, 8, 64, 512, torch.bfloat16, "edges"),     # tensor-core path, head_dim 64, G = 8
    (2, 3, 5, 128, 1000, torch.bfloat16, "random"),  # capacity not a multiple of 16: CUDA cores
    (1, 64, 4, 128, 256, torch.bfloat16, "random"),  # more warps than tiles
    (1, 1, 8, 128, 32768, torch.bfloat16, "full"),    # one unit, hundreds of partial records
    # few long units: split-K, each head's records merged by a cluster of CTAs
    (2, 2, 4, 128, 24576, torch.bfloat16, "edges"),   # empty and one-row units among them
    (1, 2, 4, 64, 16384, torch.bfloat16, "random"),   # head_dim 64
    # cluster kernel (units * C covering most SMs, long per-CTA ranges)
    (16, 4, 7, 128, 1600, torch.bfloat16, "edges"),   # 64 units, clusters of 2, empty units
    (8, 8, 8, 64, 1600, torch.bfloat16, "random"),    # head_dim 64, G = 8
    # one CTA per unit (no partner CTAs) for more units than half the SMs
    (8, 12, 4, 128, 256, torch.bfloat16, "edges"),    # 96 units
    (10, 10, 8, 64, 160, torch.bfloat16, "random"),   # 100 units, head_dim 64
    # one CTA per unit, in waves at least 80% full, for more units than SMs
    (32, 8, 4, 128, 256, torch.bfloat16, "edges"),    # 256 units
    (24, 12, 8, 64, 160, torch.bfloat16, "random"),   # 288 units, head_dim 64, G = 8
    # split-K with more units than SMs (thin last wave, units too short or long)
    (20, 10, 4, 128, 256, torch.bfloat16, "edges"),   # 200 units: a 66%-full last wave
    (20, 10, 4, 128, 96, torch.bfloat16, "edges"),    # 200 units of 6 tiles
    (4, 40, 4, 128, 8256, torch.bfloat16, "random"),  # 160 units of 516 tiles
    # groups of 1 and 3 heads: the hi/lo weight parts share one MMA (rows g, g + 4)
    (2, 4, 1, 128, 512, torch.bfloat16, "edges"),
    (6, 8, 3, 64, 256, torch.bfloat16, "random"),
    # groups of 9..16 heads: two slices of <= 8 heads, one pass each
    (2, 4, 12, 128, 512, torch.bfloat16, "edges"),    # split-K, slices of 6
    (16, 4, 12, 128, 1600, torch.bfloat16, "random"), # one CTA per unit, slices of 6
    (3, 2, 16, 64, 320, torch.bfloat16, "random"),    # split-K, slices of 8, head_dim 64
    (40, 8, 16, 128, 256, torch.bfloat16, "edges"),   # 320 units, slices of 8
    (2, 2, 12, 64, 200, torch.float32, "edges"),      # CUDA cores
    (2, 3, 9, 128, 1000, torch.bfloat16, "random"),   # CUDA cores, slices of 4 + 5
]


def _synthetic_cache(B, H, cap, d, dtype, pattern, seed, vmean=0.3, outliers=0):
    """Compact cache with V ~ N(vmean, 1) on every channel; `outliers` channels
    per unit (drawn by seed) scaled by 8, mean included, as the outlier
    channels of the 7B-shaped workload."""
    g = torch.Generator().manual_seed(seed)
    Kc = torch.randn((B, H, cap, d), generator=g).to(dtype)
    Vf = torch.randn((B, H, cap, d), generator=g) + vmean
    if outliers:
        for b in range(B):
            for h in range(H):
                ch = torch.randperm(d, generator=g)[:outliers]
                Vf[b, h, :, ch] *= 8.0
    Vc = Vf.to(dtype)
    pi = torch.rand((B, H, cap), generator=g) * 0.999 + 1e-3
    pi[torch.rand((B, H, cap), generator=g) < 0.3] = 1.0  # certainty-set rows
    logw = (-torch.log(pi.double())).float()
    units = B * H
    if pattern == "random":
        n = torch.randint(cap // 2, cap + 1, (units,), generator=g)
    elif pattern == "full":
        n = torch.full((units,), cap)
    else:
        # an overflowed unit (n_kept > cap: the decode reads the cap rows it has)
        base = [0, 1, cap, cap - 1, 63, 65, cap // 2 + 3, cap + 5]
        n = torch.tensor([base[i % len(base)] for i in range(units)])
    return Kc, Vc, logw, n.view(B, H).int()


@pytest.mark.parametrize("exact", [False, True])
@pytest.mark.parametrize("B,H,G,d,cap,dtype,pattern", DECODE_CASES)
def test_decode_matches_oracle_on_synthetic_cache(E, B, H, G, d, cap, dtype, pattern, exact):
    Kc, Vc, logw, n = _synthetic_cache(B, H, cap, d, dtype, pattern, seed=B * 100 + G)
    g = torch.Generator().manual_seed(7)
    Q = torch.randn((B, H * G, d), generator=g).to(dtype)
    out = _decode(E, Q.to(DEV), Kc.to(DEV), Vc.to(DEV), logw.to(DEV), n.to(DEV), exact)
    Qd, Kd, Vd, ld = Q.double().numpy(), Kc.double().numpy(), Vc.double().numpy(), logw.double().numpy()
    for b in range(B):
        for h in range(H):
            k = int(n[b, h])
            dec = O.hajek_decode(Qd[b, h * G:(h + 1) * G], Kd[b, h, :k], Vd[b, h, :k], ld[b, h, :k])
            sl = slice(h * G, (h + 1) * G)
            compare_decode_heads(dec, out[0][b, sl], out[1][b, sl], out[2][b, sl], out[3][b, sl],
                                 out[4][b, sl], exact)


# Values sharing a large mean on every channel: V_hat (Theorem 2) is the
# spread of the retained values about y_hat, a small fraction of their second
# moment about the origin (1/257 of it at a mean of 16 with unit spread).
# One case per decode path: clusters of CTAs, one CTA per unit in waves,
# split-K with many records per unit, split-K with more units than SMs, the
# CUDA-core kernels for float32 and for a capacity that is not a multiple of
# 16; the Qwen-7B-shaped outlier channels (x 8) carry the mean too.
MEAN_CASES = [
    # B, H, G, d, cap, dtype, pattern, mean, outlier channels
    (16, 4, 7, 128, 1600, torch.bfloat16, "edges", 16.0, 0),   # clusters of 2
    (1, 4, 7, 128, 1600, torch.bfloat16, "random", 4.0, 4),    # clusters of 8
    (32, 8, 4, 128, 256, torch.bfloat16, "edges", 16.0, 0),    # one CTA per unit, 2 waves
    (1, 1, 8, 128, 32768, torch.bfloat16, "full", 16.0, 0),    # split-K, one unit
    (2, 2, 4, 128, 24576, torch.bfloat16, "edges", 4.0, 4),    # few long units: clustered merge
    (2, 4, 7, 128, 256, torch.bfloat16, "random", 16.0, 0),    # clusters shrunk to 8 tiles per CTA
    (20, 10, 4, 128, 256, torch.bfloat16, "edges", 4.0, 4),    # split-K, 200 units
    (2, 2, 8, 64, 512, torch.bfloat16, "edges", 16.0, 0),      # split-K, head_dim 64
    (2, 2, 8, 64, 320, torch.float32, "edges", 16.0, 0),       # CUDA cores, float32
    (2, 3, 5, 128, 1000, torch.bfloat16, "random", 16.0, 4),   # CUDA cores, bf16
]


@pytest.mark.parametrize("exact", [False, True])
@pytest.mark.parametrize("B,H,G,d,cap,dtype,pattern,mean,outliers", MEAN_CASES)
def test_decode_certificate_with_large_common_mean(E, B, H, G, d, cap, dtype, pattern, mean,
                                                   outliers, exact):
    Kc, Vc, logw, n = _synthetic_cache(B, H, cap, d, dtype, pattern, seed=B * 31 + G + int(mean),
                                       vmean=mean, outliers=outliers)
    g = torch.Generator().manual_seed(17)
    Q = torch.randn((B, H * G, d), generator=g).to(dtype)
    out = _decode(E, Q.to(DEV), Kc.to(DEV), Vc.to(DEV), logw.to(DEV), n.to(DEV), exact)
    Qd, Kd, Vd, ld = Q.double().numpy(), Kc.double().numpy(), Vc.double().numpy(), logw.double().numpy()
    checked = 0
    for b in range(B):
        for h in range(H):
            k = min(int(n[b, h]), cap)
            dec = O.hajek_decode(Qd[b, h * G:(h + 1) * G], Kd[b, h, :k], Vd[b, h, :k], ld[b, h, :k])
            sl = slice(h * G, (h + 1) * G)
            compare_decode_heads(dec, out[0][b, sl], out[1][b, sl], out[2][b, sl], out[3][b, sl],
                                 out[4][b, sl], exact)
            yn2 = np.sum(dec.y * dec.y, axis=1)
            checked += int(np.sum(dec.var > 1e-9 * yn2))
    assert checked > 0  # the relative bar was exercised, not only the floor


def _decode_outputs(E, args, B, Hq, d):
    y = torch.empty((B, Hq, d), dtype=torch.float32, device=DEV)
    lse, var, bt, r = (torch.empty((B, Hq), dtype=torch.float32, device=DEV) for _ in range(4))
    E.ebd_certified_decode(*args, y, lse, var, bt, r)
    torch.cuda.synchronize()
    return y, lse, var, bt, r


@pytest.mark.parametrize("design", ["full_budget", "top_k_only"])
def test_certain_designs_give_exact_attention_and_zero_certificate(E, design):
    """Degenerate designs the method fixes exactly, end to end through both
    calls.  A budget covering the context keeps every token with pi = 1: Eq. 3
    is then Eq. 1 (full attention) and Theorem 2's (1 - pi) factor makes V_hat,
    b_t and r_t exactly zero.  A budget of just the certainty set (4 sinks, 32
    recent, the top slice; no Poisson tail) gives exact attention over the kept
    rows, again with a zero certificate."""
    B, H, G, d, N, k_head = 2, 2, 4, 128, 1000, 40
    budget = N if design == "full_budget" else 4 + 32 + k_head
    cap = 1008
    g = torch.Generator().manual_seed(31)
    K = torch.randn((B, H, N, d), generator=g).to(torch.bfloat16)
    V = torch.randn((B, H, N, d), generator=g).to(torch.bfloat16)
    Q = torch.randn((B, H * G, d), generator=g).to(torch.bfloat16)
    s = torch.exp(1.5 * torch.randn((B, H, N), generator=g))
    des = _design(E, B, H, G, d, N, 0, 9, k_head, budget)
    cc = E.alloc_compact(B, H, cap, d, torch.bfloat16, DEV)
    E.ebd_evict(des, K.to(DEV), V.to(DEV), s.to(DEV), None, cc)
    y, lse, var, bt, r = _decode_outputs(E, [Q.to(DEV), cc.K_c, cc.V_c, cc.logw_c, cc.n_kept],
                                         B, H * G, d)
    assert cc.dev_status.item() == 0
    n = cc.n_kept.cpu()
    assert bool((n == budget).all())
    assert bool((cc.logw_c.cpu()[..., :budget] == 0).all())
    for t in (var, bt, r):
        assert bool((t == 0).all())
    Kd, Vd, Qd = K.double(), V.double(), Q.double()
    for b in range(B):
        for h in range(H):
            rows = cc.idx_c[b, h, :budget].long().cpu()
            if design == "full_budget":
                assert torch.equal(rows, torch.arange(N))
            q = Qd[b, h * G:(h + 1) * G]
            a = torch.softmax(q @ Kd[b, h, rows].T / math.sqrt(d), dim=-1)
            ref = a @ Vd[b, h, rows]
            got = y[b, h * G:(h + 1) * G].double().cpu()
            scale = ref.abs().max(dim=-1, keepdim=True).values
            assert bool(((got - ref).abs() <= 2e-3 * scale).all())


def test_gather_skips_rows_with_out_of_range_indices(E):
    """ebd_gather copies exactly the rows whose index lies in [0, n_ctx): a row
    named by a negative or too large index is left as it was (a corrupt index
    list cannot make the copy read out of bounds), every other row is copied
    bit for bit."""
    B, H, N, d, cap = 2, 3, 1000, 128, 64
    g = torch.Generator().manual_seed(5)
    K = torch.randn((B, H, N, d), generator=g).to(torch.bfloat16).to(DEV)
    V = torch.randn((B, H, N, d), generator=g).to(torch.bfloat16).to(DEV)
    des = _design(E, B, H, 1, d, N, 0, 1, 10, 60)
    cc = E.alloc_compact(B, H, cap, d, torch.bfloat16, DEV)
    idx = torch.randint(0, N, (B, H, cap), generator=g).int()
    bad = torch.rand((B, H, cap), generator=g) < 0.25
    idx[bad & (torch.rand((B, H, cap), generator=g) < 0.5)] = -3
    idx[bad & (idx >= 0)] = N + 17
    cc.idx_c.copy_(idx)
    n = torch.tensor([[cap, cap - 5, 0], [1, 37, cap]], dtype=torch.int32)
    cc.n_kept.copy_(n)
    cc.K_c.fill_(7.0)
    cc.V_c.fill_(-7.0)
    E.ebd_gather(des, K, V, cc)
    torch.cuda.synchronize()
    Kc, Vc, Kh, Vh = cc.K_c.cpu(), cc.V_c.cpu(), K.cpu(), V.cpu()
    for b in range(B):
        for h in range(H):
            for p in range(cap):
                r = int(idx[b, h, p])
                if p < int(n[b, h]) and 0 <= r < N:
                    assert torch.equal(Kc[b, h, p], Kh[b, h, r])
                    assert torch.equal(Vc[b, h, p], Vh[b, h, r])
                else:
                    assert bool((Kc[b, h, p] == 7.0).all()) and bool((Vc[b, h, p] == -7.0).all())


def test_decode_workspace_needs_no_clearing_and_is_deterministic(E):
    """The decode writes every partial record before its merge reads it: a
    workspace full of garbage gives the same bits as a fresh one, call after
    call (both kernels of the tensor-core path reduce in a fixed order)."""
    B, H, G, d, cap = 4, 8, 4, 128, 2048
    Kc, Vc, logw, n = _synthetic_cache(B, H, cap, d, torch.bfloat16, "random", seed=11)
    Q = torch.randn((B, H * G, d), generator=torch.Generator().manual_seed(3)).to(torch.bfloat16)
    nb = E.ebd_decode_workspace_bytes(E.EBD_BF16, B, H, G, d, cap)
    ws = torch.full((nb,), 0x7f, dtype=torch.uint8, device=DEV)
    args = [t.to(DEV) for t in (Q, Kc, Vc, logw, n)]
    outs = []
    for i in range(3):
        if i == 2:
            ws.fill_(0xff)  # NaN patterns everywhere
        y = torch.empty((B, H * G, d), dtype=torch.float32, device=DEV)
        lse, var, bt, r = (torch.empty((B, H * G), dtype=torch.float32, device=DEV) for _ in range(4))
        E.ebd_certified_decode(*args, y, lse, var, bt, r, workspace=ws)
        torch.cuda.synchronize()
        outs.append(torch.cat([y.flatten(), lse.flatten(), var.flatten(), bt.flatten(), r.flatten()]))
    assert torch.isfinite(outs[0]).all()
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])


def test_decode_many_units_global_tile_prefix(E):
    """Above 4096 units the tile prefix no longer fits in shared memory and
    comes from a separate prefix kernel; same results against the oracle."""
    B, H, G, d, cap = 1040, 4, 2, 64, 64
    Kc, Vc, logw, n = _synthetic_cache(B, H, cap, d, torch.bfloat16, "edges", seed=5)
    Q = torch.randn((B, H * G, d), generator=torch.Generator().manual_seed(9)).to(torch.bfloat16)
    out = _decode(E, Q.to(DEV), Kc.to(DEV), Vc.to(DEV), logw.to(DEV), n.to(DEV))
    Qd, Kd, Vd, ld = Q.double().numpy(), Kc.double().numpy(), Vc.double().numpy(), logw.double().numpy()
    for b in list(range(0, B, 37)) + [B - 1]:
        for h in range(H):
            k = int(n[b, h])
            dec = O.hajek_decode(Qd[b, h * G:(h + 1) * G], Kd[b, h, :k], Vd[b, h, :k], ld[b, h, :k])
            sl = slice(h * G, (h + 1) * G)
            compare_decode_heads(dec, out[0][b, sl], out[1][b, sl], out[2][b, sl], out[3][b, sl],
                                 out[4][b, sl], False)


def test_evict_then_decode_tiny_end_to_end(E):
    from paper_2607_21475_gb300.workloads import WORKLOADS, make_layer_inputs
    w = WORKLOADS["tiny"]
    inp = make_layer_inputs(w, 0, "cpu")
    B, H, N, d, G, cap = w.batch, w.n_kv_heads, w.n_ctx, w.head_dim, w.group, w.capacity
    des = _design(E, B, H, G, d, N, 0, w.philox_seed, w.k_head, w.budget_tokens)
    cc = E.alloc_compact(B, H, cap, d, torch.float32, DEV)
    E.ebd_evict(des, inp["K"].to(DEV), inp["V"].to(DEV), inp["scores"].to(DEV), None, cc)
    out = _decode(E, inp["Q"].to(DEV), cc.K_c, cc.V_c, cc.logw_c, cc.n_kept)
    npi = {k: v.double().numpy() for k, v in inp.items()}
    decoded = ties = 0
    for b in range(B):
        for h in range(H):
            ref = oracle_unit(w, npi, b, h, 0, scores=inp["scores"][b, h].numpy())
            n = int(cc.n_kept[b, h])
            ties += int(np.sum(~ref.certain & (np.abs(ref.u - ref.pi) < TIE_BAND)))
            same = n == ref.n_kept and np.array_equal(cc.idx_c[b, h, :n].cpu().numpy(), ref.idx)
            if not same:
                continue  # a near tie moved one token; covered by test_evict_matches_oracle
            dec = O.hajek_decode(npi["Q"][b, h * G:(h + 1) * G], ref.K_c, ref.V_c, ref.logw)
            sl = slice(h * G, (h + 1) * G)
            compare_decode_heads(dec, out[0][b, sl], out[1][b, sl], out[2][b, sl], out[3][b, sl],
                                 out[4][b, sl], False)
            decoded += 1
    # every unit without a draw in the tie band is decoded and checked
    assert decoded >= 1 and decoded >= B * H - ties


# ------------------------------------------------------------------ scoring
@pytest.mark.parametrize("B,H,R,N,d,dtype", [
    (1, 2, 7, 300, 64, torch.float32),
    (2, 2, 448, 1030, 128, torch.bfloat16),
    (1, 1, 33, 129, 128, torch.bfloat16),
    (1, 3, 512, 777, 64, torch.bfloat16),    # tcgen05 path at its 512-row limit, d = 64
    (3, 1, 129, 256, 128, torch.bfloat16),   # two 128-row tiles, one partial; N = one key tile
    (2, 2, 256, 100, 128, torch.bfloat16),   # two full row tiles; N under half a key tile
    (1, 1, 1, 1, 128, torch.bfloat16),       # single row, single key
    (1, 2, 600, 500, 128, torch.bfloat16),   # above 512 rows: the mma.sync kernels
])
def test_score_matches_oracle(E, B, H, R, N, d, dtype):
    g = torch.Generator().manual_seed(R + N)
    K = (torch.randn((B, H, N, d), generator=g) * 1.5).to(dtype)
    q = torch.randn((B, H, R, d), generator=g).to(dtype)
    s = torch.empty((B, H, N), dtype=torch.float32, device=DEV)
    E.ebd_score(q.to(DEV), K.to(DEV), s)
    torch.cuda.synchronize()
    got = f64(s)
    for b in range(B):
        for h in range(H):
            ref = O.accumulated_attention_scores(q[b, h].double().numpy(), K[b, h].double().numpy())
            np.testing.assert_allclose(got[b, h], ref, rtol=E0_RTOL, atol=0)
            assert abs(got[b, h].sum() - R) < 1e-3 * R


# ------------------------------------------------------ deployed certificate
@pytest.mark.parametrize("L,B,Hq,stride", [(28, 5, 28, 4), (3, 1, 7, 4), (2, 70, 32, 1)])
def test_certificate_update_matches_oracle(E, L, B, Hq, stride):
    g = torch.Generator().manual_seed(L * 1000 + B)
    steps = torch.rand((6, L, B, Hq), generator=g) * 2.0
    cert = torch.full((B,), 123.0, device=DEV)  # overwritten at the first step
    mean = torch.empty((B,), device=DEV)
    flag = torch.empty((B,), dtype=torch.int32, device=DEV)
    means = []
    for t in range(6):
        E.ebd_certificate_update(steps[t].to(DEV), cert, first_step=(t == 0), head_stride=stride,
                                 tau=1.0, step_mean=mean, red_flag=flag)
        means.append(mean.cpu().double().numpy().copy())
    torch.cuda.synchronize()
    ref, ref_means = O.deployed_certificate(steps.double().numpy(), head_stride=stride)
    np.testing.assert_allclose(np.stack(means), ref_means, rtol=2e-6, atol=0)
    got = cert.cpu().double().numpy()
    np.testing.assert_allclose(got, ref, rtol=2e-6, atol=0)
    sure = np.abs(ref - 1.0) > 1e-5
    assert np.array_equal(flag.cpu().numpy()[sure].astype(bool), O.red_flag(ref)[sure])


# ------------------------------------------------------- append and re-eviction
def bits_t(t):
    """Bit patterns of a device tensor (bf16 compared as int16)."""
    return t.view(torch.int16) if t.dtype == torch.bfloat16 else t

def test_append_then_reevict_then_decode_matches_oracle(E):
    """A compact cache grows by 40 decode tokens (pi = 1), is evicted again with
    fresh draws (log(1/pi) composes), and the certified decode runs on the
    result; each step against the oracle on the same inputs."""
    from paper_2607_21475_gb300.workloads import WORKLOADS, make_layer_inputs
    w = WORKLOADS["qwen7b_16k_b25"].with_(batch=2, n_ctx=3000)
    layer = 2
    inp = make_layer_inputs(w, layer, DEV)
    B, H, G, d, N = w.batch, w.n_kv_heads, w.group, w.head_dim, w.n_ctx
    n_app = 40
    cap = w.capacity + n_app
    des = _design(E, B, H, G, d, N, layer, w.philox_seed, w.k_head, w.budget_tokens)
    cc = E.alloc_compact(B, H, cap, d, w.torch_dtype, DEV)
    E.ebd_evict(des, inp["K"], inp["V"], inp["scores"], None, cc)
    torch.cuda.synchronize()
    n0 = cc.n_kept.clone()
    g = torch.Generator().manual_seed(17)
    k_new = torch.randn((n_app, B, H, d), generator=g).to(w.torch_dtype)
    v_new = torch.randn((n_app, B, H, d), generator=g).to(w.torch_dtype)
    for t in range(n_app):
        pos = torch.full((B,), N + t, dtype=torch.int32, device=DEV)
        E.ebd_append(cc, k_new[t].to(DEV), v_new[t].to(DEV), pos)
    torch.cuda.synchronize()
    assert cc.dev_status.item() == 0
    assert torch.equal(cc.n_kept, n0 + n_app)
    for b in range(B):
        for h in range(H):
            n = int(n0[b, h])
            assert torch.equal(bits_t(cc.K_c[b, h, n:n + n_app]), bits_t(k_new[:, b, h].to(DEV)))
            assert torch.equal(bits_t(cc.V_c[b, h, n:n + n_app]), bits_t(v_new[:, b, h].to(DEV)))
            assert torch.all(cc.logw_c[b, h, n:n + n_app] == 0)
            assert torch.equal(cc.idx_c[b, h, n:n + n_app].cpu(), torch.arange(N, N + n_app, dtype=torch.int32))
    # re-evict with new scores and a new seed
    scores2 = torch.exp(torch.randn((B, H, cap), generator=g) * 1.5).to(DEV)
    budget2 = w.budget_tokens // 2
    cap2 = w.with_(budget=budget2 / N).capacity
    des2 = _design(E, B, H, G, d, cap, layer, w.philox_seed + 1, budget2 // 5, budget2)
    out = E.alloc_compact(B, H, cap2, d, w.torch_dtype, DEV)
    E.ebd_reevict(des2, scores2, cc, out)
    torch.cuda.synchronize()
    assert out.dev_status.item() == 0
    y = torch.empty((B, H * G, d), dtype=torch.float32, device=DEV)
    lse, var, bt, r = (torch.empty((B, H * G), dtype=torch.float32, device=DEV) for _ in range(4))
    E.ebd_certified_decode(inp["Q"], out.K_c, out.V_c, out.logw_c, out.n_kept, y, lse, var, bt, r)
    torch.cuda.synchronize()
    ties = 0
    for b in range(B):
        for h in range(H):
            n = int(cc.n_kept[b, h])
            Kr = cc.K_c[b, h, :n].double().cpu().numpy()
            Vr = cc.V_c[b, h, :n].double().cpu().numpy()
            lw = cc.logw_c[b, h, :n].double().cpu().numpy()
            ix = cc.idx_c[b, h, :n].cpu().numpy()
            ref = O.reevict_unit(Kr, Vr, lw, ix, scores2[b, h, :n].cpu().numpy(), n_sink=w.n_sink,
                                 n_recent=w.n_recent, k_head=des2.k_head, budget_tokens=budget2,
                                 eps=w.eps, seed=w.philox_seed + 1, layer=layer, b=b, kvh=h,
                                 capacity=cap2)
            inner = ref.inner
            near = (~inner.certain) & (np.abs(inner.u - inner.pi) < TIE_BAND)
            ties += int(near.sum())
            m = min(int(out.n_kept[b, h]), cap2)
            got_pos = set(np.searchsorted(ix, out.idx_c[b, h, :m].cpu().numpy()).tolist())
            diff = got_pos ^ set(inner.idx.tolist())
            assert all(near[i] for i in diff), f"unit {(b, h)}: kept sets differ at {sorted(diff)[:8]}"
            if diff:
                continue
            assert np.array_equal(out.idx_c[b, h, :m].cpu().numpy(), ref.idx)
            np.testing.assert_allclose(out.logw_c[b, h, :m].double().cpu().numpy(), ref.logw,
                                       rtol=2e-5, atol=4e-6)
            assert torch.equal(bits_t(out.K_c[b, h, :m]), bits_t(cc.K_c[b, h, inner.idx]))
            dec = O.hajek_decode(inp["Q"][b, h * G:(h + 1) * G].double().cpu().numpy(), ref.K_c,
                                 ref.V_c, ref.logw)
            sl = slice(h * G, (h + 1) * G)
            compare_decode_heads(dec, *(t[b, sl].double().cpu().numpy() for t in (y, lse, var, bt, r)),
                                 False)
    print("near ties", ties)


def test_append_and_decode_back_to_back_match_oracle(E):
    """Append -> certified decode, six times back to back on one stream with no
    synchronisation: the append lets its successor launch early, so each
    decode starts (and asks L2 for its rows, from a possibly stale n_kept)
    while the append that writes its last row, n_kept and log(1/pi) may still
    run.  Every step's outputs are checked against the oracle on that step's
    cache (the evicted rows plus the rows appended so far, pi = 1)."""
    from paper_2607_21475_gb300.workloads import WORKLOADS, make_layer_inputs
    w = WORKLOADS["qwen7b_16k_b25"].with_(batch=2, n_ctx=6000)
    layer, steps = 3, 6
    inp = make_layer_inputs(w, layer, DEV)
    B, H, G, d, N = w.batch, w.n_kv_heads, w.group, w.head_dim, w.n_ctx
    # whole 16-row tiles: the tensor-core path (8 units: clusters of 8 CTAs)
    cap = (w.capacity + steps + 15) // 16 * 16
    des = _design(E, B, H, G, d, N, layer, w.philox_seed, w.k_head, w.budget_tokens)
    cc = E.alloc_compact(B, H, cap, d, w.torch_dtype, DEV)
    E.ebd_evict(des, inp["K"], inp["V"], inp["scores"], None, cc)
    torch.cuda.synchronize()
    assert cc.dev_status.item() == 0
    n0 = cc.n_kept.cpu().numpy().copy()
    assert n0.max() + steps <= cap
    K0 = [[cc.K_c[b, h, :n0[b, h]].double().cpu().numpy() for h in range(H)] for b in range(B)]
    V0 = [[cc.V_c[b, h, :n0[b, h]].double().cpu().numpy() for h in range(H)] for b in range(B)]
    L0 = [[cc.logw_c[b, h, :n0[b, h]].double().cpu().numpy() for h in range(H)] for b in range(B)]
    g = torch.Generator().manual_seed(29)
    k_new = torch.randn((steps, B, H, d), generator=g).to(w.torch_dtype).to(DEV)
    v_new = (torch.randn((steps, B, H, d), generator=g) + 0.5).to(w.torch_dtype).to(DEV)
    qs = torch.randn((steps, B, H * G, d), generator=g).to(w.torch_dtype).to(DEV)
    outs = []
    for t in range(steps):  # all enqueued, one synchronisation at the end
        E.ebd_append(cc, k_new[t], v_new[t], torch.full((B,), N + t, dtype=torch.int32, device=DEV))
        y = torch.full((B, H * G, d), float("nan"), device=DEV)
        rest = [torch.full((B, H * G), float("nan"), device=DEV) for _ in range(4)]
        E.ebd_certified_decode(qs[t], cc.K_c, cc.V_c, cc.logw_c, cc.n_kept, y, *rest)
        outs.append([y] + rest)
    torch.cuda.synchronize()
    assert cc.dev_status.item() == 0
    kn, vn = k_new.double().cpu().numpy(), v_new.double().cpu().numpy()
    for t in range(steps):
        got = [o.double().cpu().numpy() for o in outs[t]]
        for b in range(B):
            for h in range(H):
                K = np.concatenate([K0[b][h], kn[:t + 1, b, h]])
                V = np.concatenate([V0[b][h], vn[:t + 1, b, h]])
                lw = np.concatenate([L0[b][h], np.zeros(t + 1)])
                dec = O.hajek_decode(qs[t, b, h * G:(h + 1) * G].double().cpu().numpy(), K, V, lw)
                sl = slice(h * G, (h + 1) * G)
                compare_decode_heads(dec, *(x[b, sl] for x in got), False)


# ------------------------------------------------------- systematic design
@pytest.mark.parametrize("B,H,N,budget,dist", [(2, 3, 1000, 100, "lognormal"),
                                               (1, 4, 20000, 2000, "pareto"),
                                               (2, 2, 32768, 3277, "lognormal"),
                                               (1, 2, 70001, 7000, "lognormal"),
                                               (1, 2, 131072, 13107, "pareto"),
                                               # beyond 8 x 32768 tokens: the select whose
                                               # scores stay in global memory
                                               (1, 1, 300000, 30000, "lognormal")])
def test_systematic_select_matches_oracle(E, B, H, N, budget, dist):
    g = torch.Generator().manual_seed(N + budget)
    if dist == "lognormal":
        s = torch.exp(torch.randn((B, H, N), generator=g, dtype=torch.float64) * 1.5).float()
    else:
        s = (1.0 / torch.rand((B, H, N), generator=g, dtype=torch.float64) ** (1 / 1.2)).float()
    k_head = budget // 5
    cap = budget + 64
    des = _design(E, B, H, 1, 64, N, 3, 0xABCDEF, k_head, budget)
    des.sampling = E.EBD_SAMPLING_SYSTEMATIC
    cc = E.alloc_compact(B, H, cap, 64, torch.bfloat16, DEV)
    idx, logw, n_kept, st = cc.idx_c, cc.logw_c, cc.n_kept, cc.dev_status
    sd = s.to(DEV)
    E.ebd_select(des, sd, cc)
    pi_gpu = torch.empty_like(sd)
    E.ebd_compute_pi(des, sd, pi_gpu)
    torch.cuda.synchronize()
    assert st.item() == 0
    ties = 0
    for b in range(B):
        for h in range(H):
            sc = s[b, h].double().numpy()
            ref = O.evict_unit_systematic(np.zeros((N, 1)), np.zeros((N, 1)), s[b, h].numpy(),
                                          n_sink=4, n_recent=32, k_head=k_head, budget_tokens=budget,
                                          eps=1e-6, seed=0xABCDEF, layer=3, b=b, kvh=h, capacity=cap)
            n = int(n_kept[b, h])
            got = idx[b, h, :min(n, cap)].cpu().numpy()
            # the tail sample size is floor/ceil of the device's own sum of pi
            tail = ~ref.certain
            S = pi_gpu[b, h].double().cpu().numpy()[tail].sum()
            n_tail = n - int(ref.certain.sum())
            assert math.floor(S) - 1 <= n_tail <= math.ceil(S) + 1
            # the kept set: identical except where a cumulative sum sits within
            # the float32 rounding of pi (accumulated along the tail) of an integer
            C = np.cumsum(np.where(tail, ref.pi, 0.0))
            u = ref.u[0]
            band = 1e-6 * (1.0 + C)
            d_hi = np.abs((C - u) - np.round(C - u))
            Cp = C - np.where(tail, ref.pi, 0.0)
            d_lo = np.abs((Cp - u) - np.round(Cp - u))
            near = tail & ((d_hi < band) | (d_lo < band))
            diff = set(got.tolist()) ^ set(ref.idx.tolist())
            bad = [i for i in diff if not near[i]]
            assert not bad, f"unit {(b, h)}: kept sets differ at {bad[:8]}"
            ties += int(near.sum())
            assert set(np.flatnonzero(ref.certain).tolist()) <= set(got.tolist())
            lw_ref = -np.log(ref.pi[got])
            np.testing.assert_allclose(logw[b, h, :len(got)].double().cpu().numpy(), lw_ref,
                                       rtol=2e-5, atol=2e-6)
    print("systematic near crossings", ties)


# --------------------------------------------- observation queries and contributions
def test_snapkv_window_scores_match_oracle(E):
    """E0 from the SnapKV-style window (queries of the last 64 prefill positions)."""
    B, H, G, N, d = 2, 2, 4, 1500, 128
    g = torch.Generator().manual_seed(31)
    Qp = torch.randn((B, H * G, N, d), generator=g).to(torch.bfloat16)
    K = (torch.randn((B, H, N, d), generator=g) * 1.3).to(torch.bfloat16)
    pos = torch.arange(N - 64, N, dtype=torch.int32)
    q_obs = E.ebd_gather_queries(Qp.to(DEV), pos.to(DEV), H)
    ref_q = O.gather_queries(Qp.view(torch.int16).numpy(), pos.numpy(), H)
    assert np.array_equal(q_obs.cpu().view(torch.int16).numpy(), ref_q)
    s = torch.empty((B, H, N), dtype=torch.float32, device=DEV)
    E.ebd_score(q_obs, K.to(DEV), s)
    torch.cuda.synchronize()
    qd = O.gather_queries(Qp.double().numpy(), pos.numpy(), H)
    for b in range(B):
        for h in range(H):
            ref = O.accumulated_attention_scores(qd[b, h], K[b, h].double().numpy())
            np.testing.assert_allclose(f64(s)[b, h], ref, rtol=E0_RTOL, atol=0)


@pytest.mark.parametrize("B,H,G,d,cap,dtype", [(2, 4, 7, 128, 1600, torch.bfloat16),
                                               (2, 2, 8, 64, 512, torch.bfloat16),
                                               (1, 2, 8, 128, 256, torch.bfloat16),
                                               (1, 2, 3, 64, 320, torch.bfloat16),
                                               (1, 3, 4, 128, 1000, torch.bfloat16),
                                               (1, 2, 4, 64, 300, torch.float32)])
@pytest.mark.parametrize("vmean", [0.3, 16.0])
def test_variance_contributions_and_block_scores_match_oracle(E, B, H, G, d, cap, dtype, vmean):
    """Per-token terms of Theorem 2's V_hat and 64-token block scores; a common
    mean of 16 on every value channel checks that each term is formed about a
    retained row rather than from ||v||^2 - 2 v.y + ||y||^2."""
    Kc, Vc, logw, n = _synthetic_cache(B, H, cap, d, dtype, "random", seed=77, vmean=vmean)
    idx = torch.sort(torch.randperm(cap * 4, generator=torch.Generator().manual_seed(5))[:cap])[0]
    idx_c = idx.int().view(1, 1, cap).expand(B, H, cap).contiguous()
    Q = torch.randn((B, H * G, d), generator=torch.Generator().manual_seed(8)).to(dtype)
    args = [t.to(DEV) for t in (Q, Kc, Vc, logw, n)]
    y = torch.empty((B, H * G, d), dtype=torch.float32, device=DEV)
    lse, var, bt, r = (torch.empty((B, H * G), dtype=torch.float32, device=DEV) for _ in range(4))
    E.ebd_certified_decode(*args, y, lse, var, bt, r)
    contrib = E.ebd_variance_contributions(*args, y, lse)
    n_blocks = (cap * 4 + 63) // 64
    bs = E.ebd_block_scores(contrib, idx_c.to(DEV), args[4], 64, n_blocks)
    torch.cuda.synchronize()
    cg, bg, vg = f64(contrib), f64(bs), f64(var)
    for b in range(B):
        for h in range(H):
            k = int(n[b, h])
            sl = slice(h * G, (h + 1) * G)
            ref = O.variance_contributions(Q[b, sl].double().numpy(), Kc[b, h, :k].double().numpy(),
                                           Vc[b, h, :k].double().numpy(), logw[b, h, :k].double().numpy())
            scale = ref.max(axis=1, keepdims=True) + 1e-30
            assert np.all(np.abs(cg[b, sl, :k] - ref) <= 2e-3 * scale + 1e-12)
            assert np.all(cg[b, sl, k:] == 0.0)
            # they add up to the decode's own V_hat
            np.testing.assert_allclose(cg[b, sl, :k].sum(axis=1), vg[b, sl], rtol=2e-3, atol=1e-9)
            ref_bs = O.block_scores(ref, idx[:k].numpy(), 64, n_blocks)
            assert np.all(np.abs(bg[b, h] - ref_bs) <= 2e-3 * ref_bs.max() + 1e-12)
