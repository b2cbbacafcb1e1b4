"""Parity at the full sizes of the paper-shaped workloads, in the launch
configuration the benchmark times (one ebd_evict + one ebd_certified_decode
over the whole layer).  The float64 oracle recomputes the eviction of every
(batch row, KV head) unit (n_kept, the kept set outside the tie band, the
copied rows and log(1/pi)); the decode is checked on every unit up to 64
units and on an evenly spaced sample of 64 beyond that."""
import gc

import numpy as np
import pytest
import torch

from oracle import ebd_oracle as O
from tests.parity import E0_RTOL, compare_decode_heads, compare_evict_unit

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


def bits(t):
    t = t.detach().cpu()
    return t.view(torch.int16).numpy() if t.dtype == torch.bfloat16 else t.numpy()


def _design(E, w, layer):
    return E.design_for(batch=w.batch, n_kv_heads=w.n_kv_heads, group=w.group,
                        head_dim=w.head_dim, n_ctx=w.n_ctx, layer=layer, seed=w.philox_seed,
                        n_sink=w.n_sink, n_recent=w.n_recent, k_head=w.k_head,
                        budget_tokens=w.budget_tokens, bisect_iters=w.bisect_iters, eps=w.eps)


def _sample_units(B, H):
    return sorted({(0, 0), (B - 1, H - 1), (B // 2, H // 2)})


MAX_DECODE_UNITS = 64


def _decode_units(B, H):
    """Units whose decode is checked: all of them up to 64, else 64 evenly
    spaced ones (first and last included)."""
    n = B * H
    if n <= MAX_DECODE_UNITS:
        return set(range(n))
    return {round(i * (n - 1) / (MAX_DECODE_UNITS - 1)) for i in range(MAX_DECODE_UNITS)}


def _decode(E, Q, cc):
    B, Hq, d = Q.shape
    y = torch.empty((B, Hq, d), dtype=torch.float32, device=DEV)
    lse, var, bt, r = (torch.empty((B, Hq), dtype=torch.float32, device=DEV) for _ in range(4))
    E.ebd_certified_decode(Q, cc.K_c, cc.V_c, cc.logw_c, cc.n_kept, y, lse, var, bt, r)
    return y, lse, var, bt, r


def _check_units(E, w, inp, cc, out, scores_np, layer):
    """Eviction of every unit against the oracle; decode of _decode_units.
    Returns (near ties, units decoded, units whose kept set matched)."""
    G, H = w.group, w.n_kv_heads
    ties = 0
    decoded = 0
    matched = 0
    dec_units = _decode_units(w.batch, H)
    n_all = cc.n_kept.cpu()
    idx_all = cc.idx_c.cpu()
    for u in range(w.batch * H):
        b, h = divmod(u, H)
        K = inp["K"][b, h]
        V = inp["V"][b, h]
        ref = O.evict_unit(K.double().cpu().numpy(), V.double().cpu().numpy(), scores_np(b, h),
                           n_sink=w.n_sink, n_recent=w.n_recent, k_head=w.k_head,
                           budget_tokens=w.budget_tokens, eps=w.eps, seed=w.philox_seed,
                           layer=layer, b=b, kvh=h, capacity=w.capacity)
        n = int(n_all[b, h])
        kg = min(n, w.capacity)
        idx = idx_all[b, h, :kg].numpy()
        ties += compare_evict_unit(ref, n, idx, cc.logw_c[b, h, :kg].cpu().double().numpy(),
                                   bits(cc.K_c[b, h, :kg]), bits(cc.V_c[b, h, :kg]), bits(K),
                                   bits(V), w.capacity)
        same = n == ref.n_kept and np.array_equal(idx, ref.idx)
        matched += int(same)
        if same and u in dec_units:
            q = inp["Q"][b, h * G:(h + 1) * G].double().cpu().numpy()
            dec = O.hajek_decode(q, ref.K_c, ref.V_c, ref.logw)
            sl = slice(h * G, (h + 1) * G)
            compare_decode_heads(dec, *(t[b, sl].double().cpu().numpy() for t in out), False)
            decoded += 1
    return ties, decoded, matched


def _cleanup():
    gc.collect()
    torch.cuda.empty_cache()


@pytest.mark.parametrize("name", ["qwen7b_16k_b10", "qwen7b_16k_b25", "qwen7b_16k_b50",
                                  "dialogue_32k"])
def test_fullsize_scored_workloads(E, name):
    from paper_2607_21475_gb300.workloads import WORKLOADS, make_layer_inputs
    w = WORKLOADS[name]
    layer = 3
    inp = make_layer_inputs(w, layer, DEV)
    cc = E.alloc_compact(w.batch, w.n_kv_heads, w.capacity, w.head_dim, w.torch_dtype, DEV)
    E.ebd_evict(_design(E, w, layer), inp["K"], inp["V"], inp["scores"], None, cc)
    out = _decode(E, inp["Q"], cc)
    torch.cuda.synchronize()
    assert cc.dev_status.item() == 0
    s = inp["scores"]
    ties, decoded, matched = _check_units(E, w, inp, cc, out,
                                          lambda b, h: s[b, h].cpu().numpy(), layer)
    units = w.batch * w.n_kv_heads
    # a unit's kept set differs from the oracle's only through a near tie
    assert matched >= units - ties
    assert decoded >= min(len(_decode_units(w.batch, w.n_kv_heads)), units) - ties
    print(f"{name}: {units} units evicted, near ties {ties}, decoded units {decoded}")
    del inp, cc, out
    _cleanup()


def test_fullsize_attention_scored_workload(E):
    """Qwen-7B-shaped layer with E0 scoring from 64 x 7 observation queries."""
    from paper_2607_21475_gb300.workloads import WORKLOADS, make_layer_inputs
    w = WORKLOADS["qwen7b_6k"]
    layer = 5
    inp = make_layer_inputs(w, layer, DEV)
    B, H, N, R = w.batch, w.n_kv_heads, w.n_ctx, w.n_obs * w.group
    # E0 against the oracle on sampled units
    scores = torch.empty((B, H, N), dtype=torch.float32, device=DEV)
    E.ebd_score(inp["q_obs"], inp["K"], scores)
    torch.cuda.synchronize()
    for b, h in _sample_units(B, H):
        ref = O.accumulated_attention_scores(inp["q_obs"][b, h].double().cpu().numpy(),
                                             inp["K"][b, h].double().cpu().numpy())
        np.testing.assert_allclose(scores[b, h].double().cpu().numpy(), ref, rtol=E0_RTOL, atol=0)
    # the fused path (scores computed inside ebd_evict) keeps exactly what the
    # two-call path keeps on the scores ebd_score produced
    des = _design(E, w, layer)
    fused = E.alloc_compact(B, H, w.capacity, w.head_dim, w.torch_dtype, DEV)
    E.ebd_evict(des, inp["K"], inp["V"], None, inp["q_obs"], fused)
    split = E.alloc_compact(B, H, w.capacity, w.head_dim, w.torch_dtype, DEV)
    E.ebd_evict(des, inp["K"], inp["V"], scores, None, split)
    torch.cuda.synchronize()
    assert fused.dev_status.item() == 0 and split.dev_status.item() == 0
    assert torch.equal(fused.n_kept, split.n_kept)
    for b in range(B):
        for h in range(H):
            n = min(int(fused.n_kept[b, h]), w.capacity)
            assert torch.equal(fused.idx_c[b, h, :n], split.idx_c[b, h, :n])
    # E1-E4 and decode bit-for-bit against the oracle on the oracle's own scores
    # (rounded to float32, the precision the device decides in)
    oscores = torch.empty_like(scores)
    for b in range(B):
        for h in range(H):
            oscores[b, h] = torch.from_numpy(O.accumulated_attention_scores(
                inp["q_obs"][b, h].double().cpu().numpy(),
                inp["K"][b, h].double().cpu().numpy()).astype(np.float32))
    cc = E.alloc_compact(B, H, w.capacity, w.head_dim, w.torch_dtype, DEV)
    E.ebd_evict(des, inp["K"], inp["V"], oscores, None, cc)
    out = _decode(E, inp["Q"], cc)
    torch.cuda.synchronize()
    ties, decoded, matched = _check_units(E, w, inp, cc, out,
                                          lambda b, h: oscores[b, h].cpu().numpy(), layer)
    assert matched >= B * H - ties
    assert decoded >= min(len(_decode_units(B, H)), B * H) - ties
    del inp, cc, out, fused, split
    _cleanup()


@pytest.mark.parametrize("B,N,beta", [(1, 4096, 0.05), (8, 16384, 0.25), (32, 65536, 0.10),
                                      (64, 131072, 0.50)])
def test_fullsize_sweep_points(E, B, N, beta):
    from paper_2607_21475_gb300.workloads import sweep_workloads, make_layer_inputs
    w = [x for x in sweep_workloads()
         if x.batch == B and x.n_ctx == N and abs(x.budget - beta) < 1e-9][0]
    inp = make_layer_inputs(w, 0, DEV)
    cc = E.alloc_compact(w.batch, w.n_kv_heads, w.capacity, w.head_dim, w.torch_dtype, DEV)
    E.ebd_evict(_design(E, w, 0), inp["K"], inp["V"], inp["scores"], None, cc)
    out = _decode(E, inp["Q"], cc)
    torch.cuda.synchronize()
    assert cc.dev_status.item() == 0
    s = inp["scores"]
    ties, decoded, matched = _check_units(E, w, inp, cc, out,
                                          lambda b, h: s[b, h].cpu().numpy(), 0)
    units = w.batch * w.n_kv_heads
    assert matched >= units - ties
    assert decoded >= min(len(_decode_units(w.batch, w.n_kv_heads)), units) - ties
    del inp, cc, out
    _cleanup()


@pytest.mark.parametrize("N", [1 << 20, (1 << 20) - 3])
def test_maximum_context_eviction(E, N):
    """The largest context the library takes (2^20 tokens; and a ragged one
    just below, read with scalar loads): certainty set, pi, draws and
    compaction against the oracle, on one unit with head_dim 64."""
    d, k_head, budget = 64, round(0.02 * N), round(0.10 * N)
    cap = (budget + int(8 * budget ** 0.5) + 64 + 63) // 64 * 64
    g = torch.Generator().manual_seed(N % 997)
    K = torch.randn((1, 1, N, d), generator=g)
    V = torch.randn((1, 1, N, d), generator=g)
    s = torch.exp(1.5 * torch.randn((1, 1, N), generator=g))
    des = E.design_for(batch=1, n_kv_heads=1, group=1, head_dim=d, n_ctx=N, layer=1, seed=5,
                       k_head=k_head, budget_tokens=budget)
    cc = E.alloc_compact(1, 1, cap, d, torch.float32, DEV)
    E.ebd_evict(des, K.to(DEV), V.to(DEV), s.to(DEV), None, cc)
    torch.cuda.synchronize()
    assert cc.dev_status.item() == 0
    ref = O.evict_unit(K[0, 0].double().numpy(), V[0, 0].double().numpy(), s[0, 0].numpy(),
                       n_sink=4, n_recent=32, k_head=k_head, budget_tokens=budget, eps=1e-6,
                       seed=5, layer=1, b=0, kvh=0, capacity=cap)
    n = int(cc.n_kept[0, 0])
    kg = min(n, cap)
    compare_evict_unit(ref, n, cc.idx_c[0, 0, :kg].cpu().numpy(),
                       cc.logw_c[0, 0, :kg].cpu().double().numpy(),
                       bits(cc.K_c[0, 0, :kg]), bits(cc.V_c[0, 0, :kg]), bits(K[0, 0]),
                       bits(V[0, 0]), cap)
    del K, V, s, cc
    _cleanup()
