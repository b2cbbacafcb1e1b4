"""Shared comparison logic for the GPU-vs-oracle parity tests.

Tolerances (fp32 device arithmetic against the float64 oracle):
* top-k set, Philox words, kept-index set: bit-exact, except tail tokens whose
  uniform lies within 1e-5 of pi (a float32 pi from a float32 bisection may
  fall on the other side); those are counted and reported.
* compacted K/V rows: bit-exact copies; log(1/pi): 2e-5 relative + 2e-6 absolute.
* y_hat: max |dy| / max |y| <= 2e-3 per query head.
* V_hat, b_t, r_t: 1e-3 relative.  Absolute floors only where the
  certificate is ~0 (no tail row retained, or V_hat below 1e-12 ||y||^2):
  V_hat 1e-12 ||y||^2; b_t 1e-6 ||y|| (the square root of that floor); r_t
  1e-6 plus the V_hat floor through the square root of Eq. 4.
"""
from __future__ import annotations

import numpy as np

from oracle import ebd_oracle as O

TIE_BAND = 1e-5
Y_TOL = 2e-3
CERT_TOL = 1e-3
VAR_FLOOR = 1e-12  # times ||y_hat||^2
# E0 accumulated-attention scores against the float64 oracle: 1e-5 relative on
# every score, no absolute floor (float32 logits from exact bf16 products,
# float32 exp2 and sums; measured at most 1.0e-6 relative on the test shapes
# and on full Qwen-shaped units of 448 rows x 6144 keys)
E0_RTOL = 1e-5


def oracle_unit(w, inp_np, b, h, layer, scores=None, cap=None, k_head=None, budget=None):
    """Oracle eviction of one unit.  inp_np: dict of float64 numpy arrays."""
    s = scores if scores is not None else inp_np["scores"][b, h]
    return O.evict_unit(inp_np["K"][b, h], inp_np["V"][b, h], s, n_sink=w.n_sink,
                        n_recent=w.n_recent, k_head=w.k_head if k_head is None else k_head,
                        budget_tokens=w.budget_tokens if budget is None else budget, eps=w.eps,
                        seed=w.philox_seed, layer=layer, b=b, kvh=h,
                        capacity=w.capacity if cap is None else cap)


def compare_evict_unit(ref, n_gpu, idx_gpu, logw_gpu, Kc_gpu, Vc_gpu, K_unit, V_unit, cap):
    """Compare one unit's compaction; returns the number of near ties.

    idx_gpu / logw_gpu / Kc_gpu / Vc_gpu: numpy arrays of the first
    min(n_gpu, cap) rows.  K_unit / V_unit: the unit's uncompacted inputs in
    their storage dtype (as numpy, bit patterns preserved)."""
    tail = ~ref.certain
    near = tail & (np.abs(ref.u - ref.pi) < TIE_BAND)
    kg = min(n_gpu, cap)
    sg = set(int(i) for i in idx_gpu[:kg])
    so = set(int(i) for i in ref.idx)
    diff = sg ^ so
    bad = [i for i in diff if not near[i]]
    assert not bad, f"kept sets differ outside the tie band at tokens {bad[:10]}"
    assert np.all(np.diff(idx_gpu[:kg]) > 0), "kept indices not increasing"
    # certainty set always kept
    assert set(np.flatnonzero(ref.certain).tolist()) <= sg or n_gpu > cap
    # copies are exact, whichever set was kept
    assert np.array_equal(Kc_gpu[:kg], K_unit[idx_gpu[:kg]])
    assert np.array_equal(Vc_gpu[:kg], V_unit[idx_gpu[:kg]])
    # logw against the oracle's pi at the kept tokens
    lw_ref = -np.log(ref.pi[idx_gpu[:kg]])
    np.testing.assert_allclose(logw_gpu[:kg], lw_ref, rtol=2e-5, atol=2e-6)
    if not diff:
        assert n_gpu == ref.n_kept
    return int(near.sum())


def compare_decode_heads(dec, y, lse, var, bt, radius, exact: bool):
    """dec: oracle DecodeResult for G heads; the rest: numpy float arrays [G, ...]."""
    G = dec.y.shape[0]
    for g in range(G):
        yo = dec.y[g]
        ymax = np.abs(yo).max()
        yn = np.linalg.norm(yo)
        if ymax == 0:
            assert np.all(y[g] == 0)
            assert np.isneginf(lse[g]) == np.isneginf(dec.lse[g])
            continue
        err = np.abs(y[g] - yo).max() / ymax
        assert err <= Y_TOL, f"head {g}: y rel err {err:.3e}"
        assert abs(lse[g] - dec.lse[g]) <= 1e-4 * max(1.0, abs(dec.lse[g])), (lse[g], dec.lse[g])
        vo = dec.var[g]
        vfloor = VAR_FLOOR * yn * yn
        assert abs(var[g] - vo) <= CERT_TOL * vo + vfloor, f"head {g}: var {var[g]} vs {vo}"
        bo = dec.b_exact[g] if exact else dec.b_bound[g]
        assert abs(bt[g] - bo) <= CERT_TOL * bo + 1e-6 * yn, f"head {g}: b {bt[g]} vs {bo}"
        ro = dec.r_exact[g] if exact else dec.r_bound[g]
        rfloor = 1e-6 + np.sqrt(2 * vfloor * np.log(10.0)) / (yn + 1e-9)
        assert abs(radius[g] - ro) <= CERT_TOL * ro + rfloor, f"head {g}: r {radius[g]} vs {ro}"
