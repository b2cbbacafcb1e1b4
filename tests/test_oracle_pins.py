"""Pins for the float64 oracle: each checks it against something other than
itself -- published known-answer vectors, library routines, closed forms,
brute force on tiny inputs, exact enumeration of every retention pattern,
and Monte Carlo over many seeds.  CPU only.
"""
import itertools
import math
import os

import numpy as np
import pytest
import scipy.special
import scipy.stats
import torch

from oracle.ebd_oracle import (
    deployed_certificate, red_flag, append_token, reevict_unit, systematic_keep,
    systematic_uniform, evict_unit_systematic, gather_queries, variance_contributions,
    block_scores,
    accumulated_attention_scores,
    certainty_set,
    certificate_radius,
    compact,
    evict_unit,
    full_attention,
    hajek_decode,
    inclusion_probabilities,
    inclusion_probabilities_one_shot,
    philox4x32_10,
    philox_uniforms,
    poisson_keep,
)

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# --------------------------------------------------------------------- Philox
def _kat_rows():
    rows = []
    with open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            w = [int(x, 16) for x in line.split()]
            rows.append((w[0:4], w[4:6], w[6:10]))
    return rows


@pytest.mark.parametrize("ctr,key,expect", _kat_rows())
def test_philox_known_answers(ctr, key, expect):
    out = philox4x32_10(ctr, key)
    assert [int(x) for x in out] == expect


def test_philox_vectorised_matches_scalar():
    rng = np.random.default_rng(1)
    ctr = rng.integers(0, 2**32, size=(4, 50), dtype=np.uint64)
    key = (0x12345678, 0x9ABCDEF0)
    out = philox4x32_10(tuple(ctr), key)
    for j in range(50):
        one = philox4x32_10(tuple(int(c[j]) for c in ctr), key)
        assert np.array_equal(out[:, j], one)


def test_uniforms_grid_and_distribution():
    u, x0 = philox_uniforms(seed=7, layer=3, b=2, kvh=1, n=200_000)
    k = u * 2**24
    assert np.all(k == np.floor(k)) and np.all(u >= 0) and np.all(u < 1)
    assert np.array_equal(k.astype(np.uint64), (x0 >> np.uint32(8)).astype(np.uint64))
    assert scipy.stats.kstest(u, "uniform").pvalue > 1e-4
    # the counter carries (token, kv head, layer, batch row): each word changes the stream
    base, _ = philox_uniforms(7, 3, 2, 1, 1000)
    for args in [(8, 3, 2, 1), (7, 4, 2, 1), (7, 3, 3, 1), (7, 3, 2, 0)]:
        other, _ = philox_uniforms(*args, 1000)
        assert np.mean(other == base) < 0.01
    # seed's high word is the second key word
    hi, _ = philox_uniforms(7 + (1 << 32), 3, 2, 1, 1000)
    assert np.mean(hi == base) < 0.01
    # token i of the unit is word i % 4 of the call with counter word 0 = i // 4
    for i in (0, 5, 10, 999):
        direct = philox4x32_10((i // 4, 1, 3, 2), (7, 0))[i % 4]
        assert int(direct) >> 8 == int(base[i] * 2**24)


# ------------------------------------------------------------ Eq. (1) and scoring
def test_full_attention_matches_library_sdpa():
    rng = np.random.default_rng(2)
    q = rng.normal(size=(3, 32))
    K = rng.normal(size=(77, 32))
    V = rng.normal(size=(77, 32))
    got = full_attention(q, K, V)
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.tensor(q)[None, :, None, :], torch.tensor(K)[None, None].expand(1, 3, 77, 32),
        torch.tensor(V)[None, None].expand(1, 3, 77, 32))[0, :, 0, :].numpy()
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_full_attention_special_cases():
    rng = np.random.default_rng(3)
    V = rng.normal(size=(10, 4))
    # equal keys: plain mean of the values
    K = np.ones((10, 4))
    np.testing.assert_allclose(full_attention(rng.normal(size=4), K, V), V.mean(0), rtol=1e-12)
    # one overwhelming logit selects its value
    K = np.zeros((10, 4))
    K[6] = 500.0
    np.testing.assert_allclose(full_attention(np.ones(4), K, V), V[6], rtol=1e-12)


def test_accumulated_scores_match_library_softmax():
    rng = np.random.default_rng(4)
    q = rng.normal(size=(21, 16))
    K = rng.normal(size=(300, 16)) * 2
    s = accumulated_attention_scores(q, K)
    ref = torch.softmax(torch.tensor(q) @ torch.tensor(K).T / 4.0, dim=1).sum(0).numpy()
    np.testing.assert_allclose(s, ref, rtol=1e-12)
    assert abs(s.sum() - 21) < 1e-10           # every softmax row sums to 1
    one = accumulated_attention_scores(q[:1], K)
    np.testing.assert_allclose(one, scipy.special.softmax(q[0] @ K.T / 4.0), rtol=1e-12)


# ---------------------------------------------------------------- certainty set
def _brute_certain(s, n_sink, n_recent, k):
    n = len(s)
    prot = set(range(min(n_sink, n))) | set(range(max(n - n_recent, 0), n))
    cand = sorted((i for i in range(n) if i not in prot), key=lambda i: (-s[i], i))
    top = set(cand[:k])
    return prot | top, top


@pytest.mark.parametrize("n,n_sink,n_recent,k", [
    (50, 4, 32, 5), (50, 4, 32, 14), (50, 4, 32, 100), (30, 4, 32, 3), (1, 4, 32, 2),
    (37, 0, 0, 7), (200, 4, 32, 0), (64, 4, 32, 28)])
def test_certainty_set_brute_force(n, n_sink, n_recent, k):
    rng = np.random.default_rng(n * 100 + k)
    # integer-valued scores force many ties; ties go to the lower index
    s = rng.integers(0, 6, size=n).astype(np.float32)
    cert, top = certainty_set(s, n_sink, n_recent, k)
    bc, bt = _brute_certain(s, n_sink, n_recent, k)
    assert set(np.flatnonzero(cert)) == bc
    assert set(np.flatnonzero(top)) == bt


# ------------------------------------------------------------- Eq. (2): pi
def _water_fill(sT, m, eps):
    """Independent exact solution of sum clip(c s, eps, 1) = m by sorting:
    try every split (h tokens at 1 from the top, l tokens at eps from the
    bottom) and keep the one whose linear solve is consistent."""
    s = np.sort(sT)[::-1]
    n = len(s)
    for h in range(n + 1):
        for l in range(n - h + 1):
            mid = s[h:n - l]
            if mid.size == 0 or mid.sum() <= 0:
                continue
            c = (m - h - eps * l) / mid.sum()
            if c <= 0:
                continue
            ok_mid = np.all(c * mid <= 1 + 1e-12) and np.all(c * mid >= eps - 1e-18)
            ok_h = h == 0 or c * s[h - 1] >= 1 - 1e-12
            ok_l = l == 0 or c * s[n - l] <= eps + 1e-18
            if ok_mid and ok_h and ok_l:
                return c
    raise AssertionError("no consistent split")


@pytest.mark.parametrize("seed,n,bt,sigma", [(0, 40, 20, 1.5), (1, 40, 12, 3.0), (2, 60, 50, 2.0),
                                             (3, 25, 10, 0.3), (4, 45, 30, 4.0)])
def test_pi_matches_water_filling(seed, n, bt, sigma):
    rng = np.random.default_rng(seed)
    s = np.exp(sigma * rng.normal(size=n))
    certain = np.zeros(n, dtype=bool)
    certain[:4] = True
    pi, c, m = inclusion_probabilities(s, certain, bt, 1e-6)
    c_ref = _water_fill(s[~certain], m, 1e-6)
    assert abs(c - c_ref) <= 1e-12 * c_ref
    assert abs(pi[~certain].sum() - m) < 1e-9 * m
    assert np.all(pi[certain] == 1.0)


def test_pi_budget_and_shape_properties():
    rng = np.random.default_rng(9)
    n = 5000
    s = np.exp(1.5 * rng.normal(size=n)).astype(np.float32)
    certain, _ = certainty_set(s, 4, 32, 100)
    pi, c, m = inclusion_probabilities(s, certain, 900, 1e-6)
    T = ~certain
    assert m == 900 - certain.sum()
    assert abs(pi[T].sum() - m) < 1e-9 * m
    assert np.all((pi[T] >= 1e-6) & (pi[T] <= 1))
    order = np.argsort(s[T], kind="stable")
    assert np.all(np.diff(pi[T][order]) >= 0)               # monotone in the score
    assert np.any(pi[T] == 1.0)                             # heavy tail clips at 1
    lin = (pi[T] > 1e-6) & (pi[T] < 1)
    np.testing.assert_allclose(pi[T][lin] / s[T][lin], c, rtol=1e-12)  # linear in between


def test_pi_equals_one_shot_eq2_without_clipping():
    rng = np.random.default_rng(10)
    s = rng.uniform(1.0, 1.5, size=400)                     # flat scores: nothing clips
    certain = np.zeros(400, dtype=bool)
    certain[:36] = True
    pi, _, _ = inclusion_probabilities(s, certain, 120, 1e-6)
    one = inclusion_probabilities_one_shot(s, certain, 120, 1e-6)
    np.testing.assert_allclose(pi, one, rtol=1e-12)


def test_pi_edge_cases():
    s = np.array([3.0, 2.0, 1.0, 0.0, -1.0, 5.0, 0.5, 0.25])
    certain = np.zeros(8, dtype=bool)
    certain[0] = True
    # budget >= everything: all ones on positive scores, floor on s <= 0
    pi, _, m = inclusion_probabilities(s, certain, 100, 1e-6)
    assert m == 7
    assert np.all(pi[[1, 2, 5, 6, 7]] == 1.0) and np.all(pi[[3, 4]] == 1e-6)
    # budget that the certainty set already uses up: floor everywhere on T
    pi, c, m = inclusion_probabilities(s, certain, 1, 1e-6)
    assert m == 0 and c == 0.0 and np.all(pi[1:] == 1e-6)
    # empty tail
    pi, _, m = inclusion_probabilities(s, np.ones(8, dtype=bool), 3, 1e-6)
    assert m == 0 and np.all(pi == 1)
    # scores <= 0 stay at the floor while the rest share the budget
    pi, _, m = inclusion_probabilities(s, certain, 4, 1e-6)
    assert np.all(pi[[3, 4]] == 1e-6)
    assert abs(pi[1:].sum() - 3) < 1e-9


# ------------------------------------------------------- Poisson draw + compaction
def test_poisson_inclusion_frequencies():
    n = 64
    pi = np.linspace(0.05, 0.95, n)
    pi[:4] = 1.0
    hits = np.zeros(n)
    S = 4000
    for seed in range(S):
        u, _ = philox_uniforms(seed, 0, 0, 0, n)
        hits += poisson_keep(pi, u)
    freq = hits / S
    assert np.all(freq[:4] == 1.0)
    z = (freq[4:] - pi[4:]) / np.sqrt(pi[4:] * (1 - pi[4:]) / S)
    assert np.max(np.abs(z)) < 4.5
    # independence between tokens: pairwise joint inclusion ~ pi_i pi_j
    u_all = np.array([philox_uniforms(seed, 0, 0, 0, n)[0] for seed in range(S)])
    keep = u_all < pi.astype(np.float32)
    joint = (keep[:, 10] & keep[:, 40]).mean()
    assert abs(joint - pi[10] * pi[40]) < 4.5 * math.sqrt(pi[10] * pi[40] / S)


def test_poisson_keep_float32_decision():
    pi = np.array([0.1 + 1e-12, 1.0, 1e-6])
    u = np.array([np.float32(0.1 + 1e-12), 0.9999999, 0.0])
    keep = poisson_keep(pi, u)
    assert not keep[0] and keep[1] and keep[2]


def test_compact_layout_and_capacity():
    rng = np.random.default_rng(11)
    K = rng.normal(size=(20, 3))
    V = rng.normal(size=(20, 3))
    pi = rng.uniform(0.1, 1, size=20)
    keep = rng.uniform(size=20) < 0.5
    Kc, Vc, logw, idx, n = compact(K, V, keep, pi, 100)
    assert n == keep.sum() and np.all(np.diff(idx) > 0)
    assert np.array_equal(Kc, K[keep]) and np.array_equal(Vc, V[keep])
    np.testing.assert_allclose(np.exp(-logw), pi[keep], rtol=1e-15)
    Kc2, _, _, idx2, n2 = compact(K, V, keep, pi, 3)
    assert n2 == n and idx2.size == 3 and np.array_equal(Kc2, K[keep][:3])


# ---------------------------------------------------- Eq. (3), Theorem 2, Eq. (4)
def test_hajek_with_unit_pi_is_exact_attention_and_zero_certificate():
    rng = np.random.default_rng(12)
    q = rng.normal(size=(3, 16))
    K = rng.normal(size=(50, 16))
    V = rng.normal(size=(50, 16))
    r = hajek_decode(q, K, V, np.zeros(50))
    np.testing.assert_allclose(r.y, full_attention(q, K, V), rtol=1e-12, atol=1e-14)
    assert np.all(r.var == 0) and np.all(r.b_exact == 0) and np.all(r.b_bound == 0)
    assert np.all(r.r_exact == 0) and np.all(r.r_bound == 0)
    np.testing.assert_allclose(r.lse, scipy.special.logsumexp(q @ K.T / 4.0, axis=1), rtol=1e-13)


def test_full_budget_reproduces_eq1():
    rng = np.random.default_rng(13)
    N, d = 120, 8
    K = rng.normal(size=(N, d))
    V = rng.normal(size=(N, d))
    q = rng.normal(size=(2, d))
    s = np.exp(rng.normal(size=N))
    r = evict_unit(K, V, s, n_sink=4, n_recent=32, k_head=5, budget_tokens=N, eps=1e-6,
                   seed=3, layer=0, b=0, kvh=0, capacity=N)
    assert r.n_kept == N and np.all(r.pi == 1)
    dec = hajek_decode(q, r.K_c, r.V_c, r.logw)
    np.testing.assert_allclose(dec.y, full_attention(q, K, V), rtol=1e-12)
    assert np.all(dec.r_bound == 0)


def test_lse_is_log_of_hajek_normaliser():
    rng = np.random.default_rng(14)
    q = rng.normal(size=(2, 8))
    K = rng.normal(size=(30, 8))
    V = rng.normal(size=(30, 8))
    logw = -np.log(rng.uniform(0.2, 1.0, size=30))
    r = hajek_decode(q, K, V, logw)
    a = np.exp(q @ K.T / math.sqrt(8))
    np.testing.assert_allclose(r.lse, np.log((a * np.exp(logw)).sum(1)), rtol=1e-13)
    w = a * np.exp(logw)
    np.testing.assert_allclose(r.y, (w @ V) / w.sum(1, keepdims=True), rtol=1e-12)


def _enumerate(shift, seed=0, nA=30, nT=12, d=8, offset=3.0):
    rng = np.random.default_rng(seed)
    K = rng.normal(size=(nA + nT, d))
    V = rng.normal(size=(nA + nT, d)) + offset
    q = rng.normal(size=d)
    q /= np.linalg.norm(q)
    K[:nA] += shift * math.sqrt(d) * q          # certainty tokens carry most of the mass
    pi = np.ones(nA + nT)
    pi[nA:] = rng.uniform(0.3, 0.9, size=nT)
    y = full_attention(q, K, V)
    a = np.exp(K @ q / math.sqrt(d))
    x = a[:, None] * (V - y) / a.sum()          # x_i of the proof of Theorem 2
    var_lin = np.sum((1 - pi[nA:]) / pi[nA:] * np.sum(x[nA:] ** 2, 1))
    EV = Emse = 0.0
    Ey = np.zeros(d)
    for pat in itertools.product([False, True], repeat=nT):
        I = np.array(pat)
        p = np.prod(np.where(I, pi[nA:], 1 - pi[nA:]))
        keep = np.concatenate([np.ones(nA, dtype=bool), I])
        r = hajek_decode(q[None], K[keep], V[keep], -np.log(pi[keep]))
        EV += p * r.var[0]
        Emse += p * np.sum((r.y[0] - y) ** 2)
        Ey += p * r.y[0]
    return EV, Emse, var_lin, Ey, y


def test_theorem2_by_exact_enumeration():
    """E[V_hat] = Var(e_lin) + O(B^2/m^2): exact expectation over all 2^12
    retention patterns, converging as the tail's share of mass shrinks."""
    devs = []
    for shift in (1.0, 2.0, 3.0):
        EV, Emse, var_lin, Ey, y = _enumerate(shift)
        devs.append(abs(EV / var_lin - 1))
        # the realised mean squared error is the linearised variance to first order
        assert abs(Emse / var_lin - 1) < 0.02
    assert devs[0] > devs[1] > devs[2]
    assert devs[2] < 0.02


def test_hajek_monte_carlo_unbiasedness_and_variance():
    """Over 2000 Philox seeds: the Hajek output is centred on Eq. (1) up to its
    O(1/m) ratio bias, and the mean of V_hat tracks the realised squared error."""
    rng = np.random.default_rng(5)
    N, d = 400, 16
    K = rng.normal(size=(N, d))
    V = rng.normal(size=(N, d))
    q = rng.normal(size=(1, d))
    scores = np.exp(K @ q[0] / 4) * np.exp(0.3 * rng.normal(size=N))
    y = full_attention(q, K, V)
    ratios = []
    for bt in (120, 200):
        ys, vs, rb = [], [], []
        for seed in range(2000):
            r = evict_unit(K, V, scores, n_sink=4, n_recent=32, k_head=10, budget_tokens=bt,
                           eps=1e-6, seed=seed, layer=0, b=0, kvh=0, capacity=N)
            dec = hajek_decode(q, r.K_c, r.V_c, r.logw)
            ys.append(dec.y[0])
            vs.append(dec.var[0])
            rb.append(dec.r_bound[0])
        err = np.array(ys) - y[0]
        mse = np.mean(np.sum(err ** 2, 1))
        ratios.append(np.mean(vs) / mse)
        assert np.linalg.norm(err.mean(0)) < 4 * math.sqrt(mse / len(ys))
        rel = np.linalg.norm(err, axis=1) / np.linalg.norm(np.array(ys), axis=1)
        assert np.mean(rel <= np.array(rb)) >= 0.9            # coverage at delta = 0.1
    assert abs(ratios[1] - 1) < 0.05 and abs(ratios[1] - 1) < abs(ratios[0] - 1) + 0.01


def test_range_term_relations():
    rng = np.random.default_rng(15)
    q = rng.normal(size=(2, 8))
    K = rng.normal(size=(40, 8))
    V = rng.normal(size=(40, 8)) + 2.0
    logw = np.concatenate([np.zeros(10), -np.log(rng.uniform(0.1, 0.9, size=30))])
    r = hajek_decode(q, K, V, logw)
    n_tail = 30
    assert np.all(r.b_exact ** 2 <= r.var * (1 + 1e-12))            # max^2 <= sum of squares
    assert np.all(r.var <= n_tail * r.b_exact ** 2 * (1 + 1e-12))   # sum <= n max^2
    assert np.all(r.b_bound >= r.b_exact)
    # one tail token far heavier than the other tail tokens (the certainty set
    # still carries most of the mass): b_t^2 carries all of V_hat
    qn = q[0] / np.linalg.norm(q[0])
    K2 = np.outer(np.full(40, -20.0), qn) * math.sqrt(8) / np.linalg.norm(q[0])
    K2[:10] = 0.0
    K2[25] = -1.0 * qn * math.sqrt(8) / np.linalg.norm(q[0])
    r2 = hajek_decode(q[:1], K2, V, logw)
    assert abs(r2.b_exact[0] ** 2 / r2.var[0] - 1) < 1e-6


def _three_row_design(v0, c, v2):
    """Three retained rows with zero logits: rows 0 and 1 certain (pi = 1),
    row 2 a tail row with pi = 1/2.  Then w = (1/2, 1/2, 1) e^0 after the
    max shift (log(1/pi_2) = ln 2), N_hat share p = (1/4, 1/4, 1/2),
    y_hat = v0/4 + c/4 + v2/2, and row 1 = (3 - 1) // 2 is the reference row
    c of the one-pass bound."""
    V = np.array([v0, c, v2], dtype=np.float64)
    K = np.zeros((3, V.shape[1]))
    logw = np.array([0.0, 0.0, math.log(2.0)])
    return hajek_decode(np.zeros((1, V.shape[1])), K, V, logw)


def test_range_bound_tight_when_reference_row_lies_between():
    """Eq. (4) by hand.  v0 = c - 4 e1, v2 = c + e1: y_hat = c - e1/2 lies on
    the line through c and v2, beyond c, so ||v2 - y|| = ||v2 - c|| + ||c - y||
    and the one-pass bound equals the definition:
    sqrt(1 - 1/2) * (1/2) * 3/2 = 3 sqrt(2) / 8.  V_hat = (1/2)(1/4)(9/4) = 9/32.
    The same holds after a shift of every value (c = (10, -3))."""
    for c in ([0.0, 0.0], [10.0, -3.0]):
        c = np.array(c)
        e1 = np.array([1.0, 0.0])
        r = _three_row_design(c - 4 * e1, c, c + e1)
        np.testing.assert_allclose(r.y[0], c - 0.5 * e1, rtol=0, atol=1e-12)
        assert abs(r.var[0] - 9 / 32) < 1e-12
        assert abs(r.b_exact[0] - 3 * math.sqrt(2) / 8) < 1e-12
        assert abs(r.b_bound[0] - 3 * math.sqrt(2) / 8) < 1e-12


def test_range_bound_strict_value_by_hand():
    """v0 = c + 4 e2, v2 = c + e1: y_hat = c + (1/2, 1).
    b_exact = (sqrt(2)/4) ||(1/2, -1)|| = (sqrt(2)/4)(sqrt(5)/2);
    b_bound = (sqrt(2)/4) (||v2 - c|| + ||y - c||) = (sqrt(2)/4)(1 + sqrt(5)/2).
    Shifted by c = (10, 0) the bound keeps that value; a bound about the
    origin would give (sqrt(2)/4)(11 + ||(10.5, 1)||), and one without the
    ||y - c|| term (sqrt(2)/4)."""
    for c in ([0.0, 0.0], [10.0, 0.0]):
        c = np.array(c)
        r = _three_row_design(c + np.array([0.0, 4.0]), c, c + np.array([1.0, 0.0]))
        s2 = math.sqrt(2) / 4
        assert abs(r.b_exact[0] - s2 * math.sqrt(5) / 2) < 1e-12
        assert abs(r.b_bound[0] - s2 * (1 + math.sqrt(5) / 2)) < 1e-12
        assert abs(r.var[0] - 0.5 * 0.25 * 1.25) < 1e-12


def test_radius_constants_by_hand():
    """Eq. (4): r = (sqrt(2 V log(1/delta)) + b log(1/delta)) / (||y|| + eps0),
    on literal inputs that single out each constant: a missing factor 2 under
    the root, log(2/delta) in place of log(1/delta), or eps0 left out of the
    denominator each change one of these values."""
    e = math.exp(-1.0)
    assert abs(certificate_radius(0.5, 0.0, 1.0, e, 0.0) - 1.0) < 1e-15
    assert abs(certificate_radius(0.0, 1.0, 2.0, e, 0.0) - 0.5) < 1e-15
    assert abs(certificate_radius(2.0, 0.0, 1.0, e ** 2, 0.0) - math.sqrt(8.0)) < 1e-14
    L = math.log(10.0)
    assert abs(certificate_radius(2.0, 3.0, 4.0, 0.1, 1.0)
               - (2 * math.sqrt(L) + 3 * L) / 5) < 1e-14
    assert abs(certificate_radius(0.0, 1.0, 0.0, e, 1e-9) - 1e9) < 1e-3
    # through hajek_decode: the tight three-row design at delta = 0.1
    r = _three_row_design([-4.0, 0.0], [0.0, 0.0], [1.0, 0.0])
    b = 3 * math.sqrt(2) / 8
    expect = (math.sqrt(2 * (9 / 32) * L) + b * L) / (0.5 + 1e-9)
    assert abs(r.r_exact[0] - expect) < 1e-12 and abs(r.r_bound[0] - expect) < 1e-12


def test_radius_scale_invariance_and_zero():
    rng = np.random.default_rng(16)
    q = rng.normal(size=(2, 8))
    K = rng.normal(size=(40, 8))
    V = rng.normal(size=(40, 8))
    logw = -np.log(rng.uniform(0.1, 1.0, size=40))
    r1 = hajek_decode(q, K, V, logw, eps0=0.0)
    r2 = hajek_decode(q, K, 7.0 * V, logw, eps0=0.0)
    np.testing.assert_allclose(r2.var, 49 * r1.var, rtol=1e-12)
    np.testing.assert_allclose(r2.b_exact, 7 * r1.b_exact, rtol=1e-12)
    np.testing.assert_allclose(r2.r_exact, r1.r_exact, rtol=1e-12)
    np.testing.assert_allclose(r2.r_bound, r1.r_bound, rtol=1e-12)
    # a common shift of every value leaves V_hat and both range terms unchanged
    r4 = hajek_decode(q, K, V + np.linspace(-30, 30, 8), logw, eps0=0.0)
    np.testing.assert_allclose(r4.var, r1.var, rtol=1e-9)
    np.testing.assert_allclose(r4.b_exact, r1.b_exact, rtol=1e-9)
    np.testing.assert_allclose(r4.b_bound, r1.b_bound, rtol=1e-9)
    # smaller delta widens the radius
    r3 = hajek_decode(q, K, V, logw, delta=0.01)
    assert np.all(r3.r_exact > r1.r_exact)
    assert np.all(certificate_radius(0.0, 0.0, 1.0, 0.1, 1e-9) == 0)


def test_empty_retained_set():
    r = hajek_decode(np.ones((2, 4)), np.zeros((0, 4)), np.zeros((0, 4)), np.zeros(0))
    assert np.all(r.y == 0) and np.all(np.isneginf(r.lse)) and np.all(r.r_bound == 0)


def test_theorem1_topk_only_design_is_blind_to_evicted_values():
    """Theorem 1: with a deterministic, value-blind design (no Poisson tail,
    m = 0) shifting every evicted value by c*u leaves the retained state
    bit-identical while the true error grows linearly in c."""
    rng = np.random.default_rng(17)
    N, d = 300, 16
    K = rng.normal(size=(N, d))
    V = rng.normal(size=(N, d))
    q = rng.normal(size=(1, d))
    s = np.exp(rng.normal(size=N))
    u = rng.normal(size=d)
    u /= np.linalg.norm(u)
    kw = dict(n_sink=4, n_recent=32, k_head=40, budget_tokens=76, eps=1e-6, seed=0,
              layer=0, b=0, kvh=0, capacity=N)
    base = evict_unit(K, V, s, **kw)
    assert base.m == 0
    evicted = ~base.keep
    errs = []
    for c in (0.0, 5.0, 10.0, 20.0):
        V2 = V.copy()
        V2[evicted] += c * u
        r = evict_unit(K, V2, s, **kw)
        assert np.array_equal(r.idx, base.idx) and np.array_equal(r.V_c, base.V_c)
        dec = hajek_decode(q, r.K_c, r.V_c, r.logw)
        np.testing.assert_array_equal(dec.y, hajek_decode(q, base.K_c, base.V_c, base.logw).y)
        errs.append(np.linalg.norm(dec.y[0] - full_attention(q, K, V2)[0]))
    # error(c) = || e0 - c * u * evicted_mass ||  is asymptotically linear in c
    assert errs[3] > errs[2] > errs[1]
    slope1 = (errs[3] - errs[2]) / 10.0
    slope2 = (errs[2] - errs[1]) / 5.0
    assert abs(slope1 - slope2) < 0.05 * slope1


# ---------------------------------------------------------------- deployed certificate
# The deployed certificate (Section 5 setup): average the radius over every
# fourth head of every layer at each of the first six decode steps, then take
# the maximum over the steps.  The pins separate that order from its
# alternatives (max over units, mean over steps, all heads).
def test_certificate_constant_radii_give_the_constant():
    r = np.full((6, 28, 3, 28), 0.37)
    cert, means = deployed_certificate(r)
    assert np.allclose(cert, 0.37) and np.allclose(means, 0.37)


def test_certificate_reads_only_every_fourth_head():
    r = np.zeros((6, 4, 2, 28))
    r[:, :, :, 1::4] = 5.0  # heads 1, 5, 9, ... are not probed
    r[:, :, :, 2::4] = 7.0
    r[:, :, :, 3::4] = 9.0
    cert, _ = deployed_certificate(r)
    assert np.all(cert == 0.0)
    r[2, 1, 0, 8] = 2.8  # one probed head of one layer at step 3, row 0
    cert, means = deployed_certificate(r)
    # 4 layers x 7 probed heads = 28 terms in the step average
    assert cert[0] == pytest.approx(2.8 / 28) and cert[1] == 0.0
    assert means[2, 0] == pytest.approx(0.1) and np.all(np.delete(means[:, 0], 2) == 0)


def test_certificate_is_mean_over_units_then_max_over_steps():
    r = np.zeros((6, 2, 1, 4))
    r[0, 0, 0, 0] = 1.0   # step 1: units (layer, head 0) average to 0.5
    r[1, :, 0, 0] = 0.2   # step 2: average 0.2
    cert, means = deployed_certificate(r)
    assert cert[0] == pytest.approx(0.5)           # not 1.0 (max over units)
    assert means[:, 0].mean() != pytest.approx(cert[0])  # not the mean over steps
    assert means[0, 0] == pytest.approx(0.5) and means[1, 0] == pytest.approx(0.2)


def test_certificate_invariant_to_layer_order_and_red_flag_threshold():
    rng = np.random.default_rng(3)
    r = rng.gamma(2.0, 0.4, size=(6, 28, 4, 28))
    cert, _ = deployed_certificate(r)
    cert_perm, _ = deployed_certificate(r[:, rng.permutation(28)])
    assert np.allclose(cert, cert_perm)
    assert np.array_equal(red_flag(cert), cert >= 1.0)
    assert red_flag(np.array([1.0]))[0] and not red_flag(np.array([0.999999]))[0]



# ---------------------------------------------------------------- append and re-eviction
# A token generated after an eviction enters with pi = 1; re-evicting the
# resident cache composes two independent Poisson designs (pi = pi_1 pi_2, so
# log(1/pi) adds).  Pins: a budget that covers the resident cache reproduces
# it, appended recent tokens are certain, and the composed weights keep the
# Horvitz-Thompson total unbiased over both rounds' draws.
def _resident(n=200, d=8, seed=1, budget=60, cap=128):
    rng = np.random.default_rng(seed)
    K = rng.standard_normal((n, d))
    V = rng.standard_normal((n, d))
    s = rng.lognormal(0.0, 1.5, n)
    r = evict_unit(K, V, s, n_sink=4, n_recent=8, k_head=6, budget_tokens=budget, eps=1e-6,
                   seed=seed, layer=0, b=0, kvh=0, capacity=cap)
    return r, rng


def test_reevict_with_a_covering_budget_reproduces_the_cache():
    r, rng = _resident()
    n = r.n_kept
    s2 = rng.lognormal(0.0, 1.0, n)
    rr = reevict_unit(r.K_c, r.V_c, r.logw, r.idx, s2, n_sink=4, n_recent=8, k_head=6,
                      budget_tokens=n + 5, eps=1e-6, seed=9, layer=0, b=0, kvh=0, capacity=256)
    assert rr.n_kept == n
    assert np.array_equal(rr.idx, r.idx) and np.allclose(rr.logw, r.logw)
    assert np.array_equal(rr.K_c, r.K_c) and np.array_equal(rr.V_c, r.V_c)


def test_appended_tokens_enter_certain_and_survive_reeviction():
    r, rng = _resident()
    K_c, V_c, lw, idx = r.K_c, r.V_c, r.logw, r.idx
    for t in range(5):
        K_c, V_c, lw, idx = append_token(K_c, V_c, lw, idx, rng.standard_normal(8),
                                         rng.standard_normal(8), 200 + t)
    assert np.all(lw[-5:] == 0.0) and list(idx[-5:]) == [200, 201, 202, 203, 204]
    s2 = rng.lognormal(0.0, 1.0, len(idx))
    rr = reevict_unit(K_c, V_c, lw, idx, s2, n_sink=4, n_recent=8, k_head=6, budget_tokens=40,
                      eps=1e-6, seed=3, layer=0, b=0, kvh=0, capacity=256)
    # the recency window of the resident order holds the appended tokens: certain, kept, pi = 1
    assert set(range(200, 205)) <= set(rr.idx.tolist())
    kept_new = np.isin(rr.idx, np.arange(200, 205))
    assert np.all(rr.logw[kept_new] == 0.0)
    # a token kept twice carries both rounds' log(1/pi)
    pos = {int(t): k for k, t in enumerate(idx)}
    for t, l in zip(rr.idx, rr.logw):
        j = pos[int(t)]
        assert l == pytest.approx(lw[j] + (-np.log(rr.inner.pi[j])), rel=1e-12, abs=1e-12)


def test_composed_weights_keep_the_total_unbiased_over_two_rounds():
    # Horvitz-Thompson total of x over both rounds' draws: E[sum_kept x e^{logw}] = sum x
    rng = np.random.default_rng(5)
    n, d = 30, 2
    K = rng.standard_normal((n, d))
    V = rng.standard_normal((n, d))
    s1 = rng.lognormal(0.0, 1.0, n)
    s2_full = rng.lognormal(0.0, 1.0, n)
    x = rng.uniform(0.5, 2.0, n)
    est, one_round = [], []
    for seed in range(3000):
        r = evict_unit(K, V, s1, n_sink=2, n_recent=2, k_head=2, budget_tokens=16, eps=1e-6,
                       seed=seed, layer=0, b=0, kvh=0, capacity=n)
        rr = reevict_unit(r.K_c, r.V_c, r.logw, r.idx, s2_full[r.idx], n_sink=2, n_recent=2,
                          k_head=1, budget_tokens=9, eps=1e-6, seed=10_000 + seed, layer=1, b=0,
                          kvh=0, capacity=n)
        est.append(np.sum(x[rr.idx] * np.exp(rr.logw)))
        one_round.append(np.sum(x[rr.idx] * np.exp(rr.inner.logw)))
    est = np.asarray(est)
    se = est.std(ddof=1) / np.sqrt(len(est))
    assert abs(est.mean() - x.sum()) < 4 * se
    # the second round's weights alone (the first round forgotten) are biased low
    one_round = np.asarray(one_round)
    assert one_round.mean() < x.sum() - 4 * one_round.std(ddof=1) / np.sqrt(len(one_round))



# ---------------------------------------------------------------- systematic design
# Systematic sampling at the same pi (Hajek 1964): each token is kept with
# probability exactly pi_i over the uniform, the tail sample size is floor or
# ceil of sum pi for every uniform, and the certainty set is always kept.
# Enumerating the uniform over an even grid makes these exact checks.
def _sys_case(n=23, seed=4):
    rng = np.random.default_rng(seed)
    pi = np.minimum(1.0, rng.uniform(0.02, 0.9, n))
    pi[5] = 1.0
    certain = np.zeros(n, dtype=bool)
    certain[[0, 7, 22]] = True
    pi[certain] = 1.0
    return pi, certain


def test_systematic_inclusion_probabilities_are_pi():
    pi, certain = _sys_case()
    grid = 1 << 12
    hits = np.zeros(len(pi))
    for k in range(grid):
        hits += systematic_keep(pi, certain, k << 12)
    freq = hits / grid
    assert np.all(freq[certain] == 1.0)
    pi32 = pi.astype(np.float32).astype(np.float64)
    np.testing.assert_allclose(freq[~certain], pi32[~certain], atol=1.0 / grid + 1e-9)


def test_systematic_sample_size_is_floor_or_ceil_of_sum():
    pi, certain = _sys_case()
    total = pi.astype(np.float32).astype(np.float64)[~certain].sum()
    for k in range(0, 1 << 24, 99991):
        keep = systematic_keep(pi, certain, k)
        n_tail = int(keep[~certain].sum())
        assert math.floor(total) <= n_tail <= math.ceil(total)
        assert np.all(keep[certain])


def test_systematic_horvitz_thompson_total_is_exact_in_expectation():
    pi, certain = _sys_case(n=31, seed=9)
    x = np.random.default_rng(2).uniform(0.1, 3.0, len(pi))
    pi32 = pi.astype(np.float32).astype(np.float64)
    grid = 1 << 12
    est = np.mean([np.sum((x / pi32)[systematic_keep(pi, certain, k << 12)])
                   for k in range(grid)])
    assert est == pytest.approx(x.sum(), rel=2e-3)


def test_systematic_eviction_keeps_the_budget():
    rng = np.random.default_rng(12)
    n = 400
    s = rng.lognormal(0.0, 1.5, n)
    K = rng.standard_normal((n, 4))
    for seed in range(6):
        r = evict_unit_systematic(K, K, s, n_sink=4, n_recent=8, k_head=10, budget_tokens=60,
                                  eps=1e-6, seed=seed, layer=2, b=1, kvh=3, capacity=128)
        n_cert = int(r.certain.sum())
        assert r.m == 60 - n_cert
        assert abs(r.n_kept - 60) <= 1  # the Poisson design only matches it in expectation
    assert 0 <= systematic_uniform(7, 2, 1, 3) < (1 << 24)



# ---------------------------------------------------------------- contributions and queries
# The per-token contributions are the terms of Theorem 2's V_hat: they sum to
# the decode's V_hat (pinned above by enumeration and Monte Carlo), certain
# rows add nothing, and the block scores partition their total.
def test_contributions_sum_to_v_hat_and_certain_rows_add_nothing():
    rng = np.random.default_rng(21)
    n, d, G = 120, 16, 3
    K = rng.standard_normal((n, d))
    V = rng.standard_normal((n, d)) + 0.5
    pi = rng.uniform(0.05, 1.0, n)
    pi[:30] = 1.0
    logw = -np.log(pi)
    q = rng.standard_normal((G, d))
    c = variance_contributions(q, K, V, logw)
    dec = hajek_decode(q, K, V, logw)
    np.testing.assert_allclose(c.sum(axis=1), dec.var, rtol=1e-10)
    assert np.all(c[:, :30] == 0.0) and np.all(c >= 0.0)


def test_block_scores_partition_the_contributions():
    c = np.array([[1.0, 2.0, 3.0, 4.0, 5.0], [0.5, 0.0, 0.25, 0.0, 1.0]])
    idx = np.array([3, 63, 64, 130, 200])
    out = block_scores(c, idx, 64, 4)
    assert list(out) == [3.5, 3.25, 4.0, 6.0]
    assert out.sum() == c.sum()


def test_gather_queries_layout():
    Q = np.arange(2 * 4 * 10 * 2).reshape(2, 4, 10, 2)  # B=2, Hq=4, Nq=10, d=2
    pos = [9, 3]
    q = gather_queries(Q, pos, n_kv_heads=2)             # G = 2, P = 2
    assert q.shape == (2, 2, 4, 2)
    # unit (b=1, kvh=1): rows g*P + p = Q[1, 2 + g, pos[p]]
    assert np.array_equal(q[1, 1, 0], Q[1, 2, 9]) and np.array_equal(q[1, 1, 1], Q[1, 2, 3])
    assert np.array_equal(q[1, 1, 2], Q[1, 3, 9]) and np.array_equal(q[1, 1, 3], Q[1, 3, 3])
