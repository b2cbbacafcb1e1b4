"""Float64 CPU oracle for the eviction-by-design (EBD) hot path.

TEST INFRASTRUCTURE ONLY.  The test suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` are the only callers.  The product path (the
CUDA library behind ``include/ebd.h`` and its Python binding) never imports,
links or executes anything in this directory, and this module imports nothing
from the product package.

It is a plain, slow, step-by-step restatement of what the paper
("Error Certificates for KV-Cache Eviction via Randomized Design",
arXiv 2607.21475) computes, in float64, one (batch row, KV head) unit at a
time.  Each function names the passage it follows.  Library primitives
(matrix products, a stable sort, exp/log) serve as single steps; there is no
blocking, fusion or reordering beyond the definitions.

Readings where the paper is silent or ambiguous (listed with their reasons in
the repository's design notes):

* Eq. (2) with clip-saturated tokens joining the certainty set is read as the
  fixed point  sum_T clip(c * s_i, eps, 1) = m , solved for c by bisection.
  When nothing clips this is Eq. (2) literally (``inclusion_probabilities_one_shot``).
* The certainty set is 4 sinks + 32 recent positions + the top ``k_head``
  unprotected tokens by (score descending, index ascending).
* Grouped-query attention: eviction is per KV head; the certificate is per
  query head.
* The Poisson draw uses Philox4x32-10 (Salmon et al., SC'11) with key
  (seed low word, seed high word) and counter (token // 4, kv head, layer,
  batch row); token i takes output word i % 4 and its uniform is the top 24
  bits of that word times 2^-24,
  and a tail token is kept iff  u < float32(pi)  -- the comparison is taken in
  single precision on both sides because that is the precision the device
  path decides it in.
* The range term b_t of Eq. (4) is produced in two forms: ``exact`` (the
  definition, needs y_hat inside the max) and ``bound`` (triangle inequality
  about a reference row c, computable in one pass; always >= exact).  c is
  the middle retained row, V_c[(n - 1) // 2]: like b_t itself the bound is
  then unchanged when every value moves by the same vector.

Every function here is pinned by the ``-m "not gpu"`` tests against closed
forms, library routines, brute-force enumeration and Monte Carlo; none is
"parity unpinned".
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

__all__ = [
    "philox4x32_10",
    "philox_uniforms",
    "full_attention",
    "accumulated_attention_scores",
    "certainty_set",
    "tail_budget",
    "inclusion_probabilities",
    "inclusion_probabilities_one_shot",
    "poisson_keep",
    "compact",
    "evict_unit",
    "hajek_decode",
    "certificate_radius",
    "EvictResult",
    "DecodeResult",
]

_MASK32 = 0xFFFFFFFF


# ---------------------------------------------------------------------------
# Philox4x32-10 counter-based generator.
# Salmon, Moraes, Dror, Shaw, "Parallel Random Numbers: As Easy as 1, 2, 3",
# SC'11, Section 5 (Philox): the round is two 32x32->64 multiplications by
# the constants below, the high halves XORed with the other two counter words
# and the key, followed by a Weyl increment of the key between rounds.
# ---------------------------------------------------------------------------
_PHILOX_M0 = np.uint64(0xD2511F53)
_PHILOX_M1 = np.uint64(0xCD9E8D57)
_PHILOX_W0 = 0x9E3779B9
_PHILOX_W1 = 0xBB67AE85


def philox4x32_10(counter, key):
    """Philox4x32 with 10 rounds.

    counter: four equally shaped arrays (or ints) of 32-bit words
    (c0, c1, c2, c3); key: (k0, k1).  Returns a uint32 array of shape
    (4, ...) holding the four output words.
    """
    c = [np.asarray(w, dtype=np.uint64) & np.uint64(_MASK32) for w in counter]
    c0, c1, c2, c3 = np.broadcast_arrays(*c)
    c0, c1, c2, c3 = (x.copy() for x in (c0, c1, c2, c3))
    k0 = int(key[0]) & _MASK32
    k1 = int(key[1]) & _MASK32
    m32 = np.uint64(_MASK32)
    s32 = np.uint64(32)
    for rnd in range(10):
        if rnd > 0:
            k0 = (k0 + _PHILOX_W0) & _MASK32
            k1 = (k1 + _PHILOX_W1) & _MASK32
        p0 = _PHILOX_M0 * c0  # < 2^64: exact in uint64
        p1 = _PHILOX_M1 * c2
        hi0, lo0 = p0 >> s32, p0 & m32
        hi1, lo1 = p1 >> s32, p1 & m32
        c0, c1, c2, c3 = (hi1 ^ c1 ^ np.uint64(k0), lo1,
                          hi0 ^ c3 ^ np.uint64(k1), lo0)
    return np.stack([c0, c1, c2, c3]).astype(np.uint32)


def philox_uniforms(seed: int, layer: int, b: int, kvh: int, n: int):
    """Uniforms u_i in [0, 1) for tokens i = 0..n-1 of one (layer, b, kvh) unit.

    Poisson sampling (Section 3.3) needs one independent Bernoulli(pi_i) draw
    per tail token.  One Philox4x32-10 call serves four consecutive tokens:
    key = (seed & 0xffffffff, seed >> 32), counter = (i // 4, kvh, layer, b),
    and token i takes output word i % 4.  u = (word >> 8) * 2^-24 is exact in
    float32 and float64.  Returns (u as float64, the raw words as uint32).
    """
    i = np.arange(n, dtype=np.uint64)
    out = philox4x32_10((i >> np.uint64(2), kvh, layer, b),
                        (seed & _MASK32, (seed >> 32) & _MASK32))
    words = out[(i & np.uint64(3)).astype(np.intp), np.arange(n)]
    u = (words >> np.uint32(8)).astype(np.float64) * 2.0 ** -24
    return u, words


# ---------------------------------------------------------------------------
# Section 3.1, Eq. (1): full-cache attention output of one head.
# ---------------------------------------------------------------------------
def full_attention(q, K, V):
    """y = sum_i a_i v_i / sum_i a_i with a_i = exp(q . k_i / sqrt(d))  (Eq. 1).

    q: (d,) or (G, d); K, V: (n, d).  Returns float64 of q's leading shape + (d,).
    The max logit is subtracted before exponentiating (it cancels in the ratio).
    """
    q = np.asarray(q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    d = K.shape[-1]
    logits = (q @ K.T) / math.sqrt(d)
    a = np.exp(logits - logits.max(axis=-1, keepdims=True))
    return (a @ V) / a.sum(axis=-1, keepdims=True)


# ---------------------------------------------------------------------------
# Appendix B (harness): importance scores from accumulated attention.
# ---------------------------------------------------------------------------
def accumulated_attention_scores(q_obs, K):
    """s_j = sum_r softmax_j(q_r . K^T / sqrt(d)).

    The harness scores each cached token by the attention mass it receives
    from a set of observation queries (H2O-style accumulated attention).  For
    grouped-query attention the rows r run over every observation position
    of every query head of the KV head's group.  q_obs: (R, d); K: (N, d).
    """
    q_obs = np.asarray(q_obs, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    d = K.shape[-1]
    logits = (q_obs @ K.T) / math.sqrt(d)
    p = np.exp(logits - logits.max(axis=1, keepdims=True))
    p /= p.sum(axis=1, keepdims=True)
    return p.sum(axis=0)


# ---------------------------------------------------------------------------
# Section 3.3 and Appendix B: the certainty set A.
# ---------------------------------------------------------------------------
def certainty_set(scores, n_sink: int, n_recent: int, k_head: int):
    """Certainty set A = protected positions U top-k_head unprotected tokens.

    Protected: the first ``n_sink`` positions (attention sinks) and the last
    ``n_recent`` positions (recency window); they are never evicted.  The
    score top slice is the ``k_head`` unprotected tokens with the largest
    score, equal scores going to the lower index.  When the windows overlap
    (short contexts) their union is taken.

    Returns (certain mask, top-k mask), both bool arrays of length N.
    """
    s = np.asarray(scores, dtype=np.float64)
    n = s.shape[0]
    protected = np.zeros(n, dtype=bool)
    protected[: min(n_sink, n)] = True
    protected[max(n - n_recent, 0):] = True
    cand = np.flatnonzero(~protected)
    k = min(max(k_head, 0), cand.size)
    # lexsort: last key is primary -> score descending, then index ascending
    order = np.lexsort((cand, -s[cand]))
    top = np.zeros(n, dtype=bool)
    top[cand[order[:k]]] = True
    return protected | top, top


def tail_budget(budget_tokens: int, n_certain: int, n_tail: int) -> int:
    """Expected tail size m = B_t - |A|, clamped to [0, |T|].

    The budget counts every retained token (certainty layer plus the expected
    Poisson tail), the "same budget accounting" as the deterministic arms.
    """
    return int(min(max(budget_tokens - n_certain, 0), n_tail))


# ---------------------------------------------------------------------------
# Section 3.3, Eq. (2): inclusion probabilities on the tail T = C \ A.
# ---------------------------------------------------------------------------
def inclusion_probabilities(scores, certain, budget_tokens: int, eps: float,
                            iters: int = 200):
    """pi_i = 1 on A; on T,  pi_i = clip(c * s_i, eps, 1)  with  sum_T pi_i = m.

    Eq. (2) normalises the tail scores to the tail budget m and clips to
    [eps, 1]; tokens whose allocation hits the upper clip join the certainty
    layer.  Renormalising the remaining tail after moving them is the fixed
    point  sum_T clip(c s_i, eps, 1) = m  in one scalar c, which is found here
    by bisection on log c for ``iters`` steps (200 in float64 is converged).
    Scores <= 0 sit at the floor eps.  Edge cases: m <= eps |T| gives pi = eps
    on all of T (c = 0); a budget above what positive scores can absorb gives
    pi = 1 on every positive-score tail token.

    Returns (pi float64[N], c, m).
    """
    s = np.asarray(scores, dtype=np.float64)
    certain = np.asarray(certain, dtype=bool)
    pi = np.ones(s.shape[0], dtype=np.float64)
    tail = ~certain
    sT = s[tail]
    nT = sT.size
    m = tail_budget(budget_tokens, int(certain.sum()), nT)
    if nT == 0:
        return pi, 0.0, m

    def g(c):
        return np.clip(c * sT, eps, 1.0).sum()

    pos = sT > 0
    n_pos = int(pos.sum())
    if m <= eps * nT:
        c = 0.0
        piT = np.full(nT, eps)
    elif m >= n_pos + eps * (nT - n_pos):
        c = math.inf
        piT = np.where(pos, 1.0, eps)
    else:
        lo = math.log(eps / sT.max())          # g(e^lo) = eps |T| <= m
        hi = math.log(1.0 / sT[pos].min())     # g(e^hi) = n_pos + eps (nT - n_pos) >= m
        for _ in range(iters):
            mid = 0.5 * (lo + hi)
            if g(math.exp(mid)) < m:
                lo = mid
            else:
                hi = mid
        c = math.exp(0.5 * (lo + hi))
        piT = np.clip(c * sT, eps, 1.0)
    pi[tail] = piT
    return pi, c, m


def inclusion_probabilities_one_shot(scores, certain, budget_tokens: int, eps: float):
    """Eq. (2) taken literally: pi_i = clip(m s_i / sum_T s_j, eps, 1) on T.

    Equal to ``inclusion_probabilities`` whenever no tail token clips; kept
    as the alternative reading of Eq. (2).
    """
    s = np.asarray(scores, dtype=np.float64)
    certain = np.asarray(certain, dtype=bool)
    pi = np.ones(s.shape[0], dtype=np.float64)
    tail = ~certain
    sT = s[tail]
    m = tail_budget(budget_tokens, int(certain.sum()), sT.size)
    if sT.size:
        pi[tail] = np.clip(m * sT / sT.sum(), eps, 1.0)
    return pi


# ---------------------------------------------------------------------------
# Section 3.3 / Appendix B: Poisson sampling of the tail and compaction.
# ---------------------------------------------------------------------------
def poisson_keep(pi, u):
    """Independent Bernoulli(pi_i) retention: keep_i = (u_i < pi_i).

    pi_i = 1 (certainty set) always keeps since u < 1.  The comparison is
    made against pi rounded to float32, the precision the device decides in.
    """
    pi32 = np.asarray(pi, dtype=np.float64).astype(np.float32).astype(np.float64)
    return np.asarray(u, dtype=np.float64) < pi32


def compact(K, V, keep, pi, capacity: int):
    """Retained set S in increasing token order plus one scalar per token.

    Section 3.3: the output on S needs only the retained pairs and
    log(1/pi_i) ("one extra scalar per retained tail token"), 0 on A.
    Rows beyond ``capacity`` are dropped; ``n_kept`` is the true count.
    Returns (K_c, V_c, logw_c float64, idx_c int64, n_kept).
    """
    idx = np.flatnonzero(np.asarray(keep, dtype=bool))
    n_kept = int(idx.size)
    idx = idx[:capacity]
    logw = -np.log(np.asarray(pi, dtype=np.float64)[idx])
    return np.asarray(K)[idx], np.asarray(V)[idx], logw, idx, n_kept


@dataclass
class EvictResult:
    certain: np.ndarray      # bool [N]   certainty set A
    topk: np.ndarray         # bool [N]   score top slice
    pi: np.ndarray           # f64  [N]   inclusion probabilities
    c: float                 # Eq. (2) scale
    m: int                   # expected tail size
    u: np.ndarray            # f64  [N]   uniforms
    x0: np.ndarray           # u32  [N]   raw Philox words
    keep: np.ndarray         # bool [N]
    idx: np.ndarray          # int  [min(n_kept, cap)]
    logw: np.ndarray         # f64  [min(n_kept, cap)]  log(1/pi)
    K_c: np.ndarray
    V_c: np.ndarray
    n_kept: int


def evict_unit(K, V, scores, *, n_sink: int, n_recent: int, k_head: int,
               budget_tokens: int, eps: float, seed: int, layer: int, b: int,
               kvh: int, capacity: int, bisect_iters: int = 200) -> EvictResult:
    """One (layer, batch row, KV head) unit through the eviction step.

    Order as in Section 3.3 / Appendix B: certainty set, Eq. (2) probabilities
    on the tail, Poisson draw, compaction with log(1/pi).
    """
    scores = np.asarray(scores)
    n = scores.shape[0]
    certain, topk = certainty_set(scores, n_sink, n_recent, k_head)
    pi, c, m = inclusion_probabilities(scores, certain, budget_tokens, eps, bisect_iters)
    u, x0 = philox_uniforms(seed, layer, b, kvh, n)
    keep = poisson_keep(pi, u)
    K_c, V_c, logw, idx, n_kept = compact(K, V, keep, pi, capacity)
    return EvictResult(certain, topk, pi, c, m, u, x0, keep, idx, logw, K_c, V_c, n_kept)


# ---------------------------------------------------------------------------
# Section 3.3 Eq. (3), Theorem 2 and Section 3.4 Eq. (4): certified decode.
# ---------------------------------------------------------------------------
@dataclass
class DecodeResult:
    y: np.ndarray        # [G, d]  Hajek output
    lse: np.ndarray      # [G]     log N_hat
    var: np.ndarray      # [G]     V_hat
    b_exact: np.ndarray  # [G]     range term, Eq. (4) definition
    b_bound: np.ndarray  # [G]     one-pass upper bound on the range term
    r_exact: np.ndarray  # [G]     radius with b_exact
    r_bound: np.ndarray  # [G]     radius with b_bound


def certificate_radius(var, b, y_norm, delta: float, eps0: float):
    """Eq. (4): r = (sqrt(2 V log(1/delta)) + b log(1/delta)) / (||y_hat|| + eps0)."""
    L = math.log(1.0 / delta)
    return (np.sqrt(2.0 * np.asarray(var) * L) + np.asarray(b) * L) / (np.asarray(y_norm) + eps0)


def hajek_decode(q, K_c, V_c, logw_c, delta: float = 0.1, eps0: float = 1e-9) -> DecodeResult:
    """Hajek attention over the retained set and its certificate, per query head.

    q: (G, d) query heads sharing the KV head; K_c, V_c: (n, d) retained
    rows; logw_c: (n,) = log(1/pi_i) (0 on the certainty set).

    * Eq. (3): y_hat = sum_S (a_i/pi_i) v_i / sum_S a_i/pi_i, obtained by adding
      log(1/pi_i) to the logit q.k_i/sqrt(d) and normalising (the softmax does
      the renormalisation).  N_hat = sum_S a_i/pi_i, reported as lse = log N_hat.
    * Theorem 2: V_hat = N_hat^-2 sum_{S cap T} (1-pi_i)/pi_i^2 a_i^2 ||v_i - y_hat||^2.
      With w_i = a_i/pi_i this is sum (1-pi_i) w_i^2 ||v_i - y_hat||^2 / N_hat^2;
      tokens with pi_i = 1 (the certainty set) contribute 0 through (1 - pi_i).
    * Eq. (4): b_t = max_{S cap T} sqrt((1-pi_i)/pi_i^2) a_i ||v_i - y_hat|| / N_hat
      (``b_exact``), and the one-pass bound about the reference row
      c = V_c[(n - 1) // 2] (``b_bound``):
      (max sqrt(1-pi) w ||v - c|| + ||y_hat - c|| max sqrt(1-pi) w) / N_hat,
      which is >= b_exact because ||v_i - y_hat|| <= ||v_i - c|| + ||c - y_hat||.
      Both forms are unchanged by a common shift of all values (Eq. 4's b_t
      depends on the values only through v_i - y_hat).

    An empty retained set gives y = 0, lse = -inf and a zero certificate.
    """
    q = np.atleast_2d(np.asarray(q, dtype=np.float64))
    K_c = np.asarray(K_c, dtype=np.float64)
    V_c = np.asarray(V_c, dtype=np.float64)
    logw = np.asarray(logw_c, dtype=np.float64)
    G, d = q.shape
    n = K_c.shape[0]
    if n == 0:
        z = np.zeros(G)
        return DecodeResult(np.zeros((G, d)), np.full(G, -np.inf), z, z.copy(), z.copy(),
                            z.copy(), z.copy())
    one_minus_pi = -np.expm1(-logw)
    c = V_c[(n - 1) // 2]                               # reference row of the bound
    ys, lses, vs, bes, bbs = [], [], [], [], []
    for h in range(G):
        logits = (K_c @ q[h]) / math.sqrt(d) + logw     # log(a_i / pi_i)
        M = logits.max()
        w = np.exp(logits - M)                          # (a_i/pi_i) e^-M
        l = w.sum()                                     # N_hat e^-M
        y = (w @ V_c) / l
        p = w / l                                       # (a_i/pi_i) / N_hat
        dist = np.linalg.norm(V_c - y, axis=1)          # ||v_i - y_hat||
        t = np.sqrt(one_minus_pi) * p * dist            # per-token range term
        var = np.sum(one_minus_pi * p * p * dist * dist)
        b_exact = t.max()
        s = np.sqrt(one_minus_pi) * p
        b_bound = np.max(s * np.linalg.norm(V_c - c, axis=1)) + np.linalg.norm(y - c) * np.max(s)
        ys.append(y)
        lses.append(M + math.log(l))
        vs.append(var)
        bes.append(b_exact)
        bbs.append(b_bound)
    y = np.array(ys)
    var = np.array(vs)
    b_exact = np.array(bes)
    b_bound = np.array(bbs)
    yn = np.linalg.norm(y, axis=1)
    return DecodeResult(y, np.array(lses), var, b_exact, b_bound,
                        certificate_radius(var, b_exact, yn, delta, eps0),
                        certificate_radius(var, b_bound, yn, delta, eps0))


# ---------------------------------------------------------------------------
# Deployed certificate (Section 5 experimental setup and its appendix): the
# radius of Eq. (4) at delta = 0.1 on every fourth query head of every layer
# during the first six decode steps, averaged, then maximized over the steps;
# the label-free red-flag rule is cert >= tau = 1.
# ---------------------------------------------------------------------------
def deployed_certificate(radii, head_stride=4):
    """radii: [T, L, B, Hq] radii of T probed steps.  Returns (cert [B],
    step_means [T, B]): the average over layers and heads h % head_stride == 0
    at each step, and its maximum over the steps."""
    r = np.asarray(radii, dtype=np.float64)
    step_means = r[:, :, :, ::head_stride].mean(axis=(1, 3))
    return step_means.max(axis=0), step_means


def red_flag(cert, tau=1.0):
    """The label-free rule: raise a sequence whose certificate reaches tau."""
    return np.asarray(cert) >= tau


# ---------------------------------------------------------------------------
# Decode-time growth and re-eviction of a compact cache.  A token generated
# after an eviction enters with pi = 1.  Redrawing the tail every T_r steps
# (the block schedule of the anytime argument, Section 4 and its appendix)
# evicts the resident cache again; a token kept by both rounds has inclusion
# probability pi_1 pi_2 (two independent Poisson designs), so log(1/pi) adds.
# ---------------------------------------------------------------------------
def append_token(K_c, V_c, logw_c, idx_c, k_new, v_new, position):
    """Resident cache of one unit plus one new token with log(1/pi) = 0."""
    return (np.concatenate([K_c, np.asarray(k_new)[None]], 0),
            np.concatenate([V_c, np.asarray(v_new)[None]], 0),
            np.concatenate([logw_c, [0.0]]), np.concatenate([idx_c, [position]]).astype(np.int64))


@dataclass
class ReevictResult:
    inner: EvictResult      # the second-round eviction over the resident rows
    idx: np.ndarray         # original token positions of the kept rows
    logw: np.ndarray        # log(1/pi_1) + log(1/pi_2) of the kept rows
    K_c: np.ndarray
    V_c: np.ndarray
    n_kept: int


def reevict_unit(K_c, V_c, logw_c, idx_c, scores, *, n_sink, n_recent, k_head, budget_tokens,
                 eps, seed, layer, b, kvh, capacity, bisect_iters=200) -> ReevictResult:
    """Evict the resident rows of one unit again (they are the new context, in
    cache order) and compose the two designs."""
    r = evict_unit(K_c, V_c, scores, n_sink=n_sink, n_recent=n_recent, k_head=k_head,
                   budget_tokens=budget_tokens, eps=eps, seed=seed, layer=layer, b=b, kvh=kvh,
                   capacity=capacity, bisect_iters=bisect_iters)
    logw_c = np.asarray(logw_c, dtype=np.float64)
    idx_c = np.asarray(idx_c)
    return ReevictResult(r, idx_c[r.idx], logw_c[r.idx] + r.logw, r.K_c, r.V_c, r.n_kept)


# ---------------------------------------------------------------------------
# Fixed-size systematic sampling at the same inclusion probabilities (Hajek
# 1964; the exact-budget variant the paper measures in Section 5): the tail in
# token order, cumulative sums C_i of pi, one uniform u per unit; token i is
# kept when an integer lies in (C_{i-1} - u, C_i - u].  Each pi_i is first
# rounded to the nearest multiple of 2^-32 and the sums are exact integers, so
# every implementation takes the same decision.  The uniform is word 0 of
# Philox4x32-10 at counter (2^32 - 1, kvh, layer, b), u = (x >> 8) 2^-24.
# ---------------------------------------------------------------------------
SYSTEMATIC_SCALE = 1 << 32


def systematic_uniform(seed: int, layer: int, b: int, kvh: int) -> int:
    """The unit's uniform, as an integer multiple of 2^-24."""
    key = (seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF)
    w = philox4x32_10((0xFFFFFFFF, kvh & 0xFFFFFFFF, layer & 0xFFFFFFFF, b & 0xFFFFFFFF), key)
    return int(w[0]) >> 8


def systematic_keep(pi, certain, u24: int):
    """Kept mask of the systematic design; pi is rounded to float32 first (the
    precision the probabilities are stored in), then to units of 2^-32."""
    pi32 = np.asarray(pi, dtype=np.float32).astype(np.float64)
    units = np.rint(pi32 * SYSTEMATIC_SCALE).astype(np.int64)
    u = u24 << 8
    keep = np.asarray(certain, dtype=bool).copy()
    C = 0
    for i in np.flatnonzero(~np.asarray(certain, dtype=bool)):
        Cp = C
        C += int(units[i])
        if (C - u) // SYSTEMATIC_SCALE != (Cp - u) // SYSTEMATIC_SCALE:
            keep[i] = True
    return keep


def evict_unit_systematic(K, V, scores, *, n_sink, n_recent, k_head, budget_tokens, eps, seed,
                          layer, b, kvh, capacity, bisect_iters=200):
    """evict_unit with the systematic tail design."""
    scores = np.asarray(scores)
    certain, topk = certainty_set(scores, n_sink, n_recent, k_head)
    pi, c, m = inclusion_probabilities(scores, certain, budget_tokens, eps, bisect_iters)
    u24 = systematic_uniform(seed, layer, b, kvh)
    keep = systematic_keep(pi, certain, u24)
    K_c, V_c, logw, idx, n_kept = compact(K, V, keep, pi, capacity)
    return EvictResult(certain, topk, pi, c, m, np.full(len(scores), u24 * 2.0 ** -24),
                       np.zeros(len(scores), dtype=np.uint32), keep, idx, logw, K_c, V_c, n_kept)


# ---------------------------------------------------------------------------
# Observation queries (Appendix, experimental details) and per-token variance
# contributions (Theorem 2's terms; Section 5's fine-grained probe).
# ---------------------------------------------------------------------------
def gather_queries(Q, positions, n_kv_heads):
    """Q [B, Hq, Nq, d] -> q_obs [B, Hkv, G*P, d], row g*P + p = Q[b, kvh*G + g, positions[p]]."""
    Q = np.asarray(Q)
    B, Hq, _, d = Q.shape
    G = Hq // n_kv_heads
    pos = np.asarray(positions)
    sel = Q[:, :, pos, :]                      # [B, Hq, P, d]
    return sel.reshape(B, n_kv_heads, G * len(pos), d)


def variance_contributions(q, K_c, V_c, logw_c):
    """[G, n] terms (1 - pi_i) p_i^2 ||v_i - y_hat||^2 of V_hat (Theorem 2) for
    the query heads q [G, d] over one unit's retained rows."""
    q = np.atleast_2d(np.asarray(q, dtype=np.float64))
    K_c = np.asarray(K_c, dtype=np.float64)
    V_c = np.asarray(V_c, dtype=np.float64)
    logw = np.asarray(logw_c, dtype=np.float64)
    n = K_c.shape[0]
    if n == 0:
        return np.zeros((q.shape[0], 0))
    d = K_c.shape[1]
    x = q @ K_c.T / math.sqrt(d) + logw[None, :]
    p = np.exp(x - scipy_logsumexp(x))
    y = p @ V_c
    omp = -np.expm1(-logw)
    dist = ((V_c[None, :, :] - y[:, None, :]) ** 2).sum(-1)
    return omp[None, :] * p ** 2 * dist


def scipy_logsumexp(x):
    m = x.max(axis=1, keepdims=True)
    return m + np.log(np.exp(x - m).sum(axis=1, keepdims=True))


def block_scores(contrib, idx_c, block, n_blocks):
    """Sum over heads and retained rows of the contributions, per block of
    `block` original positions: contrib [G, n], idx_c [n] -> [n_blocks]."""
    out = np.zeros(n_blocks)
    tot = np.asarray(contrib).sum(axis=0)
    for i, t in enumerate(np.asarray(idx_c)):
        out[int(t) // block] += tot[i]
    return out
