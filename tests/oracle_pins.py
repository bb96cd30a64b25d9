"""Pins that tie the CPU oracle to what the paper and the mathematics fix.

Each ``pin_*`` function raises AssertionError when the oracle disagrees with
a closed form, a library routine, a value the paper prints, an invariant or a
brute-force recomputation.  ``test_oracle.py`` runs them on the oracle as it
is; ``test_oracle_mutants.py`` plants plausible mistakes in the oracle and
checks that at least one pin catches each.
"""
from __future__ import annotations

import json
import math
import os
from fractions import Fraction

import numpy as np
import scipy.spatial.distance
import scipy.stats

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_budgets.json")


def _rng(seed):
    return np.random.default_rng(seed)


def _bf16_round(a):
    """Round float64 values to bf16 (round-to-nearest-even) and back, so test
    rows hold values exactly representable in the CUDA path's input type."""
    f = np.asarray(a, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    u = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    return u.astype(np.uint32).view(np.float32).astype(np.float64)


# ---------------------------------------------------------------- Eq. 3-4
def pin_h2_equal_magnitudes():
    """|x_j| all equal (random signs): p is uniform, H2 = log D."""
    for d in (1, 7, 64, 1024, 4096):
        signs = _rng(d).choice([-1.0, 1.0], size=(3, d))
        x = signs * np.array([[0.375], [5.0], [1e-3]])
        assert np.allclose(oracle.renyi2_entropy(x), math.log(d), rtol=0, atol=1e-12)


def pin_h2_one_hot_and_k_hot():
    """One non-zero channel: H2 = 0; k equal non-zeros: H2 = log k."""
    d = 256
    x = np.zeros((4, d))
    x[0, 17] = -3.5
    x[1, [1, 2]] = [2.0, -2.0]
    x[2, :10] = 0.75
    x[3, ::2] = -1.25
    h = oracle.renyi2_entropy(x)
    assert np.allclose(h, [0.0, math.log(2), math.log(10), math.log(d // 2)], rtol=0, atol=1e-12)


def pin_h2_two_component():
    """Row (3, -1, 0, 0): p = (3/4, 1/4), sum p^2 = 10/16, H2 = log(1.6)."""
    h = oracle.renyi2_entropy(np.array([[3.0, -1.0, 0.0, 0.0], [0.0, 0.0, 1.0, 3.0]]))
    assert np.allclose(h, math.log(1.6), rtol=0, atol=1e-14)


def pin_h2_bounds_and_shannon():
    """0 <= H2 <= H1 <= log D, with H1 the Shannon entropy of p (scipy);
    Renyi entropies do not increase with their order."""
    x = _rng(1).standard_normal((64, 300)) * _rng(2).exponential(size=(64, 1))
    x[5, 7] *= 50
    h2 = oracle.renyi2_entropy(x)
    p = np.abs(x) / np.abs(x).sum(axis=1, keepdims=True)
    h1 = scipy.stats.entropy(p, axis=1)
    assert (h2 >= -1e-15).all() and (h2 <= h1 + 1e-12).all() and (h1 <= math.log(300) + 1e-12).all()
    # and strictly below Shannon for a non-uniform distribution
    assert (h2 < h1 - 1e-6).all()


def pin_h2_invariances():
    """Exact invariance under scaling by a power of two and sign flips;
    invariance under a channel permutation up to rounding."""
    x = _bf16_round(_rng(3).standard_normal((16, 512)))
    h = oracle.renyi2_entropy(x)
    assert np.array_equal(oracle.renyi2_entropy(x * 2.0 ** -9), h)
    assert np.array_equal(oracle.renyi2_entropy(-x), h)
    perm = _rng(4).permutation(512)
    assert np.allclose(oracle.renyi2_entropy(x[:, perm]), h, rtol=0, atol=1e-13)


def pin_h2_row_independence():
    """Each row's score depends on that row only, along the channel axis."""
    x = _rng(5).standard_normal((8, 33))
    h = oracle.renyi2_entropy(x)
    for i in range(8):
        assert oracle.renyi2_entropy(x[i:i + 1])[0] == h[i]
    assert not np.allclose(oracle.renyi2_entropy(x[:, :8].T.copy())[:8], h[:8])


# ---------------------------------------------------------------- Eq. 6
def pin_s_matches_scipy_cosine():
    """s = 1 - scipy's cosine distance."""
    a = _rng(6).standard_normal((40, 129))
    b = 0.3 * a + _rng(7).standard_normal((40, 129))
    s = oracle.consistency(a, b)
    ref = np.array([1.0 - scipy.spatial.distance.cosine(a[i], b[i]) for i in range(40)])
    assert np.allclose(s, ref, rtol=0, atol=1e-13)


def pin_s_special_cases():
    """s(x, x) = 1, s(x, -x) = -1, s(x, c x) = 1 for c > 0, orthogonal -> 0,
    |s| <= 1, and s with a zero vector is 0 (reading)."""
    a = _rng(8).standard_normal((5, 64))
    assert np.allclose(oracle.consistency(a, a), 1.0, atol=1e-15)
    assert np.allclose(oracle.consistency(a, -a), -1.0, atol=1e-15)
    assert np.allclose(oracle.consistency(a, 3.5 * a), 1.0, atol=1e-15)
    e = np.eye(64)[:5]
    f = np.eye(64)[5:10]
    assert np.array_equal(oracle.consistency(e, f), np.zeros(5))
    r = oracle.consistency(a, _rng(9).standard_normal((5, 64)))
    assert (np.abs(r) <= 1).all()
    z = np.zeros((1, 64))
    assert oracle.consistency(z, a[:1])[0] == 0.0 and oracle.consistency(a[:1], z)[0] == 0.0


def pin_s_similar_tokens_similar_signal():
    """Section IV-B: similar tokens give similar s.  Perturbing x'' by delta
    moves s by at most 2 ||delta|| / ||x''|| (cosine is Lipschitz)."""
    a = _rng(10).standard_normal((50, 256))
    b = _rng(11).standard_normal((50, 256))
    delta = 1e-3 * _rng(12).standard_normal((50, 256))
    ds = np.abs(oracle.consistency(a, b + delta) - oracle.consistency(a, b))
    bound = 2 * np.linalg.norm(delta, axis=1) / np.linalg.norm(b, axis=1)
    assert (ds <= bound + 1e-15).all()
    assert ds.max() > 0


# ---------------------------------------------------------------- budgets
def pin_budgets_paper_values():
    """Budgets the paper prints (tests/golden/paper_budgets.json)."""
    g = json.load(open(GOLDEN))
    for e in g["split"]:
        assert oracle.budget_split(e["k"], (1, 3)) == (e["k1"], e["k2"]), e["cite"]
    for e in g["retention"]:
        got = [oracle.budget_from_ratio(e["n"], tuple(r)) for r in e["ratios"]]
        assert got == e["k"], e["cite"]


def pin_budgets_floor_and_stride():
    """K1 = floor(lambda K) by hand, and t = max(1, floor(|X_rem|/K2))."""
    table = {(10, (1, 3)): (3, 7), (64, (1, 3)): (21, 43), (128, (1, 3)): (42, 86),
             (7, (1, 2)): (3, 4), (5, (0, 1)): (0, 5), (5, (1, 1)): (5, 0), (1, (1, 3)): (0, 1)}
    for (k, lam), want in table.items():
        assert oracle.budget_split(k, lam) == want, (k, lam)
    assert [oracle.budget_from_ratio(n, r) for n, r in [(100, (2, 3)), (1000, (1, 9)), (5, (1, 9)), (0, (1, 3))]] == \
        [66, 111, 1, 0]
    assert [oracle.stride(m, k2) for m, k2 in [(555, 43), (512, 128), (3, 3), (2, 5), (2753, 214)]] == \
        [12, 4, 1, 1, 12]


def pin_interval_positions():
    """The text's fixed interval |X_rem| / K2 (Section IV-B) as a real step:
    K2 distinct positions inside X_rem starting at 0; below every cut x of
    the sorted list sit exactly ceil(x K2 / |X_rem|) picks (uniform sampling
    along the list, counted here one position at a time); it is Algorithm 1's
    integer stride whenever K2 divides |X_rem|; hand values for the shapes of
    the configs."""
    rng = _rng(29)
    pairs = [(555, 43), (512, 128), (6011, 523), (2827, 107), (3, 3), (7, 1), (1, 1)]
    pairs += [(int(m), int(rng.integers(1, m + 1))) for m in rng.integers(1, 400, 40)]
    for m, k2 in pairs:
        pos = oracle.pick_positions(m, k2, "interval").tolist()
        assert len(pos) == k2 and pos[0] == 0 and pos[-1] < m, (m, k2)
        assert all(b > a for a, b in zip(pos, pos[1:])), (m, k2)
        picked = set(pos)
        below = 0
        for x in range(m + 1):
            assert below == -(-x * k2 // m), (m, k2, x)
            if x < m and x in picked:
                below += 1
        if m % k2 == 0:
            assert pos == oracle.pick_positions(m, k2, "alg1").tolist(), (m, k2)
    # K = 64 on N = 576: K1 = 21, |X_rem| = 555, K2 = 43 (interval 12.9 vs stride 12);
    # video clips: N = 6272, K = 784: |X_rem| = 6011, K2 = 523 (interval 11.49 vs stride 11)
    assert oracle.pick_positions(555, 43, "interval")[-1] == 542
    assert oracle.pick_positions(555, 43, "alg1")[-1] == 504
    assert oracle.pick_positions(6011, 523, "interval")[-1] == 5999
    assert oracle.pick_positions(6011, 523, "alg1")[-1] == 5742


# ---------------------------------------------------------------- Algorithm 1, brute force
def _brute_select(x, xp, xq, k, lam, mode="alg1"):
    """Independent O(N^2) rank-count implementation with exact rationals.

    Importance: token i is in X_imp when fewer than K1 tokens beat it
    (larger R = L1^2 / S2, or equal R and a lower index).  Diversity: the
    rank of a remaining token among the remaining ones by (s, index) decides
    whether it sits at a stride position."""
    n = len(x)
    k1 = math.floor(Fraction(k * lam[0], lam[1]))
    k2 = k - k1
    fx = [[Fraction(float(v)) for v in row] for row in x]
    r = []
    for row in fx:
        l1 = sum((abs(v) for v in row), Fraction(0))
        s2 = sum((v * v for v in row), Fraction(0))
        r.append(Fraction(1) if l1 == 0 else l1 * l1 / s2)
    beats = lambda j, i: r[j] > r[i] or (r[j] == r[i] and j < i)
    imp = {i for i in range(n) if sum(beats(j, i) for j in range(n) if j != i) < k1}
    rem = [i for i in range(n) if i not in imp]
    sig = {}
    for i in rem:
        a = [Fraction(float(v)) for v in xp[i]]
        b = [Fraction(float(v)) for v in xq[i]]
        p = sum((u * v for u, v in zip(a, b)), Fraction(0))
        aa = sum((u * u for u in a), Fraction(0))
        bb = sum((v * v for v in b), Fraction(0))
        sig[i] = Fraction(0) if aa == 0 or bb == 0 else (1 if p > 0 else -1) * p * p / (aa * bb)
    div = set()
    if k2:
        m = len(rem)
        t = max(1, m // k2)
        for i in rem:
            pos = sum(1 for j in rem if sig[j] < sig[i] or (sig[j] == sig[i] and j < i))
            if mode == "alg1":
                hit = pos % t == 0 and pos // t < k2
            else:  # a sample of the interval m / k2 falls in [pos, pos + 1)
                hit = Fraction((pos + 1) * k2, m).__ceil__() > Fraction(pos * k2, m).__ceil__()
            if hit:
                div.add(i)
    return imp, div


def pin_select_brute_force_tiny():
    """Oracle selection equals the brute force on many tiny random images,
    including ones with duplicated rows (exact ties)."""
    rng = _rng(13)
    for trial in range(60):
        n = int(rng.integers(1, 11))
        d = int(rng.integers(1, 9))
        x = _bf16_round(rng.standard_normal((n, d)) * rng.exponential(size=(n, 1)))
        xp = _bf16_round(rng.standard_normal((n, d)))
        xq = _bf16_round(rng.standard_normal((n, d)))
        if trial % 3 == 0 and n > 2:           # duplicate rows -> exact ties
            x[1] = x[0]
            xp[2] = xp[0]
            xq[2] = xq[0]
        if trial % 5 == 0:
            x[0] = 0.0
        k = int(rng.integers(0, n + 1))
        lam = [(1, 3), (1, 2), (0, 1), (1, 1), (2, 3)][trial % 5]
        k1, _ = oracle.budget_split(k, lam)
        for mode in ("alg1", "interval"):
            got = oracle.select_image(x, xp, xq, k, k1, mode)
            imp, div = _brute_select(x, xp, xq, k, lam, mode)
            assert set(got["imp"].tolist()) == imp, (trial, mode, got["imp"], imp)
            assert set(got["div"].tolist()) == div, (trial, mode, got["div"], div)
            assert got["kept"].tolist() == sorted(imp | div)


# ---------------------------------------------------------------- Algorithm 1, properties
def _small_workload(seed=0, n=300, d=96):
    rng = _rng(seed)
    c = rng.standard_normal((12, d))
    h = c[rng.integers(0, 12, n)] + 0.1 * rng.standard_normal((n, d))
    w1 = rng.standard_normal((16, d)) / math.sqrt(d)
    w2 = rng.standard_normal((d, 16)) / 4
    hp = np.maximum(h @ w1.T, 0) @ w2.T
    return _bf16_round(h + hp), _bf16_round(h), _bf16_round(hp)


def pin_select_properties():
    """|X*| = K, unique indices, X_imp and X_div disjoint, every importance
    token scores at least every remaining token, and the diversity tokens sit
    at stride positions of the ascending s order of X_rem."""
    x, xp, xq = _small_workload()
    n = len(x)
    for k in (1, 30, 64, 100, n):
        k1, k2 = oracle.budget_split(k, (1, 3))
        r = oracle.select_image(x, xp, xq, k, k1)
        kept = r["kept"]
        assert len(kept) == k and len(np.unique(kept)) == k
        assert not set(r["imp"].tolist()) & set(r["div"].tolist())
        rem = np.setdiff1d(np.arange(n), r["imp"])
        if k1 and len(rem):
            assert r["h2"][r["imp"]].min() >= r["h2"][rem].max()
        if k2:
            s_rem = np.sort(r["s"][rem])
            t = max(1, len(rem) // k2)
            assert np.array_equal(np.sort(r["s"][r["div"]]), s_rem[np.arange(k2) * t])


def pin_select_lambda_extremes():
    """lambda = 1 keeps the K highest-entropy tokens; lambda = 0 takes a pure
    stride of floor(N/K) over the ascending s order of all N tokens."""
    x, xp, xq = _small_workload(seed=1)
    n, k = len(x), 40
    r = oracle.select_image(x, xp, xq, k, k)
    h2 = oracle.renyi2_entropy(x)
    assert set(r["kept"].tolist()) == set(np.argsort(-h2, kind="stable")[:k].tolist())
    r0 = oracle.select_image(x, xp, xq, k, 0)
    s = oracle.consistency(xp, xq)
    order = np.argsort(s, kind="stable")
    assert set(r0["kept"].tolist()) == set(order[np.arange(k) * (n // k)].tolist())


def pin_select_permutation_equivariance():
    """Permuting the tokens permutes the selection (no ties in this data)."""
    x, xp, xq = _small_workload(seed=2)
    perm = _rng(14).permutation(len(x))
    a = oracle.select_image(x, xp, xq, 90, 30)["kept"]
    b = oracle.select_image(x[perm], xp[perm], xq[perm], 90, 30)["kept"]
    assert sorted(perm[b].tolist()) == sorted(a.tolist())


def pin_select_exact_ties_by_index():
    """Rows that are channel permutations of each other have exactly equal
    R (Eq. 4) even when float64 rounds their sums differently; the lower
    index must win.  Values span many binades so the sums are inexact."""
    rng = _rng(15)
    base = (rng.standard_normal(200) * np.exp2(rng.integers(-30, 30, 200))).astype(np.float32)
    rows = [base[rng.permutation(200)] for _ in range(12)]
    x = np.array(rows, dtype=np.float64)
    h2 = oracle.renyi2_entropy(x)
    assert len(set(h2.tolist())) > 1, "test data must exercise unequal float64 keys"
    r = oracle.select_image(x, x, x[::-1].copy(), 5, 5)
    assert r["imp"].tolist() == [0, 1, 2, 3, 4]
    # s ties: (x', x'') pairs permuted by the same channel permutation have
    # exactly equal P, A and B, so exactly equal s
    perms = [rng.permutation(200) for _ in range(12)]
    other = np.roll(base, 3)
    xp2 = np.array([base[p] for p in perms], dtype=np.float64)
    xq2 = np.array([other[p] for p in perms], dtype=np.float64)
    assert len(set(oracle.consistency(xp2, xq2).tolist())) > 1
    r2 = oracle.select_image(x, xp2, xq2, 4, 0)
    assert r2["rem_sorted"].tolist() == list(range(12))


def pin_select_near_ties_resolved_exactly():
    """Keys that differ by far less than float64 resolves: a uniform row has
    the maximal R = D, a row perturbed by 2^-40 has a smaller R, so the
    uniform row must win importance although it has the higher index.  Same
    for s: x'' = x' gives s = 1 exactly, a 2^-40 perturbation gives s < 1,
    which must sort first although float64 cannot separate the two."""
    d = 64
    x = np.ones((2, d))
    x[0, 5] += 2.0 ** -40
    assert oracle.select_image(x, x, x, 1, 1)["imp"].tolist() == [1]
    xp = np.tile(np.linspace(0.5, 1.5, d), (2, 1))
    xq = xp.copy()
    xq[1, 3] += 2.0 ** -40
    s = oracle.consistency(xp, xq)
    assert abs(s[0] - s[1]) < oracle.NEAR_TIE
    assert oracle.select_image(x, xp, xq, 2, 0)["rem_sorted"].tolist() == [1, 0]
    # negative side: x'' = -x' gives s = -1 exactly, the perturbed row lies above
    assert oracle.select_image(x, xp, -xq[::-1].copy(), 2, 0)["rem_sorted"].tolist() == [1, 0]


def pin_select_nonfinite_and_zero_rows():
    """Readings: a non-finite x ranks last by importance; a non-finite x' or
    x'' sorts last by s; an all-zero x has H2 = 0."""
    x, xp, xq = _small_workload(seed=3, n=40, d=32)
    x[3, 5] = np.nan
    x[7] = 0.0
    xq[9, 0] = np.inf
    h2 = oracle.renyi2_entropy(x)
    assert h2[3] == -np.inf and h2[7] == 0.0
    r = oracle.select_image(x, xp, xq, 40, 40)
    assert r["imp"][-1] == 3
    r = oracle.select_image(x, xp, xq, 10, 0)
    assert r["rem_sorted"][-1] == 9


ALL_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_")]
