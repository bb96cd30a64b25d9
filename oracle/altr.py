"""CPU oracle for the ALTR token-reduction path (arxiv 2607.13500, Section IV).

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import this
package: only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU
baseline / reference arm use it.  It shares no code with the CUDA path.

Plain, slow and obviously correct: numpy in float64 on the stored (already
rounded) inputs, which convert to float64 exactly from bf16 and fp32.

What it computes (Section IV, Eq. 3-7; the selection in the order the
paper's Algorithm 1 gives it):

* the budget split K1 = floor(lambda K), K2 = K - K1 (Eq. 7);
* per token, the channel-magnitude distribution p_ij = |x_ij| / sum_k |x_ik|
  (Eq. 3) and its Renyi-2 entropy H2(x_i) = -log sum_j p_ij^2 (Eq. 4);
* Stage I: X_imp, the K1 tokens with the highest H2 (Section IV-A), and
  X_rem, the tokens left over;
* per token, the consistency signal s_i = x'_i . x''_i / (||x'_i|| ||x''_i||)
  (Eq. 6), with x', x'' the final-layer MLP input and output (Eq. 5);
* Stage II: X_rem sorted by s ascending and K2 tokens taken along that order
  at the stride t = max(1, floor(|X_rem| / K2)), i.e. sorted positions
  0, t, 2t, ... (Algorithm 1's 1-based 1, 1+t, ...), or, as the text of
  Section IV-B states it, at the fixed real interval |X_rem| / K2:
  positions floor(j |X_rem| / K2), j < K2 (Section IV-B);
* X* = X_imp union X_div, returned in ascending token order (Eq. 7).

Readings of points the paper leaves open:

* ties (top-K and sort) go to the lower token index;
* an all-zero row has H2 = 0 (p is undefined; 0 is the one-hot value);
  a row whose x' or x'' is all zero has s = 0;
* a row whose x holds a non-finite value ranks last by importance
  (H2 = -inf); one whose x' or x'' holds one sorts last by s (s = +inf);
* lambda is a rational lam_num/lam_den, default 1/3 (the paper's split of
  K = 192 into 64 importance and 128 diversity tokens, Section V-C).

Exact ordering.  float64 fixes H2 and s to within ~1e-12 (D <= 16384), so the
fp64 order is the true order except among keys closer than that.  Such
near-tie runs are re-ordered by exact rational keys built with ``fractions``
from the exact input values: H2 is increasing in R = L1^2 / S2
(H2 = log R since sum p^2 = S2 / L1^2), and s has the sign of P and is
increasing in sign(P) P^2 / (A B), with L1 = sum|x|, S2 = sum x^2,
P = sum x' x'', A = sum x'^2, B = sum x''^2.  The result is therefore the
selection defined by the real-valued keys of Eq. 4 and Eq. 6 with the
index tie-break, independent of any summation order.
"""
from __future__ import annotations

from fractions import Fraction

import numpy as np

# Keys closer than this (absolute, on H2 and on s) are ordered exactly.  It is
# two orders of magnitude above the float64 error of either key for D <= 16384.
NEAR_TIE = 1e-10


# --------------------------------------------------------------------------
# Budgets (Eq. 7)
# --------------------------------------------------------------------------
def budget_split(k: int, lam=(1, 3)):
    """K1 = floor(lambda K), K2 = K - K1 with lambda = lam[0] / lam[1]."""
    num, den = lam
    if not (0 <= num <= den and den > 0):
        raise ValueError("lambda must lie in [0, 1]")
    k1 = (k * num) // den
    return k1, k - k1


def budget_from_ratio(n: int, ratio):
    """K = floor(N num / den), at least 1 for a non-empty image (retention
    ratio readings of Section V-B: 1/3, 2/9, 1/9 of the tokens)."""
    num, den = ratio
    if n == 0:
        return 0
    return max(1, (n * num) // den)


def stride(n_rem: int, k2: int) -> int:
    """t = max(1, floor(|X_rem| / K2)) (Algorithm 1)."""
    return max(1, n_rem // k2)


def pick_positions(n_rem: int, k2: int, mode: str = "alg1") -> np.ndarray:
    """0-based positions of X_div along X_rem sorted by s.

    ``"alg1"``: Algorithm 1's integer stride, 0, t, 2t, ..., (K2 - 1) t.
    ``"interval"``: the fixed interval (N - |X_imp|) / K2 = |X_rem| / K2 of
    Section IV-B taken as a real number: sample j sits at the real position
    j |X_rem| / K2 and takes the sorted token at its floor, j < K2.
    """
    if k2 == 0:
        return np.zeros(0, dtype=np.int64)
    j = np.arange(k2, dtype=np.int64)
    if mode == "alg1":
        return j * stride(n_rem, k2)
    if mode == "interval":
        return (j * n_rem) // k2
    raise ValueError(f"unknown stride mode {mode!r}")


# --------------------------------------------------------------------------
# Importance: Renyi-2 entropy (Eq. 3, Eq. 4)
# --------------------------------------------------------------------------
def renyi2_entropy(x: np.ndarray) -> np.ndarray:
    """H2 per row of ``x`` [N, D] following Eq. 3 then Eq. 4, in float64."""
    x = np.asarray(x, dtype=np.float64)
    finite = np.isfinite(x).all(axis=1)
    a = np.abs(np.where(np.isfinite(x), x, 0.0))
    l1 = a.sum(axis=1)                                   # sum_k |x_ik|
    safe = np.where(l1 > 0, l1, 1.0)
    p = a / safe[:, None]                                 # Eq. 3
    h2 = -np.log(np.where(l1 > 0, (p * p).sum(axis=1), 1.0))  # Eq. 4
    h2 = np.where(l1 > 0, h2, 0.0)                        # all-zero row reading
    return np.where(finite, h2, -np.inf)


# --------------------------------------------------------------------------
# Consistency signal (Eq. 6)
# --------------------------------------------------------------------------
def consistency(x_pre: np.ndarray, x_post: np.ndarray) -> np.ndarray:
    """s_i = cos(x'_i, x''_i) per row, float64 (Eq. 6)."""
    xp = np.asarray(x_pre, dtype=np.float64)
    xq = np.asarray(x_post, dtype=np.float64)
    finite = np.isfinite(xp).all(axis=1) & np.isfinite(xq).all(axis=1)
    xp = np.where(np.isfinite(xp), xp, 0.0)
    xq = np.where(np.isfinite(xq), xq, 0.0)
    dot = (xp * xq).sum(axis=1)
    na = np.sqrt((xp * xp).sum(axis=1))
    nb = np.sqrt((xq * xq).sum(axis=1))
    zero = (na == 0) | (nb == 0)
    s = dot / np.where(zero, 1.0, na * nb)
    s = np.where(zero, 0.0, s)
    return np.where(finite, s, np.inf)


# --------------------------------------------------------------------------
# Exact keys (used only to order near-ties)
# --------------------------------------------------------------------------
def _fsum_exact(values) -> Fraction:
    return sum((Fraction(float(v)) for v in values), Fraction(0))


def exact_r(row) -> tuple:
    """Sort key for importance, descending by H2: (class, R) with R = L1^2/S2
    exactly; class 1 marks a non-finite row, which ranks last."""
    row = np.asarray(row, dtype=np.float64)
    if not np.isfinite(row).all():
        return (1, Fraction(0))
    l1 = sum((abs(Fraction(float(v))) for v in row), Fraction(0))
    if l1 == 0:
        return (0, Fraction(1))
    s2 = sum((Fraction(float(v)) ** 2 for v in row), Fraction(0))
    return (0, l1 * l1 / s2)


def exact_sigma(row_pre, row_post) -> tuple:
    """Sort key for consistency, ascending by s: (class, sign(P) P^2/(A B))
    exactly; class 1 marks a non-finite row, which sorts last."""
    a_row = np.asarray(row_pre, dtype=np.float64)
    b_row = np.asarray(row_post, dtype=np.float64)
    if not (np.isfinite(a_row).all() and np.isfinite(b_row).all()):
        return (1, Fraction(0))
    fa = [Fraction(float(v)) for v in a_row]
    fb = [Fraction(float(v)) for v in b_row]
    a = sum((v * v for v in fa), Fraction(0))
    b = sum((v * v for v in fb), Fraction(0))
    if a == 0 or b == 0:
        return (0, Fraction(0))
    p = sum((u * v for u, v in zip(fa, fb)), Fraction(0))
    sign = 1 if p > 0 else (-1 if p < 0 else 0)
    return (0, sign * p * p / (a * b))


def _order(values: np.ndarray, exact_key, descending: bool) -> np.ndarray:
    """Indices 0..n-1 ordered by ``values`` (descending or ascending), lower
    index first among equal keys, with near-tie runs ordered exactly."""
    n = len(values)
    idx = np.arange(n)
    v = np.asarray(values, dtype=np.float64)
    primary = -v if descending else v
    order = np.lexsort((idx, primary))
    if n < 2:
        return order
    sv = v[order]
    with np.errstate(invalid="ignore"):
        gaps = np.abs(np.diff(sv))
    near = ~(gaps > NEAR_TIE)          # NaN gaps (inf - inf) count as ties
    out = order.copy()
    start = 0
    while start < n - 1:
        if not near[start]:
            start += 1
            continue
        end = start
        while end < n - 1 and near[end]:
            end += 1
        run = order[start:end + 1]
        keys = {int(i): exact_key(int(i)) for i in run}
        if descending:
            ranked = sorted(run, key=lambda i: ((keys[int(i)][0], -keys[int(i)][1]), int(i)))
        else:
            ranked = sorted(run, key=lambda i: ((keys[int(i)][0], keys[int(i)][1]), int(i)))
        out[start:end + 1] = ranked
        start = end + 1
    return out


# --------------------------------------------------------------------------
# One image: Stage I and Stage II (Section IV-A, IV-B; Algorithm 1)
# --------------------------------------------------------------------------
def select_image(x, x_pre, x_post, k: int, k1: int, stride_mode: str = "alg1") -> dict:
    """Run Algorithm 1 on one image: x, x', x'' are [N, D] arrays.

    Returns a dict with ``imp`` (importance tokens, in H2 order), ``div``
    (diversity tokens, in pick order), ``kept`` (ascending token indices),
    ``h2``, ``s`` and the stride ``t``.  ``stride_mode`` chooses the
    positions of X_div (see ``pick_positions``).
    """
    x = np.asarray(x, dtype=np.float64)
    n = x.shape[0]
    if not (0 <= k1 <= k <= n):
        raise ValueError("need 0 <= K1 <= K <= N")
    k2 = k - k1
    h2 = renyi2_entropy(x)
    imp_order = _order(h2, lambda i: exact_r(x[i]), descending=True)
    imp = imp_order[:k1]
    rem = np.sort(imp_order[k1:])                     # X_rem = X \ X_imp
    s = consistency(x_pre, x_post)
    xp = np.asarray(x_pre, dtype=np.float64)
    xq = np.asarray(x_post, dtype=np.float64)
    rem_sorted = rem[_order(s[rem], lambda j: exact_sigma(xp[rem[j]], xq[rem[j]]), descending=False)]
    if k2 > 0:
        t = stride(len(rem), k2)
        div = rem_sorted[pick_positions(len(rem), k2, stride_mode)]
    else:
        t = 0
        div = np.zeros(0, dtype=np.int64)
    kept = np.sort(np.concatenate([imp, div]))
    return dict(imp=imp, div=div, kept=kept, h2=h2, s=s, t=t, rem_sorted=rem_sorted)
