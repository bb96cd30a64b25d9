"""Plant plausible mistakes in a copy of the oracle and check that the pins
catch every one of them (a dropped term, a wrong sign, a transposed operand,
a reversed order, an off-by-one stride, a wrong rounding).  CPU only."""
import importlib.util
import os

import pytest

import oracle
import oracle.altr
from oracle_pins import ALL_PINS

SRC = os.path.join(os.path.dirname(oracle.altr.__file__), "altr.py")

MUTANTS = {
    "entropy_without_abs": ("a = np.abs(np.where(np.isfinite(x), x, 0.0))", "a = np.where(np.isfinite(x), x, 0.0)"),
    "entropy_without_square": ("(p * p).sum(axis=1)", "p.sum(axis=1)"),
    "entropy_normalised_over_tokens": ("p = a / safe[:, None]",
                                       "p = a / np.maximum(a.sum(axis=0, keepdims=True), 1e-300)"),
    "entropy_sign_flipped": ("h2 = -np.log(", "h2 = np.log("),
    "cosine_wrong_norm_operand": ("nb = np.sqrt((xq * xq).sum(axis=1))", "nb = np.sqrt((xp * xp).sum(axis=1))"),
    "cosine_sign_flipped": ("dot = (xp * xq).sum(axis=1)", "dot = -(xp * xq).sum(axis=1)"),
    "cosine_missing_one_norm": ("s = dot / np.where(zero, 1.0, na * nb)", "s = dot / np.where(zero, 1.0, na)"),
    "importance_ascending": ("imp_order = _order(h2, lambda i: exact_r(x[i]), descending=True)",
                             "imp_order = _order(h2, lambda i: exact_r(x[i]), descending=False)"),
    "consistency_sorted_descending": ("exact_sigma(xp[rem[j]], xq[rem[j]]), descending=False)",
                                      "exact_sigma(xp[rem[j]], xq[rem[j]]), descending=True)"),
    "stride_picks_interval_ends": ("return j * stride(n_rem, k2)", "return (j + 1) * stride(n_rem, k2) - 1"),
    "interval_ceil_not_floor": ("return (j * n_rem) // k2", "return -((-j * n_rem) // k2)"),
    "interval_rounded": ("return (j * n_rem) // k2", "return np.round(j * n_rem / k2).astype(np.int64)"),
    "stride_rounded": ("return max(1, n_rem // k2)", "return max(1, round(n_rem / k2))"),
    "k1_rounded_up": ("k1 = (k * num) // den", "k1 = -((-k * num) // den)"),
    "ratio_rounded": ("return max(1, (n * num) // den)", "return max(1, round(n * num / den))"),
    "tie_break_higher_index": ("-keys[int(i)][1]), int(i))", "-keys[int(i)][1]), -int(i))"),
    "exact_importance_reversed": ("key=lambda i: ((keys[int(i)][0], -keys[int(i)][1]), int(i))",
                                  "key=lambda i: ((keys[int(i)][0], keys[int(i)][1]), int(i))"),
    "exact_sigma_drops_sign": ("return (0, sign * p * p / (a * b))", "return (0, p * p / (a * b))"),
    "zero_row_entropy_nan": ("h2 = np.where(l1 > 0, h2, 0.0)", "h2 = np.where(l1 > 0, h2, np.nan)"),
}


def _load_mutant(old, new):
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation anchor not unique: {old!r}"
    spec = importlib.util.spec_from_loader("oracle_mutant", loader=None)
    mod = importlib.util.module_from_spec(spec)
    exec(compile(src.replace(old, new), SRC + " (mutant)", "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_mutant(name, monkeypatch):
    mod = _load_mutant(*MUTANTS[name])
    for attr in oracle.__all__:
        monkeypatch.setattr(oracle, attr, getattr(mod, attr))
    caught = []
    for pin in ALL_PINS:
        try:
            pin()
        except Exception as e:  # an assertion or a crash both expose the mistake
            caught.append((pin.__name__, type(e).__name__))
    assert caught, f"no pin catches mutant {name}"
