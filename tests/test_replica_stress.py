"""Repeated single-call and small-batch pipeline reductions of tie-heavy
images, checked bit for bit against the oracle on every repetition.

On a uniform batch with fewer images than SMs, tr_reduce (and the pipeline,
for one or two images of at most 1024 tokens) runs each image's selection in
several replica CTAs at once; each copies its share of the kept rows.  Every
row of these images is a channel permutation of one vector, so the keys of
Eq. 4 and Eq. 6 tie exactly across rows, every decision goes to the exact
sums, and all replicas recompute the same rows' exact records at the same
time.  Each repetition must give the oracle's indices and exactly the rows
they name.
"""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu

REPS = 50


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_13500_gb300 import _build
    _build.build()


def _f64(t):
    return t.float().cpu().numpy().astype(np.float64)


def _bits(t):
    return t.view(torch.int32) if t.dtype == torch.float32 else t.view(torch.int16)


def _permuted_rows(n, d, seed, dtype, tiny):
    # x and x' rows are channel permutations of one vector, x'' rows the same
    # permutations of another: L1, S2, P, A and B are equal on every row.
    # With `tiny`, the vectors also hold entries down to 2^-75, whose squares
    # fall below the 128-bit window of the exact sums (digit accumulator).
    g = torch.Generator().manual_seed(seed)
    base = torch.randn(d, generator=g)
    other = torch.randn(d, generator=g)
    if tiny:
        base[:6] = torch.tensor([2.0 ** -60, -(2.0 ** -60), 2.0 ** -75, 3 * 2.0 ** -75, 2.0 ** -62, -(2.0 ** -70)])
        other[:3] = torch.tensor([2.0 ** -64, 2.0 ** -71, -(2.0 ** -66)])
    base, other = base.to(dtype), other.to(dtype)
    perms = [torch.randperm(d, generator=g) for _ in range(n)]
    x = torch.stack([base[p] for p in perms])
    return x, x.clone(), torch.stack([other[p] for p in perms])


CASES = [
    ("f32_digits", torch.float32, True),
    ("bf16_digits", torch.bfloat16, True),
    ("bf16_window", torch.bfloat16, False),
]


def _batch(batch, dtype, tiny, n=64, d=256):
    parts = [_permuted_rows(n, d, 100 + b, dtype, tiny) for b in range(batch)]
    return tuple(torch.cat([p[i] for p in parts]) for i in range(3))


def _refs(x, xp, xq, batch, n, k, k1):
    return [oracle.select_image(_f64(x[b * n:(b + 1) * n]), _f64(xp[b * n:(b + 1) * n]),
                                _f64(xq[b * n:(b + 1) * n]), k, k1) for b in range(batch)]


def _check(idx, y, status, x, refs, n, k, tag):
    assert status[1] == 0 and status[3] == 0, (tag, status)
    for b, ref in enumerate(refs):
        got = idx[b * k:(b + 1) * k]
        assert np.array_equal(got, ref["kept"]), (tag, b, got, ref["kept"])
        rows = x[b * n:(b + 1) * n][torch.from_numpy(ref["kept"].astype(np.int64))]
        assert torch.equal(_bits(y[b * k:(b + 1) * k]), _bits(rows)), (tag, b)


@pytest.mark.parametrize("batch", [1, 2])
@pytest.mark.parametrize("name,dtype,tiny", CASES, ids=[c[0] for c in CASES])
def test_single_call_replicas_repeated(name, dtype, tiny, batch):
    import paper_2607_13500_gb300 as altr
    n, k, k1 = 64, 20, 7
    x, xp, xq = _batch(batch, dtype, tiny)
    refs = _refs(x, xp, xq, batch, n, k, k1)
    dev = torch.device("cuda")
    dx, dp, dq = x.to(dev), xp.to(dev), xq.to(dev)
    budget = ([k] * batch, [k1] * batch, [k * b for b in range(batch + 1)])
    results = [altr.reduce(dx, dp, dq, seqlens=[n] * batch, budget=budget) for _ in range(REPS)]
    torch.cuda.synchronize()
    for rep, r in enumerate(results):
        _check(r.idx.cpu().numpy(), r.y.cpu(), r.status.cpu().tolist(), x, refs, n, k, (name, batch, rep))


@pytest.mark.parametrize("batch", [1, 2])
@pytest.mark.parametrize("name,dtype,tiny", CASES, ids=[c[0] for c in CASES])
def test_pipeline_small_batch_repeated(name, dtype, tiny, batch):
    # One or two images of 64 tokens: the pipeline selects and gathers them
    # with one replicated launch per step.
    import paper_2607_13500_gb300 as altr
    n, k, k1 = 64, 30, 10
    x, xp, xq = _batch(batch, dtype, tiny)
    refs = _refs(x, xp, xq, batch, n, k, k1)
    dev = torch.device("cuda")
    dx, dp, dq = x.to(dev), xp.to(dev), xq.to(dev)
    budget = ([k] * batch, [k1] * batch, [k * b for b in range(batch + 1)])
    pipe = altr.Pipeline([n] * batch, x.shape[1], dtype, dev, budget=budget, slots=2)
    try:
        for rep in range(REPS):
            r = pipe.submit(dx, dp, dq)
            pipe.synchronize()
            _check(r.idx.cpu().numpy(), r.y.cpu(), r.status.cpu().tolist(), x, refs, n, k, (name, batch, rep))
        assert pipe.kernels == REPS * 2  # score + one select-and-gather launch per step
    finally:
        pipe.close()
