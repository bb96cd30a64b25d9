"""The encoder's final-layer MLP on the tensor cores with the scoring fused
into its second GEMM (tr_mlp_hidden, tr_mlp_score; Eq. 5, Section IV-B).

* H = sigma(x' W1^T + b1) and x'' = H W2^T + b2 against float64 references
  on the CPU (the x'' reference takes the kernel's own H, so each GEMM is
  checked alone).  Tolerance per element: 2^-8 |ref| (the bf16 rounding of
  the output, with a factor 2 of margin) + 2^-16 sum_k |a_k b_k| (fp32
  accumulation of K products; a pairwise or blocked fp32 sum of K = 4096
  terms stays near log2(K) u = 2^-20.4 of that, the bound leaves 16x) +
  for H, the same propagated through sigma (|sigma'| <= 1.13).
* x = bf16(resid + x'') bit for bit, recomputed from the stored x''.
* The statistics records against the exact sums of the stored x, x', x''.
* The selection that tr_select makes from these records: kept indices and
  gathered rows bit for bit against the oracle run on the stored tensors,
  and identical to the selection from tr_score's records.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_13500_gb300 import _build
    _build.build()


def _alt():
    import paper_2607_13500_gb300 as altr
    return altr


def _f64(t):
    return t.float().cpu().numpy().astype(np.float64)


def _sigma(v, act):
    if act == "gelu":
        return 0.5 * v * (1.0 + torch.special.erf(v / math.sqrt(2.0)))
    if act == "quick_gelu":
        return v * torch.sigmoid(1.702 * v)
    return v


def _gemm_ref(a, b, bias):
    """a [m, k] b [n, k]^T (+ bias) and sum_k |a_k b_k| in float64 on the CPU."""
    a64, b64 = a.double().cpu(), b.double().cpu()
    v = a64 @ b64.T
    mag = a64.abs() @ b64.abs().T
    if bias is not None:
        v = v + bias.double().cpu()
    return v, mag


def _check_close(got, ref, mag, slope=1.0):
    got = got.double().cpu()
    tol = 2.0 ** -8 * ref.abs() + slope * 2.0 ** -16 * mag + 1e-6
    bad = (got - ref).abs() > tol
    assert not bad.any(), (int(bad.sum()), float(((got - ref).abs() / tol).max()))


def _inputs(t, d, dh, seed, resid=True, bias=True):
    g = torch.Generator().manual_seed(seed)
    x_pre = torch.randn(t, d, generator=g).to(torch.bfloat16)
    w1 = (torch.randn(dh, d, generator=g) / math.sqrt(d)).to(torch.bfloat16)
    w2 = (torch.randn(d, dh, generator=g) / math.sqrt(dh)).to(torch.bfloat16)
    b1 = 0.1 * torch.randn(dh, generator=g) if bias else None
    b2 = 0.1 * torch.randn(d, generator=g) if bias else None
    r = torch.randn(t, d, generator=g).to(torch.bfloat16) if resid else None
    dev = torch.device("cuda")
    mv = lambda v: None if v is None else v.to(dev)
    return mv(x_pre), mv(w1), mv(w2), mv(b1), mv(b2), mv(r)


CASES = [
    # name, rows, D, hidden, activation, residual, bias
    ("clip_l", 300, 1024, 4096, "gelu", True, True),           # 3 row blocks, the last ragged
    ("ragged_dims", 200, 1152, 4304, "quick_gelu", True, False),  # a half column block, a K tail of 16
    ("one_row", 1, 256, 512, "none", False, True),              # x = x'' (no residual)
    ("even_tiles_ragged", 600, 1296, 4400, "gelu", True, True),  # even column tile counts, every edge ragged
]


@pytest.mark.parametrize("name,t,d,dh,act,resid,bias", CASES, ids=[c[0] for c in CASES])
def test_mlp_outputs_and_records(name, t, d, dh, act, resid, bias):
    altr = _alt()
    xp, w1, w2, b1, b2, r = _inputs(t, d, dh, seed=len(name), resid=resid, bias=bias)
    m = altr.Mlp(t, w1, w2, b1, b2, act=act, scores=True)
    out = m.run(xp, r)
    torch.cuda.synchronize()
    assert out.error.item() == 0
    # H against float64, through sigma
    v1, mag1 = _gemm_ref(xp, w1, b1)
    _check_close(out.h, _sigma(v1, act), mag1, slope=1.13)
    # x'' against float64 on the kernel's own H
    v2, mag2 = _gemm_ref(out.h, w2, b2)
    _check_close(out.x_post, v2, mag2)
    # x = bf16(resid + x'') exactly
    want_x = (r.float() + out.x_post.float()).to(torch.bfloat16) if resid else out.x_post
    assert torch.equal(out.x.view(torch.int16), want_x.view(torch.int16))
    # records: the sums of the stored tensors
    st = out.stats.double().cpu().numpy()
    xx, pp, qq = _f64(out.x), _f64(xp), _f64(out.x_post)
    l1, s2 = np.abs(xx).sum(1), (xx * xx).sum(1)
    a, b, p = (pp * pp).sum(1), (qq * qq).sum(1), (pp * qq).sum(1)
    for col, want in ((0, l1), (1, s2), (2, a), (3, b)):
        assert np.allclose(st[:, col], want, rtol=2.0 ** -23, atol=0), col
    assert np.all(np.abs(st[:, 4] + st[:, 5] - p) <= 1e-9 * np.sqrt(a * b))
    assert np.allclose(st[:, 6], l1 * l1 / s2, rtol=2.0 ** -22)
    assert np.allclose(st[:, 7], p / np.sqrt(a * b), rtol=0, atol=2.0 ** -23)
    # the same records as the scoring pass over the stored tensors
    ref_stats, _, _ = altr.score(out.x, xp, out.x_post)
    torch.cuda.synchronize()
    rs = ref_stats.double().cpu().numpy()
    assert np.allclose(st[:, :4], rs[:, :4], rtol=4e-7, atol=0)
    # a second call gives the same bits (the arrival counters start again at zero)
    h0, q0, x0, s0 = (v.clone() for v in (out.h, out.x_post, out.x, out.stats))
    out2 = m.run(xp, r)
    torch.cuda.synchronize()
    for u, w in ((h0, out2.h), (q0, out2.x_post), (x0, out2.x), (s0, out2.stats)):
        assert torch.equal(u, w)
    assert out2.error.item() == 0


def _select_and_check(altr, out, xp, seqlens, budget, images):
    """tr_select on the fused records: indices and gathered rows against the
    oracle on the stored tensors, and equal to the selection on tr_score's."""
    ks, k1s, cu = budget
    idx, _, _, status = altr.select(out.x, xp, out.x_post, out.stats, seqlens=seqlens, budget=budget)
    stats2, _, _ = altr.score(out.x, xp, out.x_post, seqlens=seqlens)
    idx2, _, _, _ = altr.select(out.x, xp, out.x_post, stats2, seqlens=seqlens, budget=budget)
    torch.cuda.synchronize()
    st = status.cpu().tolist()
    assert st[1] == 0 and st[3] == 0, st
    assert torch.equal(idx, idx2)
    from paper_2607_13500_gb300 import _lib
    from paper_2607_13500_gb300.api import _Tokens, _ptr, _stream
    tok = _Tokens(out.x, xp, out.x_post, seqlens)
    y = torch.empty(max(cu[-1], 1), out.x.shape[1], dtype=torch.bfloat16, device=out.x.device)
    d_cu = torch.tensor(cu, dtype=torch.int32, device=out.x.device)
    _lib.check("tr_gather", _lib.load().tr_gather(tok.ref(), _ptr(d_cu), _ptr(idx), cu[-1], _ptr(y),
                                                  _stream(out.x.device)))
    torch.cuda.synchronize()
    idx_h, y_h = idx.cpu().numpy(), y.cpu()
    offs = np.concatenate([[0], np.cumsum(seqlens)]).astype(np.int64)
    for b in images:
        o0, o1 = int(offs[b]), int(offs[b + 1])
        ref = oracle.select_image(_f64(out.x[o0:o1]), _f64(xp[o0:o1]), _f64(out.x_post[o0:o1]), ks[b], k1s[b])
        assert np.array_equal(idx_h[cu[b]:cu[b + 1]], ref["kept"]), b
        rows = out.x[o0:o1].cpu()[torch.from_numpy(ref["kept"].astype(np.int64))]
        assert torch.equal(y_h[cu[b]:cu[b + 1]].view(torch.int16), rows.view(torch.int16)), b


def test_fused_selection_small():
    # Three 576-token images of the CLIP-L-shaped workload (cluster mixture,
    # activation outliers), K = 192 and K = 64.
    altr = _alt()
    w = synth.make_mlp(seed=3, device="cuda", batch=3)
    m = altr.Mlp(w.total, w.w1, w.w2, w.b1, w.b2, act="gelu")
    out = m.run(w.x_pre, w.resid)
    torch.cuda.synchronize()
    assert out.error.item() == 0
    for k in (192, 64):
        budget = altr.budgets(w.seqlens, k=k)
        _select_and_check(altr, out, w.x_pre, w.seqlens, budget, range(w.batch))


def test_fused_selection_full_size():
    # The full CLIP-L-shaped batch (64 images x 576 tokens, D = 1024,
    # hidden 4096): GEMM outputs on sampled rows, the selection of sampled
    # images against the oracle.
    altr = _alt()
    w = synth.make_mlp(seed=0, device="cuda")
    m = altr.Mlp(w.total, w.w1, w.w2, w.b1, w.b2, act="gelu")
    out = m.run(w.x_pre, w.resid)
    torch.cuda.synchronize()
    assert out.error.item() == 0
    rows = torch.tensor([0, 1, 577, 9000, 20000, w.total - 1])
    v1, mag1 = _gemm_ref(w.x_pre[rows], w.w1, w.b1)
    _check_close(out.h[rows], _sigma(v1, "gelu"), mag1, slope=1.13)
    v2, mag2 = _gemm_ref(out.h[rows], w.w2, w.b2)
    _check_close(out.x_post[rows], v2, mag2)
    want_x = (w.resid.float() + out.x_post.float()).to(torch.bfloat16)
    assert torch.equal(out.x.view(torch.int16), want_x.view(torch.int16))
    budget = altr.budgets(w.seqlens, k=w.k)
    _select_and_check(altr, out, w.x_pre, w.seqlens, budget, [0, 37, 63])


# ---------------------------------------------------------------- projector on the kept tokens
@pytest.mark.parametrize("name,over,bud,d_out,act", [
    ("llava576", dict(batch=3, d=1024), dict(k=192), 4096, "gelu"),           # LLaVA-1.5's 1024 -> 4096 layer
    ("ragged_dynres", dict(batch=5, n=(256, 3000), d=1152), dict(ratio=(2, 9)), 1280, "quick_gelu"),
    ("llava576", dict(batch=2, d=1040), dict(k=64), 512, "gelu"),              # a partial last k-block
], ids=["llava576", "ragged_dynres", "partial_kblock"])
def test_project_kept(name, over, bud, d_out, act):
    # Selection, then the projector's first layer on the kept tokens read
    # from x by index: bit for bit tr_project on the gathered copy y (the
    # hidden-GEMM kernel with plain TMA loads), and within the GEMM tolerance
    # of float64 on the kept rows.
    altr = _alt()
    w_in = synth.make(name, seed=17, device="cuda", **over)
    budget = altr.budgets(w_in.seqlens, **bud)
    r = altr.reduce(w_in.x, w_in.x_pre, w_in.x_post, seqlens=w_in.seqlens, budget=budget)
    g = torch.Generator(device="cuda").manual_seed(5)
    w = (torch.randn(d_out, w_in.d, generator=g, device="cuda") / math.sqrt(w_in.d)).to(torch.bfloat16)
    bias = 0.05 * torch.randn(d_out, generator=g, device="cuda")
    z, err = altr.project_kept(w_in.x, r.idx, budget[2], w, bias, act=act, seqlens=w_in.seqlens)
    zh, err_h = altr.project(r.y, w, bias, act=act)
    torch.cuda.synchronize()
    assert err.item() == 0 and err_h.item() == 0
    assert torch.equal(z.view(torch.int16), zh.view(torch.int16))
    v, mag = _gemm_ref(r.y, w, bias)
    _check_close(z, _sigma(v, act), mag, slope=1.13)


def test_project_kept_index_outside_its_image():
    # A kept index past its image's tokens (or negative) feeds a zero row:
    # its output row is sigma(bias), the other rows are untouched by it.
    altr = _alt()
    x = _inputs(100, 256, 512, seed=9, resid=False, bias=False)[0]
    idx = torch.tensor([0, 10, 55, -3, 1, 49, 50], dtype=torch.int32, device="cuda")
    cu = [0, 4, 7]
    g = torch.Generator(device="cuda").manual_seed(6)
    w = (torch.randn(256, 256, generator=g, device="cuda") / 16).to(torch.bfloat16)
    bias = 0.1 * torch.randn(256, generator=g, device="cuda")
    z, err = altr.project_kept(x, idx, cu, w, bias, act="gelu", seqlens=[50, 50])
    torch.cuda.synchronize()
    assert err.item() == 0
    rows = torch.zeros(7, 256, dtype=torch.bfloat16, device="cuda")  # slots 2, 3, 6 stay zero rows
    for slot, row in [(0, 0), (1, 10), (4, 51), (5, 99)]:
        rows[slot] = x[row]
    v, mag = _gemm_ref(rows, w, bias)
    _check_close(z, _sigma(v, "gelu"), mag, slope=1.13)
