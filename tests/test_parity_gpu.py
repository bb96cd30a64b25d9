"""CUDA path versus the CPU oracle, element by element, through the C ABI.

Kept indices and gathered rows must match bit for bit; H2 within 1e-5
relative (fp32 inputs), 2e-3 relative (bf16 inputs) or 1e-3 relative (fp16
inputs) and s within 1e-5 absolute.  Small cases check every image; the full-size workloads (the
launch configuration bench.py times) check sampled images one by one.
"""
import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

H2_RTOL = {torch.float32: 1e-5, torch.bfloat16: 2e-3, torch.float16: 1e-3}
S_ATOL = 1e-5


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


def _bits(t):
    return t.view(torch.int32) if t.dtype == torch.float32 else t.view(torch.int16)


def check_reduce(x, x_pre, x_post, seqlens, budget, images=None, alias=False, expect_nonfinite=False,
                 stride="alg1"):
    """Runs tr_reduce on the device and compares sampled images with the oracle."""
    altr = _alt()
    dev = torch.device("cuda")
    dx, dq = x.to(dev), x_post.to(dev)
    dp = None if alias else x_pre.to(dev)
    r = altr.reduce(dx, dp, dq, seqlens=seqlens, budget=budget, scores=True, stride=stride)
    torch.cuda.synchronize()
    return compare_result(r, x, x_pre, x_post, seqlens, budget, images, alias, expect_nonfinite, stride)


def compare_result(r, x, x_pre, x_post, seqlens, budget, images=None, alias=False, expect_nonfinite=False,
                   stride="alg1"):
    """A ReduceResult (already complete) against the oracle, image by image."""
    return compare_results([r], x, x_pre, x_post, seqlens, budget, images, alias, expect_nonfinite, stride)[0]


def compare_results(rs, x, x_pre, x_post, seqlens, budget, images=None, alias=False, expect_nonfinite=False,
                    stride="alg1"):
    """Several ReduceResults of the same batch against one oracle run per image."""
    ks, k1s, cu = budget
    statuses, host = [], []
    for r in rs:
        status = r.status.cpu().tolist()
        assert status[1] == 0, f"unresolved rows: {status}"
        assert status[3] == 0, f"invalid budget or kept-count mismatch: {status}"
        if expect_nonfinite:
            assert status[0] > 0
        statuses.append(status)
        host.append((r.idx.cpu().numpy(), r.y.cpu(), r.h2.cpu().numpy().astype(np.float64),
                     r.s.cpu().numpy().astype(np.float64)))
    offs = np.concatenate([[0], np.cumsum(seqlens)]).astype(np.int64)
    images = range(len(seqlens)) if images is None else images
    pre = x if alias else x_pre
    for b in images:
        o0, o1 = int(offs[b]), int(offs[b + 1])
        xb, pb, qb = _f64(x[o0:o1]), _f64(pre[o0:o1]), _f64(x_post[o0:o1])
        ref = oracle.select_image(xb, pb, qb, ks[b], k1s[b], stride)
        want_rows = x[o0:o1][torch.from_numpy(ref["kept"].astype(np.int64))]
        fin = np.isfinite(ref["h2"])
        sf = np.isfinite(ref["s"])
        rt = H2_RTOL[x.dtype]
        for j, (idx, y, h2, s) in enumerate(host):
            got = idx[cu[b]:cu[b + 1]]
            assert np.array_equal(got, ref["kept"]), (j, b, np.setdiff1d(got, ref["kept"]),
                                                      np.setdiff1d(ref["kept"], got))
            assert torch.equal(_bits(y[cu[b]:cu[b + 1]]), _bits(want_rows)), (j, b)
            assert np.all(np.abs(h2[o0:o1][fin] - ref["h2"][fin]) <= rt * np.abs(ref["h2"][fin]) + 1e-6), (j, b)
            assert np.array_equal(np.isneginf(h2[o0:o1][~fin]), np.ones((~fin).sum(), bool)), (j, b)
            assert np.all(np.abs(s[o0:o1][sf] - ref["s"][sf]) <= S_ATOL), (j, b)
    return statuses


def _budget(w, k=None, ratio=None, lam=(1, 3)):
    return _alt().budgets(w.seqlens, k=k, ratio=ratio, lam=lam)


# ---------------------------------------------------------------- the five workloads, shrunk
SMALL = [
    ("single_clip336", {}, [dict(k=64)]),
    ("llava576", dict(batch=6), [dict(k=64), dict(k=128), dict(k=192)]),
    ("multitile2880", dict(batch=2), [dict(k=160), dict(k=320)]),
    ("ragged_dynres", dict(batch=5, n=(256, 3000)), [dict(ratio=(1, 9)), dict(ratio=(2, 9))]),
    ("video6272", dict(batch=2), [dict(ratio=(1, 8))]),
]


@pytest.mark.parametrize("name,over,budgets", SMALL, ids=[s[0] for s in SMALL])
def test_workloads_small(name, over, budgets):
    w = synth.make(name, seed=11, device="cuda", **over)
    x, xp, xq = w.x.cpu(), w.x_pre.cpu(), w.x_post.cpu()
    for bk in budgets:
        check_reduce(x, xp, xq, w.seqlens, _budget(w, **bk))


# ---------------------------------------------------------------- full-size workloads (sampled)
FULL = [
    ("llava576", dict(k=192), None),
    ("multitile2880", dict(k=320), None),
    ("ragged_dynres", dict(ratio=(2, 9)), "largest3"),
    ("video6272", dict(ratio=(1, 8)), [0, 7]),
    ("single_clip336", dict(k=64), None),
]


@pytest.mark.parametrize("name,bk,sample", FULL, ids=[f[0] for f in FULL])
def test_workloads_full_size(name, bk, sample):
    # The full-size batch through tr_reduce and through the two-slot
    # pipeline bench.py times (three submissions: both slots, then slot 0
    # again; for a batch small enough that bench.py replays graphs of
    # pipelined steps, a replayed graph of three too), each checked image by
    # image on the sampled images.
    altr = _alt()
    w = synth.make(name, seed=0, device="cuda")
    if sample == "largest3":
        sample = sorted(range(w.batch), key=lambda b: -w.seqlens[b])[:2] + [0]
    budget = altr.budgets(w.seqlens, **bk)
    single = altr.reduce(w.x, w.x_pre, w.x_post, seqlens=w.seqlens, budget=budget, scores=True)
    pipe = altr.Pipeline(w.seqlens, w.d, w.x.dtype, w.x.device, budget=budget, scores=True, slots=2)
    results = [single]
    try:
        results.append([pipe.submit(w.x, w.x_pre, w.x_post) for _ in range(3)][-1])
        pipe.synchronize()
        import bench
        gpipe = None
        if bench.step_bytes(w, budget[0])[0] < bench.GRAPH_BELOW_BYTES:
            # bench.py replays CUDA graphs of pipelined steps for a batch this small
            gpipe = altr.Pipeline(w.seqlens, w.d, w.x.dtype, w.x.device, budget=budget, scores=True, slots=2)
            g = gpipe.graph(w.x, w.x_pre, w.x_post, steps=3)
            g.replay()
            torch.cuda.synchronize()
            o = gpipe.outs[2 % gpipe.slots]
            results.append(altr.ReduceResult(o["y"][:gpipe.total_k], o["idx"][:gpipe.total_k], gpipe.cu_k, o["h2"],
                                             o["s"], o["status"]))
        x, xp, xq = w.x.cpu(), w.x_pre.cpu(), w.x_post.cpu()
        compare_results(results, x, xp, xq, w.seqlens, budget, images=sample)
        if gpipe is not None:
            del g
            gpipe.close()
    finally:
        pipe.close()


@pytest.mark.parametrize("name,over,bud", [
    ("llava576", dict(batch=4), dict(k=64)),            # |X_rem| = 555, K2 = 43: interval 12.9
    ("multitile2880", dict(batch=2), dict(k=160)),      # 2827 / 107: interval 26.4
    ("ragged_dynres", dict(batch=5, n=(256, 3000)), dict(ratio=(1, 9))),
    ("video6272", dict(batch=2), dict(ratio=(1, 8))),    # 6011 / 523: interval 11.49
], ids=["llava576", "multitile2880", "ragged_dynres", "video6272"])
def test_interval_stride(name, over, bud):
    # Section IV-B's real interval |X_rem| / K2 (TR_STRIDE_INTERVAL), through
    # the single call and through the pipeline.
    w = synth.make(name, seed=5, **over)
    budget = _budget(w, **bud)
    check_reduce(w.x, w.x_pre, w.x_post, w.seqlens, budget, stride="interval")
    altr = _alt()
    dev = torch.device("cuda")
    pipe = altr.Pipeline(w.seqlens, w.d, w.x.dtype, dev, budget=budget, scores=True, stride="interval")
    try:
        r = pipe.submit(w.x.to(dev), w.x_pre.to(dev), w.x_post.to(dev))
        pipe.synchronize()
        compare_result(r, w.x, w.x_pre, w.x_post, w.seqlens, budget, stride="interval")
    finally:
        pipe.close()


def test_video_per_frame_budgets():
    # Every 196-token frame of a clip selected on its own (ratio 1/8: 24 of
    # 196 tokens per frame) instead of once per 6272-token clip.
    w = synth.make("video6272", seed=6, batch=1, frames=8).frames()
    assert w.seqlens == [196] * 8
    check_reduce(w.x, w.x_pre, w.x_post, w.seqlens, _budget(w, ratio=(1, 8)))


def test_lambda_extremes_and_alias():
    w = synth.make("llava576", seed=12, device="cuda", batch=3, d=1024)
    x, xp, xq = w.x.cpu(), w.x_pre.cpu(), w.x_post.cpu()
    for lam in [(0, 1), (1, 1), (1, 2)]:
        check_reduce(x, xp, xq, w.seqlens, _budget(w, k=100, lam=lam))
    check_reduce(x, x, xq, w.seqlens, _budget(w, k=100), alias=True)


def test_score_and_select_entry_points():
    altr = _alt()
    w = synth.make("llava576", seed=13, device="cuda", batch=2, d=2048)
    stats, h2, s = altr.score(w.x, w.x_pre, w.x_post, seqlens=w.seqlens)
    ks, k1s, cu = _budget(w, k=96)
    idx, role, cu_k, status = altr.select(w.x, w.x_pre, w.x_post, stats, seqlens=w.seqlens, budget=(ks, k1s, cu))
    torch.cuda.synchronize()
    role = role.cpu().numpy()
    for b in range(2):
        sl = slice(b * 576, (b + 1) * 576)
        ref = oracle.select_image(_f64(w.x[sl]), _f64(w.x_pre[sl]), _f64(w.x_post[sl]), ks[b], k1s[b])
        assert set(np.nonzero(role[sl] == 1)[0].tolist()) == set(ref["imp"].tolist())
        assert set(np.nonzero(role[sl] == 2)[0].tolist()) == set(ref["div"].tolist())
        assert np.array_equal(idx[cu[b]:cu[b + 1]].cpu().numpy(), ref["kept"])
    # tr_gather on the selection reproduces the rows tr_reduce gathers
    from paper_2607_13500_gb300 import _lib
    from paper_2607_13500_gb300.api import _Tokens, _ptr, _stream
    tok = _Tokens(w.x, w.x_pre, w.x_post, w.seqlens)
    y = torch.empty(cu[-1], w.d, dtype=w.x.dtype, device=w.x.device)
    d_cu = torch.tensor(cu, dtype=torch.int32, device=w.x.device)
    _lib.check("tr_gather", _lib.load().tr_gather(tok.ref(), _ptr(d_cu), _ptr(idx), cu[-1], _ptr(y),
                                                  _stream(w.x.device)))
    ref = altr.reduce(w.x, w.x_pre, w.x_post, seqlens=w.seqlens, budget=(ks, k1s, cu))
    torch.cuda.synchronize()
    assert torch.equal(y.view(torch.int16), ref.y.view(torch.int16))
    assert torch.equal(idx, ref.idx)
    st = stats.cpu().numpy().astype(np.float64)
    xx = _f64(w.x)
    assert np.allclose(st[:, 0], np.abs(xx).sum(1), rtol=2e-6)
    assert np.allclose(st[:, 1], (xx * xx).sum(1), rtol=2e-6)
    p = (_f64(w.x_pre) * _f64(w.x_post)).sum(1)
    scale = np.sqrt((_f64(w.x_pre) ** 2).sum(1) * (_f64(w.x_post) ** 2).sum(1))
    assert np.all(np.abs(st[:, 4] + st[:, 5] - p) <= 1e-9 * scale)


def test_pipeline_overlapped_batches():
    # Three different batches of one shape through a two-slot pipeline: the
    # selection of one overlaps the scoring of the next, slot 0 is reused
    # (its workspace and outputs wait for the earlier gather), and a run of
    # submissions without a host sync in between ends with the right results.
    altr = _alt()
    ws = [synth.make("multitile2880", seed=s, device="cuda", batch=3, n=700, d=1024) for s in range(3)]
    budget = _budget(ws[0], k=120)
    pipe = altr.Pipeline(ws[0].seqlens, ws[0].d, ws[0].x.dtype, "cuda", budget=budget, scores=True, slots=2)
    cpu = [(w.x.cpu(), w.x_pre.cpu(), w.x_post.cpu()) for w in ws]
    try:
        r0 = pipe.submit(ws[0].x, ws[0].x_pre, ws[0].x_post)
        r1 = pipe.submit(ws[1].x, ws[1].x_pre, ws[1].x_post)
        pipe.synchronize()
        compare_result(r0, *cpu[0], ws[0].seqlens, budget)
        compare_result(r1, *cpu[1], ws[1].seqlens, budget)
        order = [2, 0, 1, 2, 2, 1, 0, 2, 1]
        rs = [pipe.submit(ws[i].x, ws[i].x_pre, ws[i].x_post) for i in order]
        pipe.synchronize()
        compare_result(rs[-2], *cpu[order[-2]], ws[0].seqlens, budget)
        compare_result(rs[-1], *cpu[order[-1]], ws[0].seqlens, budget)
    finally:
        pipe.close()


def test_graph_replay_and_limits():
    # tr_reduce captured in a CUDA graph and replayed; one image at the
    # largest N (16384 tokens), and rows at the largest D (16384 channels).
    altr = _alt()
    dev = torch.device("cuda")
    w = synth.make("llava576", seed=8, batch=3, d=512)
    budget = _budget(w, k=100)
    red = altr.Reducer(w.seqlens, w.d, w.x.dtype, dev, budget=budget, scores=True)
    dx, dp, dq = w.x.to(dev), w.x_pre.to(dev), w.x_post.to(dev)
    g = red.graph(dx, dp, dq)
    red.y.zero_()
    red.idx.zero_()
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    res = altr.ReduceResult(red.y[:red.total_k], red.idx[:red.total_k], red.cu_k, red.h2, red.s, red.status)
    compare_result(res, w.x, w.x_pre, w.x_post, w.seqlens, budget)
    x, xp, xq = _rows(16384, 32, 21)
    check_reduce(x, xp, xq, [16384], _alt().budgets([16384], k=1500))
    x, xp, xq = _rows(40, 16384, 22, dtype=torch.float32)
    check_reduce(x, xp, xq, [40], _alt().budgets([40], k=12))
    x, xp, xq = _rows(40, 16384, 23)
    check_reduce(x, xp, xq, [25, 15], _alt().budgets([25, 15], k=10))


@pytest.mark.parametrize("batch", [2, 3])
def test_pipeline_graph_replay(batch):
    # Five pipelined steps (two slots, so the slots are reused inside the
    # graph) captured into one CUDA graph and replayed twice; every slot's
    # outputs match the oracle, the score events time each replay's score
    # kernels, and the captured pipeline refuses host submissions.  Two
    # images select and gather in one launch per step, three in two.
    altr = _alt()
    dev = torch.device("cuda")
    w = synth.make("single_clip336", seed=5, batch=batch)
    budget = _budget(w, k=64)
    pipe = altr.Pipeline(w.seqlens, w.d, w.x.dtype, dev, budget=budget, scores=True, slots=2)
    dx, dp, dq = w.x.to(dev), w.x_pre.to(dev), w.x_post.to(dev)
    try:
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(5)]
        g = pipe.graph(dx, dp, dq, steps=5, score_events=evs)
        assert pipe.kernels == 5 * (2 if batch == 2 else 3)  # fused select + gather for two small images
        for o in pipe.outs:
            o["y"].zero_()
            o["idx"].fill_(-1)
        for _ in range(2):
            g.replay()
        torch.cuda.synchronize()
        for o in pipe.outs:
            r = altr.ReduceResult(o["y"][:pipe.total_k], o["idx"][:pipe.total_k], pipe.cu_k, o["h2"], o["s"],
                                  o["status"])
            compare_result(r, w.x, w.x_pre, w.x_post, w.seqlens, budget)
        assert all(0.0 < e0.elapsed_time(e1) < 1000.0 for e0, e1 in evs)
        with pytest.raises(RuntimeError, match="captured"):
            pipe.submit(dx, dp, dq)
        del g
    finally:
        pipe.close()
    # steps over rotating inputs: with two slots and two input sets, slot j
    # always holds the reduction of input set j
    w2 = synth.make("single_clip336", seed=6, batch=batch)
    pipe = altr.Pipeline(w.seqlens, w.d, w.x.dtype, dev, budget=budget, scores=True, slots=2)
    try:
        sets = [(dx, dp, dq), tuple(t.to(dev) for t in (w2.x, w2.x_pre, w2.x_post))]
        g = pipe.graph(*sets[0], steps=4, inputs=sets)
        g.replay()
        torch.cuda.synchronize()
        for o, src in zip(pipe.outs, (w, w2)):
            r = altr.ReduceResult(o["y"][:pipe.total_k], o["idx"][:pipe.total_k], pipe.cu_k, o["h2"], o["s"],
                                  o["status"])
            compare_result(r, src.x, src.x_pre, src.x_post, src.seqlens, budget)
        del g
    finally:
        pipe.close()
    # the same timing events on host submissions
    pipe = altr.Pipeline(w.seqlens, w.d, w.x.dtype, dev, budget=budget, scores=True, slots=2)
    try:
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(3)]
        rs = [pipe.submit(dx, dp, dq, score_events=ev) for ev in evs]
        pipe.synchronize()
        assert all(0.0 < e0.elapsed_time(e1) < 1000.0 for e0, e1 in evs)
        compare_result(rs[-1], w.x, w.x_pre, w.x_post, w.seqlens, budget)
    finally:
        pipe.close()


def test_pipeline_from_host():
    # Pinned host batches in, y and idx back to pinned host buffers, three
    # different batches through two slots (uploads overlap the work).
    altr = _alt()
    ws = [synth.make("llava576", seed=40 + s, batch=3, d=256) for s in range(3)]
    budget = _budget(ws[0], k=96)
    pipe = altr.Pipeline(ws[0].seqlens, 256, torch.bfloat16, "cuda", budget=budget, scores=True)
    try:
        pin = lambda t: t.pin_memory()
        outs = []
        for w in ws:
            y_h = torch.empty(budget[2][-1], 256, dtype=torch.bfloat16).pin_memory()
            idx_h = torch.empty(budget[2][-1], dtype=torch.int32).pin_memory()
            r = pipe.submit_host(pin(w.x), pin(w.x_pre), pin(w.x_post), y_h, idx_h)
            outs.append((y_h, idx_h, r))
        pipe.synchronize()
        w, (y_h, idx_h, r) = ws[-1], outs[-1]
        compare_result(r, w.x, w.x_pre, w.x_post, w.seqlens, budget)
        for w, (y_h, idx_h, _) in zip(ws, outs):
            ks, k1s, cu = budget
            for b in range(w.batch):
                xb, pb, qb = (_f64(t[b * 576:(b + 1) * 576]) for t in (w.x, w.x_pre, w.x_post))
                ref = oracle.select_image(xb, pb, qb, ks[b], k1s[b])
                assert np.array_equal(idx_h[cu[b]:cu[b + 1]].numpy(), ref["kept"]), b
                rows = w.x[b * 576:(b + 1) * 576][torch.from_numpy(ref["kept"].astype(np.int64))]
                assert torch.equal(_bits(y_h[cu[b]:cu[b + 1]]), _bits(rows)), b
    finally:
        pipe.close()


def test_pipeline_graph_from_host():
    # The end-to-end steps (copy in, reduce, copy out) captured into one graph
    # and replayed: the pinned outputs hold the reduction of whatever the
    # pinned inputs held when the graph ran.
    altr = _alt()
    ws = [synth.make("single_clip336", seed=60 + s, batch=2) for s in range(2)]
    budget = _budget(ws[0], k=64)
    pipe = altr.Pipeline(ws[0].seqlens, ws[0].d, ws[0].x.dtype, "cuda", budget=budget)
    try:
        x_h, p_h, q_h = (t.clone().pin_memory() for t in (ws[0].x, ws[0].x_pre, ws[0].x_post))
        y_h = torch.zeros(budget[2][-1], ws[0].d, dtype=ws[0].x.dtype).pin_memory()
        idx_h = torch.zeros(budget[2][-1], dtype=torch.int32).pin_memory()
        g = pipe.graph_host(x_h, p_h, q_h, y_h, idx_h, steps=3)
        for w in ws:
            x_h.copy_(w.x)
            p_h.copy_(w.x_pre)
            q_h.copy_(w.x_post)
            y_h.zero_()
            idx_h.fill_(-1)
            g.replay()
            torch.cuda.synchronize()
            ks, k1s, cu = budget
            for b in range(w.batch):
                xb, pb, qb = (_f64(t[b * 576:(b + 1) * 576]) for t in (w.x, w.x_pre, w.x_post))
                ref = oracle.select_image(xb, pb, qb, ks[b], k1s[b])
                assert np.array_equal(idx_h[cu[b]:cu[b + 1]].numpy(), ref["kept"]), b
                rows = w.x[b * 576:(b + 1) * 576][torch.from_numpy(ref["kept"].astype(np.int64))]
                assert torch.equal(_bits(y_h[cu[b]:cu[b + 1]]), _bits(rows)), b
        del g
    finally:
        pipe.close()


def test_pipeline_edge_cases():
    # one slot and three slots, an empty image and K = 0 images in a ragged
    # batch, fp32 inputs, and a batch that keeps nothing at all
    altr = _alt()
    dev = torch.device("cuda")
    x, xp, xq = _rows(300, 256, 31, dtype=torch.float32)
    seqlens = [120, 0, 100, 80]
    for slots in (1, 3):
        budget = altr.budgets(seqlens, k=None, ratio=(1, 5))
        pipe = altr.Pipeline(seqlens, 256, torch.float32, dev, budget=budget, scores=True, slots=slots)
        try:
            rs = [pipe.submit(x.to(dev), xp.to(dev), xq.to(dev)) for _ in range(slots + 1)]
            pipe.synchronize()
            compare_result(rs[-1], x, xp, xq, seqlens, budget)
        finally:
            pipe.close()
    budget = ([0, 0, 0, 0], [0, 0, 0, 0], [0, 0, 0, 0, 0])
    pipe = altr.Pipeline(seqlens, 256, torch.float32, dev, budget=budget, scores=True)
    try:
        r = pipe.submit(x.to(dev), xp.to(dev), xq.to(dev))
        pipe.synchronize()
        assert r.idx.numel() == 0 and r.status.cpu().tolist() == [0, 0, 0, 0]
    finally:
        pipe.close()


def test_fp16_inputs():
    # IEEE half inputs: two shrunk workloads (uniform and ragged, both stride
    # modes), then rows with subnormal halves, the largest finite half
    # (65504), infinities and NaNs, which the exact path decodes itself.
    for name, over, bud in [("llava576", dict(batch=4, d=1024), dict(k=128)),
                            ("ragged_dynres", dict(batch=4, n=(256, 2500), d=512), dict(ratio=(2, 9)))]:
        w = synth.make(name, seed=9, dtype="f16", **over)
        for stride in ("alg1", "interval"):
            check_reduce(w.x, w.x_pre, w.x_post, w.seqlens, _budget(w, **bud), stride=stride)
    n, d = 64, 256
    x, xp, xq = _rows(n, d, 14, dtype=torch.float16)
    x[3] = x[3] * 2.0 ** -20                      # mostly subnormal halves
    xp[4] = xp[4] * 2.0 ** -22
    x[5, :8] = 65504.0
    xq[6, 2] = 65504.0
    x[7, 1] = float("inf")
    xq[8, 0] = float("nan")
    x[9] = x[10]                                  # an exact tie
    for k, k1 in [(64, 60), (40, 13), (20, 0)]:
        check_reduce(x, xp, xq, [n], ([k], [k1], [0, k]), expect_nonfinite=True)


# ---------------------------------------------------------------- edge cases
def _rows(n, d, seed, dtype=torch.bfloat16):
    g = torch.Generator().manual_seed(seed)
    mk = lambda: torch.randn(n, d, generator=g).to(dtype)
    return mk(), mk(), mk()


def test_edge_budgets_and_sizes():
    d = 256
    x, xp, xq = _rows(40, d, 1)
    # K = N, K = 0 (explicit), N = 1, an empty image in a ragged batch
    check_reduce(x, xp, xq, [40], ([40], [13], [0, 40]))
    check_reduce(x, xp, xq, [40], ([0], [0], [0, 0]))
    check_reduce(x, xp, xq, [1, 39], ([1, 5], [0, 1], [0, 1, 6]))
    check_reduce(x, xp, xq, [20, 0, 20], ([7, 0, 20], [2, 0, 6], [0, 7, 7, 27]))
    # several tiles and a ragged tail: N not a multiple of anything
    x, xp, xq = _rows(1000, 1032, 2)
    check_reduce(x, xp, xq, [333, 1, 666], ([100, 1, 66], [33, 0, 22], [0, 100, 101, 167]))


def test_many_tiny_images():
    # 3000 images of 1-9 tokens (ragged) and 2000 of 7 (uniform): the
    # selection grid loops over images (the pipeline caps it at a quarter of
    # the SMs) and most images keep everything or nothing but one token.
    altr = _alt()
    dev = torch.device("cuda")
    g = torch.Generator().manual_seed(77)
    seqlens = torch.randint(1, 10, (3000,), generator=g).tolist()
    t = sum(seqlens)
    x, xp, xq = _rows(t, 64, 78)
    budget = altr.budgets(seqlens, k=None, ratio=(1, 3))
    sample = list(range(0, 3000, 97))
    check_reduce(x, xp, xq, seqlens, budget, images=sample)
    pipe = altr.Pipeline(seqlens, 64, torch.bfloat16, dev, budget=budget, scores=True)
    try:
        r = pipe.submit(x.to(dev), xp.to(dev), xq.to(dev))
        pipe.synchronize()
        compare_result(r, x, xp, xq, seqlens, budget, images=sample)
    finally:
        pipe.close()
    x, xp, xq = _rows(2000 * 7, 64, 79)
    check_reduce(x, xp, xq, [7] * 2000, altr.budgets([7] * 2000, k=3), images=list(range(0, 2000, 61)))


def test_exact_ties_and_degenerate_rows():
    d, n = 512, 96
    g = torch.Generator().manual_seed(3)
    base = torch.randn(d, generator=g).to(torch.bfloat16)
    x = torch.stack([base[torch.randperm(d, generator=g)] for _ in range(n)])  # channel permutations: R ties
    other = torch.randn(d, generator=g).to(torch.bfloat16)
    perms = [torch.randperm(d, generator=g) for _ in range(n)]
    xp = torch.stack([base[p] for p in perms])
    xq = torch.stack([other[p] for p in perms])                                # P, A, B tie exactly
    x[5] = 0
    x[6] = 0
    x[7, :] = 0
    x[7, 3] = 2.5                                                               # one-hot: R = 1 like zero rows
    x[8] = x[9]                                                                 # duplicate rows
    xq[10] = 0                                                                  # zero norm: s = 0
    for k, k1 in [(30, 10), (96, 32), (50, 50), (40, 0)]:
        check_reduce(x, xp, xq, [n], ([k], [k1], [0, k]))
    # equal magnitudes with random signs: every row has R = D exactly
    sgn = torch.randint(0, 2, (n, d), generator=g) * 2 - 1
    mags = torch.tensor([0.375, 1.5, 3.0]).repeat(n // 3 + 1)[:n, None]
    xe = (sgn * mags).to(torch.bfloat16)
    check_reduce(xe, xp, xq, [n], ([40], [13], [0, 40]))


def test_sort_paths_uneven_and_tied_keys():
    # 750 distinct rows at every 4th position and 2250 copies of one row
    # whose R = 1 (one-hot) is the smallest of all.  With K1 = 800 the
    # importance cut falls inside the copies (an exact tie) and the window
    # around it is too full, so all 3000 rows are ordered: the copies crowd
    # one value bucket and the stratified sample sort orders them.  The rows
    # left for the consistency order tie in s (sample sort again); with
    # K1 = 256 the cut is certain without any order.
    n, d = 3000, 64
    x, xp, xq = _rows(n, d, 11)
    tied = [i for i in range(n) if i % 4]
    x[tied] = 0
    x[tied, 5] = 1.0
    xp[tied] = xp[1].clone()
    xq[tied] = xq[1].clone()
    for k, k1 in [(1200, 800), (700, 256), (1024, 0)]:
        check_reduce(x, xp, xq, [n], ([k], [k1], [0, k]))


def test_sort_paths_mid_sizes():
    # Between 512 and 2048 rows to order, the sort first tries value
    # buckets (each row ranked inside its bucket by one thread); when a
    # bucket would hold more than 32 rows it declines and a register bitonic
    # sort of 1024 or 2048 places orders the rows.  Distinct rows take the
    # buckets; rows of which three in four are copies of one row (equal s,
    # the smallest R) take both bitonic sizes, for the consistency order
    # and, with the importance cut inside the copies, the importance order.
    for n in (700, 1500):
        x, xp, xq = _rows(n, 64, 20 + n)
        check_reduce(x, xp, xq, [n], ([n // 3], [n // 9], [0, n // 3]))
        tied = [i for i in range(n) if i % 4]
        x[tied] = 0
        x[tied, 5] = 1.0
        xp[tied] = xp[1].clone()
        xq[tied] = xq[1].clone()
        for k, k1 in [(n // 2, n // 3), (n // 3, 0)]:
            check_reduce(x, xp, xq, [n], ([k], [k1], [0, k]))


def _mix32(v):
    v &= 0xFFFFFFFF
    v ^= v >> 16
    v = (v * 0x7FEB352D) & 0xFFFFFFFF
    v ^= v >> 15
    v = (v * 0x846CA68B) & 0xFFFFFFFF
    return v ^ (v >> 16)


def test_sort_fallback_when_samples_are_adversarial():
    # Above 1024 rows the sort first tries value buckets, then draws 512
    # samples, one at a hashed place in each equal stretch of the row list
    # (the places below repeat that scheme).  Here exactly the sampled rows
    # are distinct and every other row is a copy of one row with the
    # smallest R and the largest s: the copies crowd one value bucket and
    # one sample bucket, so both sorts decline and the radix sort orders the
    # rows, for the importance cut (which falls inside the copies) and for
    # the consistency order over all rows.
    n, d, S = 4096, 64, 512
    picked = [t * n // S + _mix32(t + 0x9E3779B9) % ((t + 1) * n // S - t * n // S) for t in range(S)]
    assert len(set(picked)) == S
    x, xp, xq = _rows(n, d, 12)
    rest = sorted(set(range(n)) - set(picked))
    x[rest] = 0
    x[rest, 9] = 1.0
    xp[rest] = 1.0
    xq[rest] = 1.0  # s = 1, the largest
    for k, k1 in [(900, 600), (3000, 0)]:
        check_reduce(x, xp, xq, [n], ([k], [k1], [0, k]))


def test_nonfinite_huge_and_tiny_rows():
    n, d = 64, 256
    x, xp, xq = _rows(n, d, 4)
    x[3, 17] = float("nan")
    x[4, 0] = float("inf")
    xp[5, 2] = float("-inf")
    xq[6, 9] = float("nan")
    x[10] *= 2.0 ** 70                   # squares overflow fp32: settled exactly
    x[11] *= 2.0 ** -70                  # squares underflow fp32: settled exactly
    xp[12] *= 2.0 ** 80
    xq[13] *= 2.0 ** -75
    for k, k1 in [(64, 60), (40, 13), (20, 0)]:
        check_reduce(x, xp, xq, [n], ([k], [k1], [0, k]), expect_nonfinite=True)


def test_exact_sums_past_the_window():
    # Every row is a channel permutation of one fp32 vector that also holds
    # 2^-60 and 2^-75 entries: R and s tie exactly across rows, so every
    # decision goes to the exact sums, and the tiny squares fall below the
    # 128-bit window anchored at the row's sum: the digit accumulator takes
    # over (the fp32 sums themselves stay inside the error model).
    n, d = 64, 256
    g = torch.Generator().manual_seed(9)
    base = torch.randn(d, generator=g)
    base[:6] = torch.tensor([2.0 ** -60, -(2.0 ** -60), 2.0 ** -75, 3 * 2.0 ** -75, 2.0 ** -62, -(2.0 ** -70)])
    other = torch.randn(d, generator=g)
    other[:3] = torch.tensor([2.0 ** -64, 2.0 ** -71, -(2.0 ** -66)])
    perms = [torch.randperm(d, generator=g) for _ in range(n)]
    x = torch.stack([base[p] for p in perms])
    xp = torch.stack([base[p] for p in perms])
    xq = torch.stack([other[p] for p in perms])
    for k, k1 in [(20, 7), (40, 0), (30, 30)]:
        check_reduce(x, xp, xq, [n], ([k], [k1], [0, k]))


def _near_tie_triples(groups, d, dtype, seed):
    """Rows in triples whose keys R and s differ by about 2^-25 inside a
    triple (inside the fp32 keys' certification band, so every triple is an
    uncertain run) and by about 2^-17 between triples (certain in fp32).
    Two channels of x set R: a coarse one (two mantissa steps of 2^-3 per
    triple, in a shuffled triple order) and a fine one (one step of 2^-10 per
    member); two channels of x'' set s the same way against x' = 4 there.
    The rows are shuffled so that index order and key order differ."""
    g = torch.Generator().manual_seed(seed)
    n = 3 * groups
    base = torch.randn(d, generator=g)
    base_p = torch.randn(d, generator=g)
    base_q = 0.5 * base_p + 0.5 * torch.randn(d, generator=g)
    x, xp, xq = base.repeat(n, 1), base_p.repeat(n, 1), base_q.repeat(n, 1)
    coarse_r = torch.randperm(groups, generator=g)
    coarse_s = torch.randperm(groups, generator=g)
    for i in range(n):
        grp, mem = divmod(i, 3)
        x[i, 11] = 2.0 ** -3 * (1 + 2 * int(coarse_r[grp]) / 128)
        x[i, 517] = 2.0 ** -10 * (1 + mem / 128)
        xq[i, 23] = 2.0 ** -3 * (1 + 2 * int(coarse_s[grp]) / 128)
        xq[i, 700] = 2.0 ** -10 * (1 + ((mem + grp) % 3) / 128)
    xp[:, 23] = 4.0
    xp[:, 700] = 4.0
    perm = torch.randperm(n, generator=g)
    return x[perm].to(dtype), xp[perm].to(dtype), xq[perm].to(dtype), perm, coarse_r, coarse_s


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32], ids=["bf16", "f32"])
def test_near_ties_beyond_fp32(dtype):
    # Every triple is an uncertain run of the fp32 keys; the double-float
    # keys separate its rows, so the selection needs no exact sums
    # (status[2] == 0) and still matches the oracle's exact decisions, at the
    # importance cut (K1 = 31 splits a triple) and at the stride picks.
    x, xp, xq, *_ = _near_tie_triples(32, 1024, dtype, 31)
    n = x.shape[0]
    for k, k1 in [(40, 31), (60, 0), (45, 16)]:
        st = check_reduce(x, xp, xq, [n], ([k], [k1], [0, k]))
        assert st[2] == 0, st
    # exact ties inside two triples (two rows equal in x, two in x''): the
    # triple that the importance cut K1 = 31 splits (the 11th from the top
    # by R) and the triple with the smallest s (the first stride pick) fall
    # back to exact sums, every other run stays with the double-float keys
    x, xp, xq, perm, cr, cs = _near_tie_triples(32, 1024, dtype, 32)
    where = torch.argsort(perm)  # where[i]: the shuffled place of row i
    gr = int((cr == 32 - 11).nonzero())
    gs = int((cs == 0).nonzero())
    x[where[3 * gr + 1]] = x[where[3 * gr]]
    xq[where[3 * gs + 1]] = xq[where[3 * gs]]
    for k, k1 in [(40, 31), (60, 0)]:
        st = check_reduce(x, xp, xq, [n], ([k], [k1], [0, k]))
        assert 0 < st[2] <= 6, st


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float16, torch.float32], ids=["bf16", "f16", "f32"])
def test_small_uniform_batches(dtype):
    # Small uniform batches through tr_reduce (scoring, then the replicated
    # selection and copy of k_select_gather): image sizes that are and are
    # not multiples of the select kernel's 16 warps, three input types, and
    # a second call on the same workspace and outputs.
    for batch, n, d, k, k1 in [(5, 40, 256, 12, 4), (2, 16, 512, 6, 2), (3, 576, 1024, 64, 21)]:
        x, xp, xq = _rows(batch * n, d, 40 + n, dtype)
        seqlens = [n] * batch
        budget = ([k] * batch, [k1] * batch, [k * b for b in range(batch + 1)])
        altr = _alt()
        red = altr.Reducer(seqlens, d, dtype, "cuda", budget=budget, scores=True)
        dx, dp, dq = x.cuda(), xp.cuda(), xq.cuda()
        for _ in range(2):
            r = red.run(dx, dp, dq)
            torch.cuda.synchronize()
            compare_result(r, x, xp, xq, seqlens, budget)


def test_fp32_wide_range():
    n, d = 300, 1024
    g = torch.Generator().manual_seed(5)
    x = torch.randn(n, d, generator=g) * torch.exp2(torch.randint(-20, 20, (n, d), generator=g).float())
    xp = torch.randn(n, d, generator=g)
    xq = 0.5 * xp + torch.randn(n, d, generator=g) * torch.exp2(torch.randint(-10, 10, (n, d), generator=g).float())
    check_reduce(x, xp, xq, [n], ([90], [30], [0, 90]))
    check_reduce(x, xp, xq, [100, 200], ([33, 66], [11, 22], [0, 33, 99]))


# ---------------------------------------------------------------- malformed offsets and indices
def _raw_tokens(x, xp, xq, batch, n=0, cu=None, total=None, max_n=0):
    from paper_2607_13500_gb300 import _lib
    return _lib.TrTokens(x=x.data_ptr(), x_pre=xp.data_ptr(), x_post=xq.data_ptr(), dtype=1, d=x.shape[1],
                         batch=batch, n=n, cu_seqlens=None if cu is None else cu.data_ptr(),
                         total=x.shape[0] if total is None else total, max_n=max_n, flags=0)


def test_malformed_offsets_are_skipped():
    # cu_seqlens whose second image runs past the packed rows (100 rows,
    # image 1 claims rows 60..130): the selection counts that image in
    # status[3] and reads and writes nothing for it, image 0 is reduced as
    # usual, and the gather writes zeros into the skipped image's slots
    # (its indices were never written).
    import ctypes
    from paper_2607_13500_gb300 import _lib
    from paper_2607_13500_gb300.api import _ptr, _stream
    lib = _lib.load()
    dev = torch.device("cuda")
    x, xp, xq = (t.to(dev) for t in _rows(100, 256, 41))
    cu = torch.tensor([0, 60, 130], dtype=torch.int32, device=dev)
    tok = _raw_tokens(x, xp, xq, 2, cu=cu, max_n=70)
    ks, k1s, cuk = [20, 20], [6, 6], [0, 20, 40]
    d_k, d_k1, d_cu = (torch.tensor(v, dtype=torch.int32, device=dev) for v in (ks, k1s, cuk))
    nbytes = lib.tr_workspace_bytes(ctypes.byref(tok))
    ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    y = torch.full((40, 256), float("nan"), dtype=torch.bfloat16, device=dev)
    idx = torch.full((40,), -1, dtype=torch.int32, device=dev)
    status = torch.zeros(4, dtype=torch.int32, device=dev)
    _lib.check("tr_reduce", lib.tr_reduce(ctypes.byref(tok), _ptr(d_k), _ptr(d_k1), _ptr(d_cu), 40, _ptr(y),
                                          _ptr(idx), None, None, _ptr(ws), nbytes, _ptr(status), _stream(dev)))
    torch.cuda.synchronize()
    assert status.cpu().tolist()[3] == 1
    ref = oracle.select_image(_f64(x[:60]), _f64(xp[:60]), _f64(xq[:60]), 20, 6)
    assert np.array_equal(idx[:20].cpu().numpy(), ref["kept"])
    assert torch.equal(_bits(y[:20].cpu()), _bits(x[:60].cpu()[torch.from_numpy(ref["kept"].astype(np.int64))]))
    assert idx[20:].cpu().tolist() == [-1] * 20
    assert torch.equal(y[20:].cpu(), torch.zeros(20, 256, dtype=torch.bfloat16))


@pytest.mark.parametrize("ragged", [False, True])
def test_gather_index_outside_its_image_writes_zeros(ragged):
    # tr_gather with indices that leave their own image (55 is a valid row
    # of the next image, -3 is negative, 50 is one past the end) writes zeros
    # for those slots and copies the others bit for bit.
    import ctypes
    from paper_2607_13500_gb300 import _lib
    from paper_2607_13500_gb300.api import _ptr, _stream
    lib = _lib.load()
    dev = torch.device("cuda")
    x, xp, xq = (t.to(dev) for t in _rows(100, 128, 42))
    cu = torch.tensor([0, 50, 100], dtype=torch.int32, device=dev) if ragged else None
    tok = _raw_tokens(x, xp, xq, 2, n=0 if ragged else 50, cu=cu, max_n=50)
    idx = torch.tensor([0, 10, 55, -3, 1, 49, 50], dtype=torch.int32, device=dev)
    d_cu = torch.tensor([0, 4, 7], dtype=torch.int32, device=dev)
    y = torch.full((7, 128), float("nan"), dtype=torch.bfloat16, device=dev)
    _lib.check("tr_gather", lib.tr_gather(ctypes.byref(tok), _ptr(d_cu), _ptr(idx), 7, _ptr(y), _stream(dev)))
    torch.cuda.synchronize()
    want = torch.zeros(7, 128, dtype=torch.bfloat16)
    for slot, row in [(0, 0), (1, 10), (4, 51), (5, 99)]:
        want[slot] = x[row].cpu()
    assert torch.equal(_bits(y.cpu()), _bits(want))
