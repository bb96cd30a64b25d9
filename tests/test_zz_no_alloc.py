"""tr_reduce_noalloc, the entry point for callers that cannot allocate device
memory, against the CPU oracle and against tr_reduce (which takes a
caller-allocated workspace).

Both run the same kernels; the no-alloc variant takes its scratch from an
array inside libtr.  Two calls in a row must each reproduce the oracle's
selection and tr_reduce's output: the shared array keeps the previous
call's contents, which must not leak into the next result.  This file is
collected last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu


def _lib():
    from paper_2607_13500_gb300 import _build, _lib as L
    _build.build()
    lib = L.load()
    VP, I32 = ctypes.c_void_p, ctypes.c_int32
    lib.tr_reduce_noalloc.argtypes = [ctypes.POINTER(L.TrTokens), VP, VP, VP, I32, VP, VP, VP, VP, VP, VP]
    lib.tr_reduce_noalloc.restype = I32
    return lib


def _p(t):
    return ctypes.c_void_p(t.data_ptr())


@pytest.mark.parametrize("name,over,budget", [
    ("llava576", dict(batch=8, d=2048), dict(k=192)),
    ("ragged_dynres", dict(batch=4, n=(256, 3000), d=1024), dict(ratio=(2, 9))),
])
def test_noalloc_matches_reduce_twice(name, over, budget):
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    lib = _lib()
    import paper_2607_13500_gb300 as altr
    from paper_2607_13500_gb300.api import _Tokens

    w = synth.make(name, seed=21, device="cuda", **over)
    ks, k1s, cu = altr.budgets(w.seqlens, **budget)
    ref = altr.reduce(w.x, w.x_pre, w.x_post, seqlens=w.seqlens, budget=(ks, k1s, cu), scores=True)
    torch.cuda.synchronize()
    tok = _Tokens(w.x, w.x_pre, w.x_post, w.seqlens)
    dev = w.x.device
    d_k = torch.tensor(ks, dtype=torch.int32, device=dev)
    d_k1 = torch.tensor(k1s, dtype=torch.int32, device=dev)
    d_cu = torch.tensor(cu, dtype=torch.int32, device=dev)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    offs = np.concatenate([[0], np.cumsum(w.seqlens)]).astype(np.int64)
    f64 = lambda t: t.float().cpu().numpy().astype(np.float64)
    refs = [oracle.select_image(f64(w.x[offs[b]:offs[b + 1]]), f64(w.x_pre[offs[b]:offs[b + 1]]),
                                f64(w.x_post[offs[b]:offs[b + 1]]), ks[b], k1s[b]) for b in range(w.batch)]
    for call in range(2):
        y = torch.full((cu[-1], w.d), float("nan"), dtype=w.x.dtype, device=dev)
        idx = torch.full((cu[-1],), -1, dtype=torch.int32, device=dev)
        h2 = torch.full((w.total,), float("nan"), device=dev)
        s = torch.full((w.total,), float("nan"), device=dev)
        status = torch.zeros(4, dtype=torch.int32, device=dev)
        rc = lib.tr_reduce_noalloc(tok.ref(), _p(d_k), _p(d_k1), _p(d_cu), cu[-1], _p(y), _p(idx), _p(h2), _p(s),
                                   _p(status), stream)
        assert rc == 0, rc
        torch.cuda.synchronize()
        idx_h, y_h = idx.cpu(), y.cpu()
        for b, r in enumerate(refs):
            assert np.array_equal(idx_h[cu[b]:cu[b + 1]].numpy(), r["kept"]), (call, b)
            rows = w.x[offs[b]:offs[b + 1]].cpu()[torch.from_numpy(r["kept"].astype(np.int64))]
            assert torch.equal(y_h[cu[b]:cu[b + 1]].view(torch.int16), rows.view(torch.int16)), (call, b)
        assert torch.equal(idx, ref.idx), call
        assert torch.equal(y.view(torch.int16), ref.y.view(torch.int16)), call
        h2r, h2n = ref.h2.cpu().numpy(), h2.cpu().numpy()
        assert np.allclose(h2n, h2r, rtol=2e-3, atol=1e-6), call
        assert np.allclose(s.cpu().numpy(), ref.s.cpu().numpy(), rtol=0, atol=1e-5), call
        assert status.cpu().tolist()[1] == 0 and status.cpu().tolist()[3] == 0


def test_noalloc_rejects_oversized_batch():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    lib = _lib()
    from paper_2607_13500_gb300 import _lib as L
    t = L.TrTokens(x=0x10000, x_pre=None, x_post=0x20000, dtype=1, d=1024, batch=64, n=1024, cu_seqlens=None,
                   total=65536, max_n=1024)
    v = ctypes.c_void_p
    rc = lib.tr_reduce_noalloc(ctypes.byref(t), v(0x40000), v(0x40100), v(0x40200), 64, v(0x70000), v(0x50000),
                               None, None, None, None)
    assert rc == 7  # TR_ERR_UNSUPPORTED: more than TR_NOALLOC_MAX_ROWS rows


def test_noalloc_skips_images_outside_the_rows():
    # Offsets that run past the packed rows (image 1 claims rows 60..130 of
    # 100) are skipped by the selection before anything is read or written,
    # so no exact record lands outside the library's scratch array; image 0
    # is reduced as usual.
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    lib = _lib()
    from paper_2607_13500_gb300 import _lib as L
    dev = torch.device("cuda")
    g = torch.Generator().manual_seed(43)
    x, xp, xq = (torch.randn(100, 256, generator=g).to(torch.bfloat16).to(dev) for _ in range(3))
    cu = torch.tensor([0, 60, 130], dtype=torch.int32, device=dev)
    tok = L.TrTokens(x=x.data_ptr(), x_pre=xp.data_ptr(), x_post=xq.data_ptr(), dtype=1, d=256, batch=2, n=0,
                     cu_seqlens=cu.data_ptr(), total=100, max_n=70, flags=0)
    d_k, d_k1, d_cu = (torch.tensor(v, dtype=torch.int32, device=dev) for v in ([20, 20], [6, 6], [0, 20, 40]))
    y = torch.zeros(40, 256, dtype=torch.bfloat16, device=dev)
    idx = torch.full((40,), -1, dtype=torch.int32, device=dev)
    status = torch.zeros(4, dtype=torch.int32, device=dev)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    rc = lib.tr_reduce_noalloc(ctypes.byref(tok), _p(d_k), _p(d_k1), _p(d_cu), 40, _p(y), _p(idx), None, None,
                               _p(status), stream)
    assert rc == 0, rc
    torch.cuda.synchronize()
    assert status.cpu().tolist()[3] == 1
    f64 = lambda t: t[:60].float().cpu().numpy().astype(np.float64)
    ref = oracle.select_image(f64(x), f64(xp), f64(xq), 20, 6)
    assert np.array_equal(idx[:20].cpu().numpy(), ref["kept"])
    assert idx[20:].cpu().tolist() == [-1] * 20
