"""tr_reduce_noalloc, the entry point for callers that cannot allocate device
memory, against tr_reduce (which takes a caller-allocated workspace).

Both run the same kernels; the no-alloc variant takes its scratch from an
array inside libtr.  Two calls in a row must each reproduce tr_reduce's
output: the shared array keeps the previous call's contents, which must not
leak into the next result.  This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

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
