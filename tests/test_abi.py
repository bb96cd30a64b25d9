"""The C ABI on the host: the library loads, exports every function the
header declares, computes budgets exactly like the oracle, and rejects bad
arguments before touching the GPU.  No GPU needed (no kernel is launched)."""
import ctypes

import pytest

import oracle
from paper_2607_13500_gb300 import _build, _lib


@pytest.fixture(scope="module")
def lib():
    _build.build()
    return _lib.load()


def test_exports_every_declared_function(lib):
    names = _lib.declared_functions()
    assert {"tr_budgets", "tr_score", "tr_select", "tr_gather", "tr_select_gather", "tr_reduce", "tr_workspace_bytes",
            "tr_status_string", "tr_version"} <= set(names)
    for name in names:
        assert hasattr(lib, name), name
    assert lib.tr_version().startswith(b"libtr")
    assert lib.tr_status_string(0) == b"ok"


def _budgets(lib, seqlens, k=0, ratio=(0, 0), lam=(1, 3)):
    b = len(seqlens)
    I = ctypes.c_int32
    hk, hk1, hcu = (I * max(b, 1))(), (I * max(b, 1))(), (I * (b + 1))()
    rc = lib.tr_budgets(b, (I * max(b, 1))(*seqlens), k, ratio[0], ratio[1], lam[0], lam[1], hk, hk1, hcu)
    return rc, list(hk)[:b], list(hk1)[:b], list(hcu)


@pytest.mark.parametrize("lam", [(1, 3), (0, 1), (1, 1), (1, 2), (2, 7)])
def test_budgets_match_oracle(lib, lam):
    seqlens = [576, 2880, 256, 16384, 1, 7, 0, 1000]
    for ratio in [(1, 9), (2, 9), (1, 3), (1, 8), (1, 1)]:
        rc, ks, k1s, cu = _budgets(lib, seqlens, ratio=ratio, lam=lam)
        assert rc == 0
        want_k = [oracle.budget_from_ratio(n, ratio) for n in seqlens]
        assert ks == want_k
        assert k1s == [oracle.budget_split(k, lam)[0] for k in want_k]
        assert cu[0] == 0 and all(cu[i + 1] - cu[i] == ks[i] for i in range(len(ks)))
    rc, ks, k1s, _ = _budgets(lib, [576] * 3, k=192, lam=lam)
    assert rc == 0 and ks == [192] * 3 and k1s == [oracle.budget_split(192, lam)[0]] * 3


def test_budget_errors(lib):
    assert _budgets(lib, [100], k=101)[0] == 2            # K > N
    assert _budgets(lib, [100], k=0, ratio=(3, 2))[0] == 2  # ratio > 1
    assert _budgets(lib, [100], k=10, lam=(4, 3))[0] == 2   # lambda > 1
    assert _budgets(lib, [100], k=10, lam=(1, 0))[0] == 2
    assert _budgets(lib, [-1], k=1)[0] == 1


def _tok(**kw):
    base = dict(x=0x10000, x_pre=None, x_post=0x20000, dtype=1, d=4096, batch=2, n=576, cu_seqlens=None,
                total=1152, max_n=576)
    base.update(kw)
    return _lib.TrTokens(**base)


def test_host_argument_checks(lib):
    stats = ctypes.c_void_p(0x30000)
    r = lambda t: lib.tr_score(ctypes.byref(t), stats, None, None, None)
    assert r(_tok(x=None)) == 1
    assert r(_tok(x_post=None)) == 1
    assert r(_tok(dtype=5)) == 3
    assert r(_tok(d=4100)) == 4            # 4100 * 2 bytes is not a multiple of 16
    assert r(_tok(x=0x10008)) == 4         # base not 16-byte aligned
    assert r(_tok(d=20000)) == 7
    assert r(_tok(n=20000)) == 7
    assert r(_tok(n=-1)) == 1
    assert r(_tok(flags=2)) == 1           # unknown selection option
    assert r(_tok(flags=-1)) == 1
    assert lib.tr_score(ctypes.byref(_tok()), None, None, None, None) == 1
    assert lib.tr_score(ctypes.byref(_tok()), ctypes.c_void_p(0x30004), None, None, None) == 4
    # workspace checks of tr_select / tr_reduce come before any launch
    t = _tok()
    need = lib.tr_workspace_bytes(ctypes.byref(t))
    assert need > 1152 * 32
    v = ctypes.c_void_p
    args = [v(0x30000), v(0x40000), v(0x40100), v(0x40200), v(0x50000), None, None, None]
    assert lib.tr_select(ctypes.byref(t), *args, None, need, None, None) == 5
    assert lib.tr_select(ctypes.byref(t), *args, v(0x60000), need - 1, None, None) == 5
    assert lib.tr_select(ctypes.byref(t), *args, v(0x60010), need, None, None) == 5
    assert lib.tr_reduce(ctypes.byref(t), v(0x40000), v(0x40100), v(0x40200), 1153, v(0x70000), v(0x50000),
                         None, None, v(0x60000), need, None, None) == 2
    assert lib.tr_reduce(ctypes.byref(t), v(0x40000), v(0x40100), v(0x40200), 10, v(0x70008), v(0x50000),
                         None, None, v(0x60000), need, None, None) == 4
    assert lib.tr_workspace_bytes(ctypes.byref(_tok(dtype=9))) == 0
    assert lib.tr_gather(ctypes.byref(t), v(0x40200), v(0x50000), 1153, v(0x70000), None) == 2
    assert lib.tr_gather(ctypes.byref(t), None, v(0x50000), 10, v(0x70000), None) == 1
    assert lib.tr_gather(ctypes.byref(t), v(0x40200), v(0x50000), 10, v(0x70004), None) == 4
    # tr_project: every check comes before any CUDA call; no rows is a no-op
    p = lambda y=v(0x40000), rows=64, d=1024, w=v(0x80000), b=None, d_out=4096, act=0, z=v(0x90000): \
        lib.tr_project(y, rows, d, w, b, d_out, act, z, None, None)
    assert p(rows=0) == 0
    assert p(y=None, rows=0) == 1
    assert p(z=None, rows=0) == 1
    assert p(rows=-1) == 1
    assert p(act=9, rows=0) == 1
    assert p(d=1000, rows=0) == 4             # not a multiple of 16
    assert p(d_out=4100, rows=0) == 4
    assert p(d=20000, rows=0) == 7
    assert p(y=v(0x40008), rows=0) == 4       # base not 16-byte aligned
    assert p(b=v(0x50004), rows=0) == 4


def test_pipeline_host_argument_checks(lib):
    # every check before the pipeline creates its CUDA events
    v, VP = ctypes.c_void_p, ctypes.c_void_p
    out = VP()
    ws2 = (VP * 2)(0x100000, 0x200000)
    st2 = (VP * 2)(None, None)
    assert lib.tr_pipeline_create(st2, None, 2, ws2, 4096, None) == 1
    assert lib.tr_pipeline_create(st2, None, 0, ws2, 4096, ctypes.byref(out)) == 1
    assert lib.tr_pipeline_create((VP * 9)(), None, 9, (VP * 9)(*[0x100000] * 9), 4096, ctypes.byref(out)) == 1
    assert lib.tr_pipeline_create(st2, None, 2, None, 4096, ctypes.byref(out)) == 1
    assert lib.tr_pipeline_create(None, None, 2, ws2, 4096, ctypes.byref(out)) == 1
    assert lib.tr_pipeline_create(st2, None, 2, (VP * 2)(0x100000, None), 4096, ctypes.byref(out)) == 5
    assert lib.tr_pipeline_create(st2, None, 2, (VP * 2)(0x100000, 0x200010), 4096, ctypes.byref(out)) == 5
    assert out.value is None
    t = _tok()
    assert lib.tr_pipeline_submit(None, ctypes.byref(t), v(0x40000), v(0x40100), v(0x40200), 10, v(0x70000),
                                  v(0x50000), None, None, None, None, None) == 1
    assert lib.tr_pipeline_wait(None, None) == 1
    assert lib.tr_pipeline_destroy(None) == 0
    assert lib.tr_pipeline_kernels(None) == 0


def test_missing_library_raises(monkeypatch, tmp_path):
    # The product path has no CPU fallback: without libtr.so every entry
    # point fails loudly instead of computing anything on the host.
    monkeypatch.setattr(_lib, "LIB_PATH", str(tmp_path / "libtr.so"))
    monkeypatch.setattr(_lib, "_lib", None)
    with pytest.raises(RuntimeError, match="missing"):
        _lib.load()
    import torch

    import paper_2607_13500_gb300 as altr
    x = torch.zeros(1, 8, 64, dtype=torch.bfloat16)  # host tensors are refused too
    with pytest.raises(ValueError, match="no CPU path"):
        altr.reduce(x, x, x, k=2)
    with pytest.raises(RuntimeError, match="missing"):
        altr.budgets([8], k=2)


def test_binding_refuses_bad_buffers_before_any_launch(lib, monkeypatch):
    # Caller-supplied buffers are checked in Python before the library sees a
    # pointer: host tensors for the MLP and the projector, and statistics of
    # the wrong dtype, size or layout for the selection (the token tensors'
    # own device check is bypassed here so that host tensors reach it).
    import torch

    from paper_2607_13500_gb300 import api
    w = torch.zeros(64, 32, dtype=torch.bfloat16)
    with pytest.raises(ValueError, match="CUDA"):
        api.Mlp(4, w, w.t().contiguous())
    with pytest.raises(ValueError, match="CUDA"):
        api.project(torch.zeros(4, 32, dtype=torch.bfloat16), w)
    monkeypatch.setattr(api, "_flatten", lambda x, xp, xq, sl: (x, xp, xq, sl or [x.shape[0]]))
    x = torch.zeros(16, 64, dtype=torch.bfloat16)
    good = torch.zeros(16, 8)
    for bad in (good.double(), good[:8], good.t()):
        with pytest.raises(ValueError, match="stats"):
            api.select(x, x, x, bad, k=4)
    with pytest.raises(ValueError, match="h2"):
        api.select(x, x, x, good, k=4, h2=torch.zeros(3))
    with pytest.raises(ValueError, match="s must"):
        api.select(x, x, x, good, k=4, s=torch.zeros(16, dtype=torch.float64))
    # and good buffers go through to the entry point (stubbed: no GPU here)
    calls = []
    monkeypatch.setattr(lib, "tr_select", lambda *args: calls.append(len(args)) or 0)
    monkeypatch.setattr(api, "_stream", lambda device: None)
    monkeypatch.setattr(api, "_workspace", lambda lib_, tok, device: (torch.empty(256, dtype=torch.uint8), 256))
    idx, role, cu_k, status = api.select(x, x, x, good, k=4, h2=torch.zeros(16), s=torch.zeros(16))
    assert calls == [13] and cu_k == [0, 4] and idx.shape == (4,) and role.shape == (16,)
