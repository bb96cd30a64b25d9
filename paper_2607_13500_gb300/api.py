"""Python binding of libtr with the C ABI's names (argument marshalling only).

Every step of the path runs in libtr's CUDA kernels; PyTorch only provides
device memory and the current stream.  There is no CPU path: the calls raise
when libtr.so is missing or a tensor is not on a CUDA device.
"""
from __future__ import annotations

import ctypes
from dataclasses import dataclass

import torch

from . import _lib
from ._lib import (STRIDE_MODES, TR_ACT, TR_BF16, TR_F16, TR_F32, TR_STATS_WORDS, TR_STATUS_WORDS, TrMlp,
                   TrTokens, check, load)

_I32 = ctypes.c_int32


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return TR_BF16
    if t.dtype == torch.float16:
        return TR_F16
    if t.dtype == torch.float32:
        return TR_F32
    raise TypeError(f"unsupported dtype {t.dtype}: expected torch.bfloat16, torch.float16 or torch.float32")


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _check_buf(t, device, dtype, min_numel, name):
    """A caller's buffer the library reads or writes: on the tokens' device,
    of the expected dtype, contiguous and large enough (None passes)."""
    if t is None:
        return
    if t.device != device or t.dtype != dtype or not t.is_contiguous() or t.numel() < min_numel:
        raise ValueError(f"{name} must be a contiguous {dtype} tensor of at least {min_numel} elements on {device}")


def _stream(device) -> ctypes.c_void_p:
    return ctypes.c_void_p(torch.cuda.current_stream(device).cuda_stream)


def _flatten(x, x_pre, x_post, seqlens):
    """[B, N, D] or [T, D] (+ seqlens) -> packed [T, D] tensors and seqlens."""
    if x.dim() == 3:
        b, n, d = x.shape
        seqlens = [n] * b
        x = x.reshape(b * n, d)
        x_pre = None if x_pre is None else x_pre.reshape(b * n, d)
        x_post = x_post.reshape(b * n, d)
    elif x.dim() == 2:
        if seqlens is None:
            seqlens = [x.shape[0]]
        seqlens = [int(v) for v in seqlens]
        if sum(seqlens) != x.shape[0]:
            raise ValueError("seqlens must sum to the number of rows of x")
    else:
        raise ValueError("x must be [B, N, D] or [T, D]")
    for t in (x, x_pre, x_post):
        if t is None:
            continue
        if t.shape != x.shape or t.dtype != x.dtype or t.device != x.device:
            raise ValueError("x, x_pre and x_post must share shape, dtype and device")
        if not t.is_contiguous():
            raise ValueError("token tensors must be contiguous")
    if x.device.type != "cuda":
        raise ValueError("token tensors must live on a CUDA device (libtr has no CPU path)")
    return x, x_pre, x_post, seqlens


class _Tokens:
    """A TrTokens struct plus the device tensors it points into."""

    def __init__(self, x, x_pre, x_post, seqlens, stride="alg1"):
        self.x, self.x_pre, self.x_post, self.seqlens = x, x_pre, x_post, seqlens
        if stride not in STRIDE_MODES:
            raise ValueError(f"stride must be one of {sorted(STRIDE_MODES)}")
        uniform = len(set(seqlens)) <= 1
        self.cu = None
        if not uniform:
            cu = [0]
            for n in seqlens:
                cu.append(cu[-1] + n)
            self.cu = torch.tensor(cu, dtype=torch.int32, device=x.device)
        self.s = TrTokens(
            x=x.data_ptr(), x_pre=None if x_pre is None else x_pre.data_ptr(), x_post=x_post.data_ptr(),
            dtype=_dtype_code(x), d=x.shape[1], batch=len(seqlens),
            n=seqlens[0] if (uniform and seqlens) else 0,
            cu_seqlens=None if self.cu is None else self.cu.data_ptr(),
            total=x.shape[0], max_n=max(seqlens) if seqlens else 0, flags=STRIDE_MODES[stride])

    def ref(self):
        return ctypes.byref(self.s)


def budgets(seqlens, k=None, ratio=None, lam=(1, 3)):
    """K_b, K1_b and cu_k per Algorithm 1's first step (tr_budgets)."""
    lib = load()
    b = len(seqlens)
    arr = (_I32 * max(b, 1))(*seqlens)
    hk, hk1, hcu = (_I32 * max(b, 1))(), (_I32 * max(b, 1))(), (_I32 * (b + 1))()
    kk = int(k) if k else 0
    rn, rd = ratio if ratio else (0, 0)
    check("tr_budgets", lib.tr_budgets(b, arr, kk, rn, rd, lam[0], lam[1], hk, hk1, hcu))
    return list(hk)[:b], list(hk1)[:b], list(hcu)


def workspace_bytes(x, x_pre, x_post, seqlens=None) -> int:
    x, x_pre, x_post, seqlens = _flatten(x, x_pre, x_post, seqlens)
    return load().tr_workspace_bytes(_Tokens(x, x_pre, x_post, seqlens).ref())


def score(x, x_pre, x_post, seqlens=None):
    """tr_score: returns (stats [T, 8] fp32, h2 [T] fp32, s [T] fp32)."""
    lib = load()
    x, x_pre, x_post, seqlens = _flatten(x, x_pre, x_post, seqlens)
    tok = _Tokens(x, x_pre, x_post, seqlens)
    t = x.shape[0]
    stats = torch.empty(t, TR_STATS_WORDS, dtype=torch.float32, device=x.device)
    h2 = torch.empty(t, dtype=torch.float32, device=x.device)
    s = torch.empty(t, dtype=torch.float32, device=x.device)
    check("tr_score", lib.tr_score(tok.ref(), _ptr(stats), _ptr(h2), _ptr(s), _stream(x.device)))
    return stats, h2, s


def _workspace(lib, tok, device):
    nbytes = lib.tr_workspace_bytes(tok.ref())
    ws = torch.empty(max(nbytes, 256), dtype=torch.uint8, device=device)
    assert ws.data_ptr() % 256 == 0
    return ws, nbytes


def select(x, x_pre, x_post, stats, k=None, ratio=None, lam=(1, 3), seqlens=None, h2=None, s=None, budget=None,
           stride="alg1"):
    """tr_select: returns (idx int32 [sum K], role uint8 [T], cu_k list, status int32 [4]).

    ``budget`` may pass explicit (ks, k1s, cu_k) lists instead of k/ratio/lam;
    ``stride`` is "alg1" (Algorithm 1) or "interval" (Section IV-B's real
    interval, TR_STRIDE_INTERVAL)."""
    lib = load()
    x, x_pre, x_post, seqlens = _flatten(x, x_pre, x_post, seqlens)
    t = x.shape[0]
    _check_buf(stats, x.device, torch.float32, t * TR_STATS_WORDS, "stats")
    _check_buf(h2, x.device, torch.float32, t, "h2")
    _check_buf(s, x.device, torch.float32, t, "s")
    tok = _Tokens(x, x_pre, x_post, seqlens, stride)
    ks, k1s, cu_k = budget if budget is not None else budgets(seqlens, k, ratio, lam)
    dev = x.device
    d_k = torch.tensor(ks, dtype=torch.int32, device=dev)
    d_k1 = torch.tensor(k1s, dtype=torch.int32, device=dev)
    d_cu = torch.tensor(cu_k, dtype=torch.int32, device=dev)
    idx = torch.empty(max(cu_k[-1], 1), dtype=torch.int32, device=dev)
    role = torch.empty(x.shape[0], dtype=torch.uint8, device=dev)
    status = torch.zeros(TR_STATUS_WORDS, dtype=torch.int32, device=dev)
    ws, nbytes = _workspace(lib, tok, dev)
    check("tr_select", lib.tr_select(tok.ref(), _ptr(stats), _ptr(d_k), _ptr(d_k1), _ptr(d_cu), _ptr(idx),
                                     _ptr(role), _ptr(h2), _ptr(s), _ptr(ws), nbytes, _ptr(status),
                                     _stream(dev)))
    return idx[:cu_k[-1]], role, cu_k, status


@dataclass
class ReduceResult:
    y: torch.Tensor        # [sum K, D] kept tokens, input dtype
    idx: torch.Tensor      # [sum K] int32 local indices, ascending per image
    cu_k: list             # prefix sums of K_b
    h2: torch.Tensor | None
    s: torch.Tensor | None
    status: torch.Tensor   # int32[4], see include/tr.h


class Reducer:
    """tr_reduce with buffers allocated once for a fixed batch shape.

    ``run`` takes device tensors (inputs already in HBM); ``run_host`` takes
    pinned host tensors, copies them in, reduces, and copies y and idx back.
    """

    def __init__(self, seqlens, d, dtype, device, k=None, ratio=None, lam=(1, 3), alias_pre=False, scores=False,
                 budget=None, stride="alg1"):
        self.lib = load()
        self.seqlens = [int(v) for v in seqlens]
        self.device = torch.device(device)
        self.d, self.dtype, self.alias_pre, self.stride = d, dtype, alias_pre, stride
        self.ks, self.k1s, self.cu_k = budget if budget is not None else budgets(self.seqlens, k, ratio, lam)
        self.total_k = self.cu_k[-1]
        t = sum(self.seqlens)
        dev = self.device
        self.d_k = torch.tensor(self.ks, dtype=torch.int32, device=dev)
        self.d_k1 = torch.tensor(self.k1s, dtype=torch.int32, device=dev)
        self.d_cu = torch.tensor(self.cu_k, dtype=torch.int32, device=dev)
        self.y = torch.empty(max(self.total_k, 1), d, dtype=dtype, device=dev)
        self.idx = torch.empty(max(self.total_k, 1), dtype=torch.int32, device=dev)
        self.h2 = torch.empty(t, dtype=torch.float32, device=dev) if scores else None
        self.s = torch.empty(t, dtype=torch.float32, device=dev) if scores else None
        self.status = torch.zeros(TR_STATUS_WORDS, dtype=torch.int32, device=dev)
        self._tok = None
        self._ws = None
        self._in = None

    def _bind(self, x, x_pre, x_post):
        x, x_pre, x_post, _ = _flatten(x, x_pre, x_post, self.seqlens)
        key = (x.data_ptr(), None if x_pre is None else x_pre.data_ptr(), x_post.data_ptr())
        if self._tok is None or self._in != key:
            self._tok = _Tokens(x, x_pre, x_post, self.seqlens, self.stride)
            self._in = key
            if self._ws is None:
                self._ws, self._ws_bytes = _workspace(self.lib, self._tok, self.device)
        return self._tok

    def run(self, x, x_pre, x_post) -> ReduceResult:
        tok = self._bind(x, x_pre, x_post)
        check("tr_reduce", self.lib.tr_reduce(
            tok.ref(), _ptr(self.d_k), _ptr(self.d_k1), _ptr(self.d_cu), self.total_k, _ptr(self.y),
            _ptr(self.idx), _ptr(self.h2), _ptr(self.s), _ptr(self._ws), self._ws_bytes, _ptr(self.status),
            _stream(self.device)))
        return ReduceResult(self.y[:self.total_k], self.idx[:self.total_k], self.cu_k, self.h2, self.s,
                            self.status)

    def graph(self, x, x_pre, x_post) -> "torch.cuda.CUDAGraph":
        """``run`` (with the status words zeroed first) captured into a CUDA
        graph for these input tensors; ``replay()`` repeats it with one
        launch.  Outputs land in this Reducer's buffers (``y``, ``idx``, ...)."""
        self.run(x, x_pre, x_post)  # outside the capture first: sets the kernels' shared-memory limit once
        torch.cuda.synchronize(self.device)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.status.zero_()
            self.run(x, x_pre, x_post)
        return g

    def run_split(self, x, x_pre, x_post, events=None):
        """The same two kernels as ``run`` through the entry points tr_score
        and tr_select_gather, with ``events`` (three torch.cuda.Event, or
        None) recorded before, between and after them on the current stream,
        so that each kernel can be timed inside a step."""
        tok = self._bind(x, x_pre, x_post)
        st = _stream(self.device)
        lib = self.lib
        stats = self._stats_view()
        if events:
            events[0].record()
        check("tr_score", lib.tr_score(tok.ref(), _ptr(stats), _ptr(self.h2), _ptr(self.s), st))
        if events:
            events[1].record()
        check("tr_select_gather", lib.tr_select_gather(
            tok.ref(), _ptr(stats), _ptr(self.d_k), _ptr(self.d_k1), _ptr(self.d_cu), self.total_k, _ptr(self.y),
            _ptr(self.idx), _ptr(self.h2), _ptr(self.s), _ptr(self._ws), self._ws_bytes, _ptr(self.status), st))
        if events:
            events[2].record()
        return ReduceResult(self.y[:self.total_k], self.idx[:self.total_k], self.cu_k, self.h2, self.s,
                            self.status)

    def run_select_gather(self, x, x_pre, x_post, stats, events=None):
        """tr_select then tr_gather on statistics records made elsewhere (e.g.
        by Mlp's fused scoring), on the current stream; ``events`` (three
        torch.cuda.Event or None) recorded before, between and after."""
        tok = self._bind(x, x_pre, x_post)
        _check_buf(stats, tok.x.device, torch.float32, tok.x.shape[0] * TR_STATS_WORDS, "stats")
        st = _stream(self.device)
        lib = self.lib
        self.status.zero_()
        if events:
            events[0].record()
        check("tr_select", lib.tr_select(
            tok.ref(), _ptr(stats), _ptr(self.d_k), _ptr(self.d_k1), _ptr(self.d_cu), _ptr(self.idx), None,
            _ptr(self.h2), _ptr(self.s), _ptr(self._ws), self._ws_bytes, _ptr(self.status), st))
        if events:
            events[1].record()
        check("tr_gather", lib.tr_gather(tok.ref(), _ptr(self.d_cu), _ptr(self.idx), self.total_k, _ptr(self.y), st))
        if events:
            events[2].record()
        return ReduceResult(self.y[:self.total_k], self.idx[:self.total_k], self.cu_k, self.h2, self.s,
                            self.status)

    def run_separate(self, x, x_pre, x_post, events=None):
        """The three kernels the pipeline launches, tr_score, tr_select and
        tr_gather, on the current stream, with ``events`` (four
        torch.cuda.Event, or None) recorded before, between and after them."""
        tok = self._bind(x, x_pre, x_post)
        st = _stream(self.device)
        lib = self.lib
        stats = self._stats_view()
        if events:
            events[0].record()
        check("tr_score", lib.tr_score(tok.ref(), _ptr(stats), _ptr(self.h2), _ptr(self.s), st))
        if events:
            events[1].record()
        check("tr_select", lib.tr_select(
            tok.ref(), _ptr(stats), _ptr(self.d_k), _ptr(self.d_k1), _ptr(self.d_cu), _ptr(self.idx), None,
            _ptr(self.h2), _ptr(self.s), _ptr(self._ws), self._ws_bytes, _ptr(self.status), st))
        if events:
            events[2].record()
        check("tr_gather", lib.tr_gather(tok.ref(), _ptr(self.d_cu), _ptr(self.idx), self.total_k, _ptr(self.y), st))
        if events:
            events[3].record()
        return ReduceResult(self.y[:self.total_k], self.idx[:self.total_k], self.cu_k, self.h2, self.s,
                            self.status)

    def _stats_view(self):
        # tr_reduce keeps the statistics at the start of the workspace; the
        # split path uses the same bytes.
        t = sum(self.seqlens)
        return self._ws[: t * TR_STATS_WORDS * 4].view(torch.float32)

    def alloc_device_inputs(self):
        t = sum(self.seqlens)
        mk = lambda: torch.empty(t, self.d, dtype=self.dtype, device=self.device)
        return mk(), (None if self.alias_pre else mk()), mk()

    def run_host(self, x_h, x_pre_h, x_post_h, dev_in, y_h, idx_h) -> ReduceResult:
        """End-to-end: pinned host inputs -> device -> reduce -> pinned host y, idx."""
        dx, dp, dq = dev_in
        dx.copy_(x_h, non_blocking=True)
        if dp is not None:
            dp.copy_(x_pre_h, non_blocking=True)
        dq.copy_(x_post_h, non_blocking=True)
        r = self.run(dx, dp, dq)
        y_h.copy_(r.y, non_blocking=True)
        idx_h.copy_(r.idx, non_blocking=True)
        return r


class Pipeline:
    """tr_pipeline: successive batches of one shape, each scored on its slot's
    stream of ``score_streams`` and then selected and gathered on
    ``select_stream`` (higher priority), so that the selection and gather of
    one batch overlap the scoring of the next, and one batch's scoring the
    drain of the previous one.  Submission i uses workspace, score stream and
    output set i mod ``slots``; its ReduceResult holds that set's tensors,
    valid once ``select_stream`` has passed the submission (``wait`` or
    ``synchronize``) and until submission i + ``slots`` is made.
    """

    def __init__(self, seqlens, d, dtype, device, k=None, ratio=None, lam=(1, 3), alias_pre=False, scores=False,
                 budget=None, slots=2, stride="alg1", score_streams=None):
        self.lib = load()
        self.seqlens = [int(v) for v in seqlens]
        self.device = torch.device(device)
        self.d, self.dtype, self.alias_pre, self.slots, self.stride = d, dtype, alias_pre, int(slots), stride
        self.ks, self.k1s, self.cu_k = budget if budget is not None else budgets(self.seqlens, k, ratio, lam)
        self.total_k = self.cu_k[-1]
        t = sum(self.seqlens)
        dev = self.device
        self.d_k = torch.tensor(self.ks, dtype=torch.int32, device=dev)
        self.d_k1 = torch.tensor(self.k1s, dtype=torch.int32, device=dev)
        self.d_cu = torch.tensor(self.cu_k, dtype=torch.int32, device=dev)
        mk = lambda *shape, dt: torch.empty(*shape, dtype=dt, device=dev)
        self.outs = [dict(y=mk(max(self.total_k, 1), d, dt=dtype), idx=mk(max(self.total_k, 1), dt=torch.int32),
                          h2=mk(t, dt=torch.float32) if scores else None, s=mk(t, dt=torch.float32) if scores else None,
                          status=torch.zeros(TR_STATUS_WORDS, dtype=torch.int32, device=dev))
                     for _ in range(self.slots)]
        n_streams = self.slots if score_streams is None else max(1, min(int(score_streams), self.slots))
        own = [torch.cuda.Stream(dev, priority=0) for _ in range(n_streams)]
        self.score_streams = [own[i % n_streams] for i in range(self.slots)]
        self.select_stream = torch.cuda.Stream(dev, priority=-100)  # the device's highest priority
        self._host = None  # submit_host: per-slot device inputs, copy streams and reuse events
        self._ws = None
        self._handle = None
        self._tok = None
        self._in = None
        self._graphed = False
        self.submitted = 0

    def _bind(self, x, x_pre, x_post):
        x, x_pre, x_post, _ = _flatten(x, x_pre, x_post, self.seqlens)
        key = (x.data_ptr(), None if x_pre is None else x_pre.data_ptr(), x_post.data_ptr())
        if self._tok is None or self._in != key:
            self._tok = _Tokens(x, x_pre, x_post, self.seqlens, self.stride)
            self._in = key
        if self._handle is None:
            nbytes = self.lib.tr_workspace_bytes(self._tok.ref())
            if nbytes == 0:
                raise ValueError("invalid token tensors for tr_pipeline")
            if self._ws is None or self._ws[0].numel() < nbytes:
                self._ws = [torch.empty(nbytes, dtype=torch.uint8, device=self.device) for _ in range(self.slots)]
            assert all(w.data_ptr() % 256 == 0 for w in self._ws)
            ptrs = (ctypes.c_void_p * self.slots)(*[w.data_ptr() for w in self._ws])
            handle = ctypes.c_void_p()
            streams = (ctypes.c_void_p * self.slots)(*[st.cuda_stream for st in self.score_streams])
            with torch.cuda.device(self.device):
                check("tr_pipeline_create", self.lib.tr_pipeline_create(
                    streams, ctypes.c_void_p(self.select_stream.cuda_stream), self.slots, ptrs, nbytes,
                    ctypes.byref(handle)))
            self._handle = handle
        return self._tok

    def submit(self, x, x_pre, x_post, score_events=None, after_current=True) -> ReduceResult:
        """Enqueues one batch; ``score_events`` (two torch.cuda.Event, or
        None) are recorded on the slot's score stream around the score
        kernel.  With
        ``after_current`` the scoring waits for the work already queued on
        the caller's current stream (where the inputs were written); pass
        False when the inputs are known to be ready."""
        if self._graphed and not torch.cuda.is_current_stream_capturing():
            raise RuntimeError("this pipeline was captured by Pipeline.graph: replay the graph instead")
        tok = self._bind(x, x_pre, x_post)
        o = self.outs[self.submitted % self.slots]
        sst = self.score_streams[self.submitted % self.slots]
        if after_current:
            sst.wait_stream(torch.cuda.current_stream(self.device))
        ev = [None, None]
        if score_events is not None:
            for e in score_events:
                if not e.cuda_event:  # torch creates its events lazily, at the first record
                    e.record(sst)
            ev = [ctypes.c_void_p(e.cuda_event) for e in score_events]
        check("tr_pipeline_submit", self.lib.tr_pipeline_submit(
            self._handle, tok.ref(), _ptr(self.d_k), _ptr(self.d_k1), _ptr(self.d_cu), self.total_k, _ptr(o["y"]),
            _ptr(o["idx"]), _ptr(o["h2"]), _ptr(o["s"]), _ptr(o["status"]), ev[0], ev[1]))
        self.submitted += 1
        return ReduceResult(o["y"][:self.total_k], o["idx"][:self.total_k], self.cu_k, o["h2"], o["s"], o["status"])

    def submit_host(self, x_h, x_pre_h, x_post_h, y_h, idx_h) -> ReduceResult:
        """End to end from pinned host memory: copies this batch's inputs into
        the slot's device buffers on a copy-in stream, submits it, and copies
        y and idx back into the pinned ``y_h`` / ``idx_h`` on a copy-out
        stream.  The next batch's upload overlaps this batch's work and
        download.  ``y_h`` and ``idx_h`` are complete after ``synchronize``."""
        slot = self.submitted % self.slots
        if self._host is None:
            t = sum(self.seqlens)
            mk = lambda: torch.empty(t, self.d, dtype=self.dtype, device=self.device)
            self._host = dict(
                bufs=[(mk(), None if self.alias_pre else mk(), mk()) for _ in range(self.slots)],
                cin=torch.cuda.Stream(self.device), cout=torch.cuda.Stream(self.device),
                in_free=[None] * self.slots, out_free=[None] * self.slots)
        h = self._host
        dx, dp, dq = h["bufs"][slot]
        if h["in_free"][slot] is not None:  # the slot's last batch has been gathered
            h["cin"].wait_event(h["in_free"][slot])
        if h["out_free"][slot] is not None:  # and its results copied out
            self.select_stream.wait_event(h["out_free"][slot])
        with torch.cuda.stream(h["cin"]):
            dx.copy_(x_h, non_blocking=True)
            if dp is not None:
                dp.copy_(x_pre_h, non_blocking=True)
            dq.copy_(x_post_h, non_blocking=True)
            r = self.submit(dx, dp, dq)  # scoring waits for the copies (the current stream)
        done = torch.cuda.Event()
        done.record(self.select_stream)
        h["in_free"][slot] = done
        h["cout"].wait_event(done)
        with torch.cuda.stream(h["cout"]):
            y_h.copy_(r.y, non_blocking=True)
            idx_h.copy_(r.idx, non_blocking=True)
            out = torch.cuda.Event()
            out.record(h["cout"])
        h["out_free"][slot] = out
        return r

    def graph(self, x, x_pre, x_post, steps=16, score_events=None, inputs=None) -> "torch.cuda.CUDAGraph":
        """``steps`` pipelined submissions of these input tensors captured into
        one CUDA graph: ``replay()`` runs them (each step's selection and
        gather overlapping the next step's scoring) with a single launch, for
        batches so small that submitting step by step from the host would
        take longer than the GPU work.  ``inputs`` (a list of (x, x_pre,
        x_post) of this shape, or None) gives step i the tensors
        inputs[i mod len(inputs)] instead.  ``score_events`` (``steps`` pairs
        of timing torch.cuda.Event, or None) become event nodes around each
        score kernel.  Step i writes output set i mod ``slots``.  The pipeline
        is dedicated to replays afterwards (``submit`` raises)."""
        if self.submitted and self._handle is not None:
            raise RuntimeError("Pipeline.graph needs a pipeline without earlier submissions")
        inputs = [(x, x_pre, x_post)] if inputs is None else list(inputs)
        cur = torch.cuda.current_stream(self.device)
        # one step outside the capture: the selection kernel's shared-memory
        # limit is raised once per device, on its first launch
        self.submit(x, x_pre, x_post)
        self.synchronize()
        self.lib.tr_pipeline_destroy(self._handle)  # a fresh handle: no earlier events to wait on
        self._handle = None
        self.submitted = 0
        self._bind(x, x_pre, x_post)
        if score_events is not None:
            for pair in score_events:
                for e in pair:
                    e.record(cur)  # created before the capture
        cur.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            cap = torch.cuda.current_stream(self.device)
            for i in range(steps):
                self.submit(*inputs[i % len(inputs)], score_events=None if score_events is None else score_events[i])
            self.wait(cap)
            for st in self.score_streams:
                cap.wait_stream(st)
        self._graphed = True
        return g

    def graph_host(self, x_h, x_pre_h, x_post_h, y_h, idx_h, steps=16) -> "torch.cuda.CUDAGraph":
        """``steps`` end-to-end steps (``submit_host``: pinned host inputs
        copied in, reduced, y and idx copied back to the pinned ``y_h`` /
        ``idx_h``) captured into one CUDA graph, so that a replay needs no
        host work per step.  The host buffers are the graph's: refill them
        between replays.  The pipeline is dedicated to replays afterwards."""
        if self.submitted and self._handle is not None:
            raise RuntimeError("Pipeline.graph_host needs a pipeline without earlier submissions")
        # one step outside the capture: device buffers and copy streams, and
        # the selection kernel's shared-memory limit
        self.submit_host(x_h, x_pre_h, x_post_h, y_h, idx_h)
        self.synchronize()
        self.lib.tr_pipeline_destroy(self._handle)
        self._handle = None
        self.submitted = 0
        h = self._host
        h["in_free"], h["out_free"] = [None] * self.slots, [None] * self.slots
        self._bind(*h["bufs"][0])
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            cap = torch.cuda.current_stream(self.device)
            h["cin"].wait_stream(cap)
            h["cout"].wait_stream(cap)
            self.select_stream.wait_stream(cap)
            for _ in range(steps):
                self.submit_host(x_h, x_pre_h, x_post_h, y_h, idx_h)
            self.wait(cap)
            for st in self.score_streams + [h["cin"], h["cout"], self.select_stream]:
                cap.wait_stream(st)
        self._graphed = True
        return g

    @property
    def kernels(self) -> int:
        """Kernels launched by the submissions of the current handle
        (tr_pipeline_kernels; after ``graph``/``graph_host``: those the
        captured graph launches per replay)."""
        return int(self.lib.tr_pipeline_kernels(self._handle)) if self._handle is not None else 0

    def wait(self, stream=None):
        """Makes ``stream`` (default: the current stream) wait for every submission."""
        st = stream if stream is not None else torch.cuda.current_stream(self.device)
        if self._handle is not None:
            check("tr_pipeline_wait", self.lib.tr_pipeline_wait(self._handle, ctypes.c_void_p(st.cuda_stream)))

    def synchronize(self):
        self.select_stream.synchronize()
        for st in self.score_streams:
            st.synchronize()
        if self._host is not None:
            self._host["cin"].synchronize()
            self._host["cout"].synchronize()

    def close(self):
        if self._handle is not None:
            self.synchronize()
            self.lib.tr_pipeline_destroy(self._handle)
            self._handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def reduce(x, x_pre, x_post, k=None, ratio=None, lam=(1, 3), seqlens=None, scores=False, budget=None,
           stride="alg1"):
    """tr_reduce in one call: returns a ReduceResult (device tensors).
    ``stride`` is "alg1" (Algorithm 1) or "interval" (Section IV-B)."""
    x2, p2, q2, seqlens = _flatten(x, x_pre, x_post, seqlens)
    r = Reducer(seqlens, x2.shape[1], x2.dtype, x2.device, k=k, ratio=ratio, lam=lam, alias_pre=p2 is None,
                scores=scores, budget=budget, stride=stride)
    out = r.run(x2, p2, q2)
    return out


# ---------------------------------------------------------------- encoder MLP with fused scoring
@dataclass
class MlpResult:
    h: torch.Tensor        # [T, d_hidden] sigma(x' W1^T + b1), bf16
    x_post: torch.Tensor   # [T, D] x'' = H W2^T + b2, bf16 (Eq. 5)
    x: torch.Tensor        # [T, D] block output resid + x'' (the tokens X), bf16
    stats: torch.Tensor    # [T, 8] fp32 row records, as tr_score writes them
    h2: torch.Tensor | None
    s: torch.Tensor | None
    error: torch.Tensor    # int32[1]: non-zero if a pipeline wait in a kernel timed out


class Mlp:
    """The encoder's final-layer MLP (Eq. 5) on the tensor cores with the
    scoring fused into its second GEMM (tr_mlp_hidden, tr_mlp_score), for a
    fixed shape; outputs and scratch are allocated once.

    ``w1`` [d_hidden, D] and ``w2`` [D, d_hidden] bf16 (nn.Linear layout),
    ``b1``/``b2`` fp32 or None, ``act`` "gelu", "quick_gelu" or "none"."""

    def __init__(self, t, w1, w2, b1=None, b2=None, act="gelu", scores=False):
        self.lib = load()
        if w1.device.type != "cuda" or w2.device != w1.device or any(
                b is not None and b.device != w1.device for b in (b1, b2)):
            raise ValueError("the MLP weights and biases must live on one CUDA device (libtr has no CPU path)")
        if w1.dtype != torch.bfloat16 or w2.dtype != torch.bfloat16:
            raise TypeError("the MLP weights must be bf16")
        dh, d = w1.shape
        if tuple(w2.shape) != (d, dh):
            raise ValueError("w2 must be [D, d_hidden] for w1 [d_hidden, D]")
        if act not in TR_ACT:
            raise ValueError(f"act must be one of {sorted(TR_ACT)}")
        self.t, self.d, self.dh, self.act = int(t), int(d), int(dh), act
        self.device = w1.device
        dev = self.device
        self.w1, self.w2 = w1.contiguous(), w2.contiguous()
        self.b1 = None if b1 is None else b1.float().contiguous()
        self.b2 = None if b2 is None else b2.float().contiguous()
        self.h = torch.empty(max(self.t, 1), dh, dtype=torch.bfloat16, device=dev)
        self.x_post = torch.empty(max(self.t, 1), d, dtype=torch.bfloat16, device=dev)
        self.x = torch.empty(max(self.t, 1), d, dtype=torch.bfloat16, device=dev)
        self.stats = torch.empty(max(self.t, 1), TR_STATS_WORDS, dtype=torch.float32, device=dev)
        self.h2 = torch.empty(max(self.t, 1), dtype=torch.float32, device=dev) if scores else None
        self.s = torch.empty(max(self.t, 1), dtype=torch.float32, device=dev) if scores else None
        self.error = torch.zeros(1, dtype=torch.int32, device=dev)
        self._ws = None

    def _struct(self, x_pre, resid):
        for t in (x_pre, resid):
            if t is None:
                continue
            if t.dtype != torch.bfloat16 or tuple(t.shape) != (self.t, self.d) or not t.is_contiguous():
                raise ValueError(f"x_pre / resid must be contiguous bf16 [{self.t}, {self.d}]")
            if t.device != self.device:
                raise ValueError("x_pre / resid must be on the weights' device")
        return TrMlp(x_pre=x_pre.data_ptr(), resid=None if resid is None else resid.data_ptr(),
                     w1=self.w1.data_ptr(), w2=self.w2.data_ptr(),
                     b1=None if self.b1 is None else self.b1.data_ptr(),
                     b2=None if self.b2 is None else self.b2.data_ptr(),
                     t=self.t, d=self.d, d_hidden=self.dh, act=TR_ACT[self.act])

    def run(self, x_pre, resid=None, events=None) -> MlpResult:
        """Both GEMMs on the current stream; ``events`` (three torch.cuda.Event
        or None) are recorded before, between and after them."""
        m = self._struct(x_pre, resid)
        ref = ctypes.byref(m)
        if self._ws is None:
            nbytes = self.lib.tr_mlp_workspace_bytes(ref)
            self._ws = torch.empty(max(nbytes, 256), dtype=torch.uint8, device=self.device)
            self._ws_bytes = nbytes
        st = _stream(self.device)
        if events:
            events[0].record()
        check("tr_mlp_hidden", self.lib.tr_mlp_hidden(ref, _ptr(self.h), _ptr(self.error), st))
        if events:
            events[1].record()
        check("tr_mlp_score", self.lib.tr_mlp_score(ref, _ptr(self.h), _ptr(self.x_post), _ptr(self.x),
                                                    _ptr(self.stats), _ptr(self.h2), _ptr(self.s), _ptr(self._ws),
                                                    self._ws_bytes, _ptr(self.error), st))
        if events:
            events[2].record()
        t = self.t
        return MlpResult(self.h[:t], self.x_post[:t], self.x[:t], self.stats[:t],
                         None if self.h2 is None else self.h2[:t], None if self.s is None else self.s[:t],
                         self.error)


def mlp(x_pre, w1, w2, b1=None, b2=None, resid=None, act="gelu", scores=False) -> MlpResult:
    """The encoder's final-layer MLP with the scoring fused in, in one call
    (Eq. 5; see Mlp)."""
    return Mlp(x_pre.shape[0], w1, w2, b1, b2, act, scores).run(x_pre, resid)


def project_kept(x, idx, cu_k, w, bias=None, act="gelu", seqlens=None, error=None):
    """tr_project_kept: z = sigma(X* W^T + bias) for the kept tokens X*, their
    rows read from ``x`` by the selection's ``idx`` (local per image, image b
    owning slots cu_k[b]..cu_k[b+1]) without a gathered copy.  ``w`` bf16
    [d_out, D], ``bias`` fp32 [d_out] or None; returns z bf16 [sum K, d_out]."""
    lib = load()
    if x.dtype != torch.bfloat16 or w.dtype != torch.bfloat16:
        raise TypeError("x and w must be bf16")
    if act not in TR_ACT:
        raise ValueError(f"act must be one of {sorted(TR_ACT)}")
    x2, _, _, seqlens = _flatten(x, None, x, seqlens)
    if w.device != x2.device or idx.device != x2.device or (bias is not None and bias.device != x2.device) or \
            (error is not None and error.device != x2.device):
        raise ValueError("w, idx, bias and error must live on x's device")
    tok = _Tokens(x2, None, x2, seqlens)
    total_k = int(cu_k[-1])
    d_out = int(w.shape[0])
    dev = x2.device
    d_cu = torch.tensor(list(cu_k), dtype=torch.int32, device=dev)
    b = None if bias is None else bias.float().contiguous()
    z = torch.empty(max(total_k, 1), d_out, dtype=torch.bfloat16, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev) if error is None else error
    check("tr_project_kept", lib.tr_project_kept(tok.ref(), _ptr(d_cu), _ptr(idx), total_k, _ptr(w.contiguous()),
                                                 _ptr(b), d_out, TR_ACT[act], _ptr(z), _ptr(err), _stream(dev)))
    return z[:total_k], err


def project(y, w, bias=None, act="gelu", error=None, out=None):
    """tr_project: z = sigma(y W^T + bias) for rows already gathered (tr_gather's
    y, bf16 [rows, D]); ``w`` bf16 [d_out, D], ``bias`` fp32 [d_out] or None;
    ``out`` an optional bf16 [rows, d_out] buffer.  Returns (z, error)."""
    lib = load()
    if y.device.type != "cuda" or w.device != y.device or (bias is not None and bias.device != y.device) or \
            (out is not None and out.device != y.device):
        raise ValueError("y, w, bias and out must live on one CUDA device (libtr has no CPU path)")
    if y.dtype != torch.bfloat16 or w.dtype != torch.bfloat16:
        raise TypeError("y and w must be bf16")
    if act not in TR_ACT:
        raise ValueError(f"act must be one of {sorted(TR_ACT)}")
    if y.dim() != 2 or not y.is_contiguous() or w.dim() != 2 or w.shape[1] != y.shape[1]:
        raise ValueError("y must be contiguous [rows, D] and w [d_out, D]")
    rows, d = int(y.shape[0]), int(y.shape[1])
    d_out = int(w.shape[0])
    dev = y.device
    b = None if bias is None else bias.float().contiguous()
    z = out if out is not None else torch.empty(max(rows, 1), d_out, dtype=torch.bfloat16, device=dev)
    if z.dtype != torch.bfloat16 or not z.is_contiguous() or z.shape[1] != d_out or z.shape[0] < rows:
        raise ValueError(f"out must be contiguous bf16 [>= {rows}, {d_out}]")
    err = torch.zeros(1, dtype=torch.int32, device=dev) if error is None else error
    check("tr_project", lib.tr_project(_ptr(y), rows, d, _ptr(w.contiguous()), _ptr(b), d_out, TR_ACT[act], _ptr(z),
                                       _ptr(err), _stream(dev)))
    return z[:rows], err
