"""The CPU oracle timed on several host cores at once.

TEST INFRASTRUCTURE ONLY: bench.py's CPU-baseline leg uses it to report the
oracle's throughput with one worker process per core next to the
one-thread figure.  It holds none of the method's arithmetic: each worker
decodes the stored inputs of one image to float64 and calls
``select_image`` on it in a loop.  Workers are separate processes (start
method "spawn"), so the numpy code runs on as many cores at once.
"""
from __future__ import annotations

import time

import numpy as np


def _decode(kind, raw, shape):
    """Stored bf16 / fp16 / fp32 values (raw bits) as float64, exactly."""
    if kind == "bf16":
        bits = np.frombuffer(raw, dtype=np.uint16).astype(np.uint32) << 16
        v = bits.view(np.float32)
    elif kind == "f16":
        v = np.frombuffer(raw, dtype=np.float16)
    else:
        v = np.frombuffer(raw, dtype=np.float32)
    return v.astype(np.float64).reshape(shape)


def worker(payload, barrier, results):
    """Runs in a worker process: one untimed call, then a common start
    (barrier), then select_image on this worker's image for `seconds`."""
    from .altr import select_image
    kind, shape, raws, k, k1, stride, seconds = payload
    x, xp, xq = (_decode(kind, r, shape) for r in raws)
    select_image(x, xp, xq, k, k1, stride)
    barrier.wait(timeout=600)
    t0 = time.monotonic()
    count = 0
    while True:
        select_image(x, xp, xq, k, k1, stride)
        count += 1
        if time.monotonic() - t0 >= seconds:
            break
    results.put((count, t0, time.monotonic()))


def time_all_cores(payloads, timeout=900.0):
    """One process per payload, all started together; returns
    (images per second over the common window, processes)."""
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    barrier = ctx.Barrier(len(payloads))
    results = ctx.Queue()
    procs = [ctx.Process(target=worker, args=(p, barrier, results), daemon=True) for p in payloads]
    for p in procs:
        p.start()
    out = [results.get(timeout=timeout) for _ in procs]
    for p in procs:
        p.join(timeout=60)
    count = sum(c for c, _, _ in out)
    window = max(e for _, _, e in out) - min(s for _, s, _ in out)
    return count / window, len(procs)
