"""The seeded input generator: shapes, determinism and recipe features."""
import pytest
import torch

import synth


def test_shapes_and_determinism():
    a = synth.make("llava576", seed=3, batch=2, n=64, d=256)
    b = synth.make("llava576", seed=3, batch=2, n=64, d=256)
    assert a.x.shape == (128, 256) and a.x.dtype == torch.bfloat16
    assert torch.equal(a.x, b.x) and torch.equal(a.x_pre, b.x_pre) and torch.equal(a.x_post, b.x_post)
    c = synth.make("llava576", seed=4, batch=2, n=64, d=256)
    assert not torch.equal(a.x, c.x)


def test_ragged_and_video():
    r = synth.make("ragged_dynres", seed=0, batch=5, n=(16, 80), d=64)
    assert len(r.seqlens) == 5 and all(16 <= n <= 80 for n in r.seqlens)
    assert r.total == sum(r.seqlens) and r.cu_seqlens().tolist()[-1] == r.total
    v = synth.make("video6272", seed=0, batch=1, frames=4, frame_tokens=10, d=64)
    assert v.total == 40
    # consecutive frames differ by small drift only (away from outlier rows)
    d01 = (v.x_pre[10:20].float() - v.x_pre[0:10].float()).abs().median()
    assert d01 < 0.1


def test_outliers_and_residual():
    w = synth.make("single_clip336", seed=1, n=2000, d=1024)
    assert w.x.dtype == torch.float32
    assert torch.allclose(w.x, w.x_pre + w.x_post, atol=1e-5)
    chans = list(synth.OUTLIER_CHANNELS)
    others = [c for c in range(1024) if c not in chans]
    assert w.x_pre[:, chans].abs().max() > 4 * w.x_pre[:, others].abs().max()


def test_video_frames_view():
    w = synth.make("video6272", seed=1, batch=2, frames=4)
    f = w.frames()
    assert f.seqlens == [196] * 8 and f.x is w.x and f.total == w.total
    with pytest.raises(ValueError):
        synth.make("llava576", batch=1, d=64).frames()
