"""Seeded synthetic token workloads shaped like the paper's VLM inputs.

This module only *draws inputs*; it holds none of the reduction method's
arithmetic.  Both the CUDA path and the CPU oracle consume what it returns:

* ``x``      -- visual tokens from the vision encoder (Section III-A), the
               Stage-I input and the gather source;
* ``x_pre``  -- the final-layer MLP input x' (Eq. 5);
* ``x_post`` -- the final-layer MLP output x'' = W2 sigma(W1 x') (Eq. 5).

Recipe (the same for every workload, sizes below):

* ``h`` is a mixture of ``M`` Gaussian clusters: centres ~ N(0, I_D), each
  token is its centre plus N(0, 0.1^2) noise, cluster ids uniform;
* 1% of the tokens (floor(0.01 N), a seeded permutation) are multiplied by 20
  on the four channels {7, 131, 509, 1021} mod D (activation outliers);
* x' = h; x'' = W2 GELU(W1 x') with W1 in R^{64 x D} ~ N(0, 1/D) and
  W2 in R^{D x 64} ~ N(0, 1/64) (a stand-in for the encoder's last MLP,
  evaluated off the clock, so similar tokens get similar consistency
  signals); x = x' + x'' (the residual output of the last block);
* everything is drawn in fp32 and stored in the workload's dtype.

The workloads stand in for the paper's benchmark feature tensors (LLaVA-1.5
on MME/TextVQA/ScienceQA/GQA, LLaVA-NeXT 5-tile images, Qwen2.5-VL dynamic
resolution); no benchmark item is used or needed, only the token shapes.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch

OUTLIER_CHANNELS = (7, 131, 509, 1021)
OUTLIER_SCALE = 20.0
NOISE_SIGMA = 0.1
MLP_HIDDEN = 64

# name -> shape and budget.  ``k`` is a per-image budget, ``ratio`` a retention
# ratio num/den; ``sweep`` lists the other budgets the workload is run at.
SPECS = {
    # CLIP-ViT-L/14-336 single image, fp32 features.
    "single_clip336": dict(batch=1, n=576, d=1024, dtype="f32", clusters=32, k=64, sweep=[64]),
    # LLaVA-1.5 576-token images, batched, bf16 (budgets of Table I).
    "llava576": dict(batch=64, n=576, d=4096, dtype="bf16", clusters=32, k=192, sweep=[64, 128, 192]),
    # LLaVA-NeXT 5 tiles x 576 tokens, tile-major.
    "multitile2880": dict(batch=16, n=2880, d=4096, dtype="bf16", clusters=64, k=320, sweep=[160, 320]),
    # Dynamic-resolution ragged batch, N_b ~ U[256, 16384], clusters ceil(N_b/64).
    "ragged_dynres": dict(batch=32, n=(256, 16384), d=3584, dtype="bf16", clusters="n/64",
                          ratio=(1, 9), sweep=[(1, 9), (2, 9)]),
    # Video clips: 32 frames x 196 tokens, per-frame drift on a 48-cluster base.
    "video6272": dict(batch=8, n=6272, d=3584, dtype="bf16", clusters=48, frames=32, frame_tokens=196,
                      drift=0.02, ratio=(1, 8), sweep=[(1, 8)]),
}


@dataclass
class Workload:
    name: str
    x: torch.Tensor
    x_pre: torch.Tensor
    x_post: torch.Tensor
    seqlens: list
    k: int | None = None
    ratio: tuple | None = None
    lam: tuple = (1, 3)
    meta: dict = field(default_factory=dict)

    @property
    def batch(self) -> int:
        return len(self.seqlens)

    @property
    def d(self) -> int:
        return self.x.shape[1]

    @property
    def total(self) -> int:
        return self.x.shape[0]

    def cu_seqlens(self, device=None) -> torch.Tensor:
        cu = [0]
        for n in self.seqlens:
            cu.append(cu[-1] + n)
        return torch.tensor(cu, dtype=torch.int32, device=device or self.x.device)

    def frames(self) -> "Workload":
        """The same tokens with every frame of a video workload as its own
        image (per-frame budgets instead of per-clip ones)."""
        ft = self.meta["spec"].get("frame_tokens")
        if not ft or any(n % ft for n in self.seqlens):
            raise ValueError(f"{self.name} has no frames")
        seqlens = [ft] * (sum(self.seqlens) // ft)
        return Workload(name=self.name, x=self.x, x_pre=self.x_pre, x_post=self.x_post, seqlens=seqlens,
                        k=self.k, ratio=self.ratio, lam=self.lam, meta=dict(self.meta, per_frame=True))

    def image(self, b: int):
        """Rows of image ``b`` as (x, x_pre, x_post) views."""
        off = sum(self.seqlens[:b])
        n = self.seqlens[b]
        return self.x[off:off + n], self.x_pre[off:off + n], self.x_post[off:off + n]


def _torch_dtype(name: str):
    return {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16}[name]


def _clustered(gen, n, d, clusters, device):
    centres = torch.randn(clusters, d, generator=gen, device=device)
    cid = torch.randint(0, clusters, (n,), generator=gen, device=device)
    return centres[cid] + NOISE_SIGMA * torch.randn(n, d, generator=gen, device=device)


def _video(gen, frames, frame_tokens, d, clusters, drift, device):
    base = _clustered(gen, frame_tokens, d, clusters, device)
    out = torch.empty(frames * frame_tokens, d, device=device)
    cur = base
    for f in range(frames):
        if f:
            cur = cur + drift * torch.randn(frame_tokens, d, generator=gen, device=device)
        out[f * frame_tokens:(f + 1) * frame_tokens] = cur
    return out


def _outliers(gen, h, device):
    n, d = h.shape
    count = n // 100
    if count == 0:
        return h
    rows = torch.randperm(n, generator=gen, device=device)[:count]
    chans = torch.tensor([c % d for c in OUTLIER_CHANNELS], device=device).unique()
    h[rows[:, None], chans[None, :]] *= OUTLIER_SCALE
    return h


def make(name: str, seed: int = 0, device="cpu", **over) -> Workload:
    """Draw workload ``name`` (a key of ``SPECS``) with ``seed``.

    Keyword overrides (``batch``, ``n``, ``d``, ``dtype``, ``clusters``,
    ``k``, ``ratio``, ``frames``, ``frame_tokens``) shrink a workload for
    tests while keeping its recipe.
    """
    spec = dict(SPECS[name])
    spec.update(over)
    device = torch.device(device)
    batch, d = spec["batch"], spec["d"]
    dtype = _torch_dtype(spec["dtype"])
    # Structural draws (sequence lengths) come from a CPU generator so they do
    # not depend on the device the features are drawn on.
    cpu_gen = torch.Generator().manual_seed(1_000_003 * (seed + 1))
    if isinstance(spec["n"], tuple):
        lo, hi = spec["n"]
        seqlens = torch.randint(lo, hi + 1, (batch,), generator=cpu_gen).tolist()
    elif "frames" in spec:
        seqlens = [spec["frames"] * spec["frame_tokens"]] * batch
    else:
        seqlens = [spec["n"]] * batch
    total = sum(seqlens)

    gen = torch.Generator(device=device).manual_seed(seed)
    w1 = torch.randn(MLP_HIDDEN, d, generator=gen, device=device) / math.sqrt(d)
    w2 = torch.randn(d, MLP_HIDDEN, generator=gen, device=device) / math.sqrt(MLP_HIDDEN)

    x = torch.empty(total, d, dtype=dtype, device=device)
    x_pre = torch.empty(total, d, dtype=dtype, device=device)
    x_post = torch.empty(total, d, dtype=dtype, device=device)
    off = 0
    for n in seqlens:
        if n == 0:
            continue
        if "frames" in spec:
            h = _video(gen, spec["frames"], spec["frame_tokens"], d, spec["clusters"], spec["drift"], device)
        else:
            m = spec["clusters"]
            m = max(1, math.ceil(n / 64)) if m == "n/64" else m
            h = _clustered(gen, n, d, m, device)
        h = _outliers(gen, h, device)
        hp = torch.nn.functional.gelu(h @ w1.T) @ w2.T
        x_pre[off:off + n] = h.to(dtype)
        x_post[off:off + n] = hp.to(dtype)
        x[off:off + n] = (h + hp).to(dtype)
        off += n
    return Workload(name=name, x=x, x_pre=x_pre, x_post=x_post, seqlens=seqlens,
                    k=spec.get("k"), ratio=spec.get("ratio"), lam=(1, 3),
                    meta=dict(seed=seed, spec=spec))


def algorithmic_bytes(seqlens, ks, d, elem_bytes, aliased_pre=False):
    """Bytes one pass must move: read x, x', x'' (or x, x'' when x' aliases x),
    read and write the K kept rows, write K int32 indices."""
    streams = 2 if aliased_pre else 3
    n = sum(seqlens)
    k = sum(ks)
    return streams * n * d * elem_bytes + 2 * k * d * elem_bytes + 4 * k


# ---------------------------------------------------------------- encoder-MLP inputs
# The encoder's final-layer MLP (Eq. 5) run on the device: its input x', the
# residual stream it is added to, and seeded weights of the shape of a
# CLIP-ViT-L/14 block (D = 1024, hidden 4096).  x'' and x are *not* drawn
# here: the MLP kernels compute them.
MLP_SPECS = {
    # CLIP-ViT-L/14-336 (LLaVA-1.5's vision tower): QuickGELU in its MLP
    "clip_mlp576": dict(batch=64, n=576, d=1024, d_hidden=4096, clusters=32, k=192, act="quick_gelu",
                        d_proj=4096),
}


@dataclass
class MlpInputs:
    name: str
    x_pre: torch.Tensor    # [T, D] bf16: the MLP input x'
    resid: torch.Tensor    # [T, D] bf16: the residual stream (x = resid + x'')
    w1: torch.Tensor       # [d_hidden, D] bf16
    w2: torch.Tensor       # [D, d_hidden] bf16
    b1: torch.Tensor       # [d_hidden] fp32
    b2: torch.Tensor       # [D] fp32
    seqlens: list
    k: int
    act: str = "gelu"
    d_proj: int = 4096   # width of the projector's first layer (LLaVA-1.5: 1024 -> 4096)

    @property
    def total(self) -> int:
        return self.x_pre.shape[0]

    @property
    def batch(self) -> int:
        return len(self.seqlens)


def make_mlp(name: str = "clip_mlp576", seed: int = 0, device="cpu", **over) -> MlpInputs:
    """x' drawn with the cluster recipe above (1% activation outliers), the
    residual equal to x' (the recipe's x = x' + x''), W1 ~ N(0, 1/D),
    W2 ~ N(0, 1/d_hidden), biases ~ N(0, 0.02^2); all seeded.  Overrides:
    batch, n, d, d_hidden, clusters, k."""
    spec = dict(MLP_SPECS[name])
    spec.update(over)
    device = torch.device(device)
    batch, n, d, dh = spec["batch"], spec["n"], spec["d"], spec["d_hidden"]
    gen = torch.Generator(device=device).manual_seed(seed)
    x_pre = torch.empty(batch * n, d, dtype=torch.bfloat16, device=device)
    for b in range(batch):
        h = _outliers(gen, _clustered(gen, n, d, spec["clusters"], device), device)
        x_pre[b * n:(b + 1) * n] = h.to(torch.bfloat16)
    w1 = (torch.randn(dh, d, generator=gen, device=device) / math.sqrt(d)).to(torch.bfloat16)
    w2 = (torch.randn(d, dh, generator=gen, device=device) / math.sqrt(dh)).to(torch.bfloat16)
    b1 = 0.02 * torch.randn(dh, generator=gen, device=device)
    b2 = 0.02 * torch.randn(d, generator=gen, device=device)
    return MlpInputs(name=name, x_pre=x_pre, resid=x_pre, w1=w1, w2=w2, b1=b1, b2=b2, seqlens=[n] * batch,
                     k=spec["k"], act=spec.get("act", "gelu"), d_proj=spec.get("d_proj", 4096))


def make_projector(d: int, d_proj: int, seed: int = 0, device="cpu"):
    """Seeded weights of the projector's first layer: W_p ~ N(0, 1/D) bf16
    [d_proj, D] and a bias ~ N(0, 0.02^2) fp32 [d_proj]."""
    gen = torch.Generator(device=torch.device(device)).manual_seed(seed + 77)
    w = (torch.randn(d_proj, d, generator=gen, device=device) / math.sqrt(d)).to(torch.bfloat16)
    return w, 0.02 * torch.randn(d_proj, generator=gen, device=device)

