"""Seeded synthetic inputs shaped like the paper's multimodal workloads.

This module only draws random numbers and lays them out; it holds none of the
scoring arithmetic, so both the CUDA path's tests and the CPU oracle may use
it.  Every tensor is bf16, laid out as the library's boundary expects:

    qwin [R, layers, Hq,  W, d]   window queries (query w sits at N-W+w)
    k, v [R, layers, Hkv, N, d]   the prefill KV cache

Shapes follow the workloads the paper evaluates (Section 5, Appendix B):
LLaVA-style images (576 visual tokens), Qwen2-VL high-resolution images
(60x60 patch grid, GQA 7:1), 32-frame video and long GUI screenshots.  The
value structure stands in for the datasets, which are not available:

  gaussian  : i.i.d. N(0, 1)/sqrt(d) queries, keys and values
  lowrank   : per-head rank-8 shared subspace plus isotropic noise
  grid      : keys smooth over the 2-D patch grid (bilinear upsampled
              random field) plus noise
  video     : per-position AR(1) correlation 0.9 between consecutive frames
  heavytail : key norms Student-t (nu = 3) distributed

Planted evidence keys (per layer and kv-head, at the same positions in every
layer) point along the mean last-row query of the kv-head's query group,
scaled so that this mean query gives them a logit of exactly `plant_logit`
before bf16 rounding: k = plant_logit * sqrt(d) * q / |q|^2.
"""

from __future__ import annotations

import dataclasses
import math

import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    layers: int
    q_heads: int
    kv_heads: int
    head_dim: int
    seq_len: int
    window: int
    pool: int
    budgets: tuple
    requests: int
    visual: tuple          # [start, end) of the visual span
    kind: str
    planted: int           # planted evidence keys per (layer, kv-head)
    plant_run: int = 4     # planted keys come in runs of consecutive positions
    plant_logit: float = 4.0
    frame_tokens: int = 0  # video: tokens per frame
    grid: int = 0          # grid: patch-grid side
    config_id: int = 0

    @property
    def group(self) -> int:
        return self.q_heads // self.kv_heads

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)

    def bytes_model(self, budget: int) -> int:
        """Algorithmic HBM bytes of one step: K read once, the window
        queries read once, B rows of K and V gathered and written."""
        per_layer = (self.kv_heads * (self.seq_len * self.head_dim * 2
                                      + 4 * budget * self.head_dim * 2)
                     + self.q_heads * self.window * self.head_dim * 2)
        return self.requests * self.layers * per_layer

    def flops_model(self) -> int:
        """One pass of the window logits: 2 * Hq * W * N * d per layer."""
        return (2 * self.requests * self.layers * self.q_heads * self.window
                * self.seq_len * self.head_dim)


CONFIGS = {
    "tiny": Workload("tiny", 2, 4, 4, 64, 640, 32, 7, (64,), 1, (16, 592),
                     "gaussian", 3, plant_run=3, config_id=0),
    "llava": Workload("llava", 32, 32, 32, 128, 1024, 32, 7, (64, 128, 256), 1,
                      (8, 584), "lowrank", 8, config_id=1),
    "qwen-img": Workload("qwen-img", 28, 28, 4, 128, 4096, 32, 7, (128, 256, 512), 1,
                         (16, 3616), "grid", 16, grid=60, config_id=2),
    "video": Workload("video", 28, 28, 4, 128, 6528, 64, 7, (326, 652), 1,
                      (16, 16 + 32 * 196), "video", 8, frame_tokens=196, config_id=3),
    "gui": Workload("gui", 28, 28, 4, 128, 16384, 64, 7, (256, 1024), 4,
                    (16, 16 + 15872), "heavytail", 32, config_id=4),
}


@dataclasses.dataclass
class Inputs:
    qwin: torch.Tensor
    k: torch.Tensor
    v: torch.Tensor
    planted: torch.Tensor  # [R, Hkv, planted] positions (int64, ascending)


def _randn(shape, gen, device):
    return torch.randn(shape, generator=gen, device=device, dtype=torch.float32)


def _plant_positions(wl: Workload, gen, device) -> torch.Tensor:
    """Runs of plant_run consecutive positions inside the visual span, the
    runs spread apart; same positions in every layer of a (request, head).
    Video: the runs alternate between two distinct random frames."""
    R, H, n = wl.requests, wl.kv_heads, wl.planted
    if n == 0:
        return torch.zeros((R, H, 0), dtype=torch.int64, device=device)
    run = max(1, min(wl.plant_run, n))
    runs = -(-n // run)
    lo, hi = wl.visual
    ar = torch.arange(runs, device=device)
    if wl.kind == "video" and wl.frame_tokens:
        ft = wl.frame_tokens
        frames = (hi - lo) // ft
        per_frame = -(-runs // 2)
        slot = ft // per_frame
        assert slot >= run + 2, "frame too short for the planted runs"
        f0 = torch.randint(0, frames, (R, H, 1), generator=gen, device=device)
        f1 = (f0 + 1 + torch.randint(0, frames - 1, (R, H, 1), generator=gen,
                                     device=device)) % frames
        frame = torch.where((ar % 2) == 0, f0, f1)
        offs = torch.randint(0, slot - run, (R, H, runs), generator=gen, device=device)
        starts = lo + frame * ft + (ar // 2) * slot + offs
    else:
        slot = (hi - lo) // runs
        assert slot >= run + 2, "visual span too short for the planted runs"
        offs = torch.randint(0, slot - run, (R, H, runs), generator=gen, device=device)
        starts = lo + ar * slot + offs
    pos = starts.unsqueeze(-1) + torch.arange(run, device=device)
    pos = pos.reshape(R, H, runs * run)[..., :n]
    return torch.sort(pos, dim=-1).values


def _keys(wl: Workload, gen, device) -> torch.Tensor:
    R, Ly, H, N, d = wl.requests, wl.layers, wl.kv_heads, wl.seq_len, wl.head_dim
    if wl.kind == "gaussian":
        return _randn((R, Ly, H, N, d), gen, device) / math.sqrt(d)
    if wl.kind == "lowrank":
        rank = 8
        U = _randn((1, Ly, H, rank, d), gen, device) / math.sqrt(rank)
        A = _randn((R, Ly, H, N, rank), gen, device)
        noise = _randn((R, Ly, H, N, d), gen, device)
        return math.sqrt(0.5) * (A @ U) + math.sqrt(0.5) * noise
    if wl.kind == "grid":
        g = wl.grid
        lo, hi = wl.visual
        coarse = _randn((R * Ly * H, d, 7, 7), gen, device)
        field = torch.nn.functional.interpolate(coarse, size=(g, g), mode="bilinear",
                                                align_corners=True)
        field = field.reshape(R, Ly, H, d, g * g).transpose(-1, -2)
        k = _randn((R, Ly, H, N, d), gen, device)
        k[..., lo:lo + g * g, :] = 0.8 * field / field.std() + 0.6 * k[..., lo:lo + g * g, :]
        return k
    if wl.kind == "video":
        lo, hi = wl.visual
        ft = wl.frame_tokens
        frames = (hi - lo) // ft
        k = _randn((R, Ly, H, N, d), gen, device)
        vis = k[..., lo:lo + frames * ft, :].reshape(R, Ly, H, frames, ft, d)
        rho = 0.9
        for f in range(1, frames):
            vis[..., f, :, :] = rho * vis[..., f - 1, :, :] + math.sqrt(1 - rho * rho) * vis[..., f, :, :]
        k[..., lo:lo + frames * ft, :] = vis.reshape(R, Ly, H, frames * ft, d)
        return k
    if wl.kind == "heavytail":
        direction = _randn((R, Ly, H, N, d), gen, device)
        direction = direction / direction.norm(dim=-1, keepdim=True)
        z = _randn((R, Ly, H, N), gen, device)
        chi = _randn((R, Ly, H, N, 3), gen, device).pow(2).sum(-1)
        t = (z / torch.sqrt(chi / 3.0)).abs()
        norm = math.sqrt(d) * t / 1.1  # E|t_3| = 2*sqrt(3)/pi ~ 1.10
        return direction * norm.unsqueeze(-1)
    raise ValueError(wl.kind)


def generate(wl: Workload, seed: int = 0, device="cpu") -> Inputs:
    """Draw one batch of inputs for the workload (seed + config id)."""
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed) * 1000 + wl.config_id)
    R, Ly, Hq, H, N, W, d = (wl.requests, wl.layers, wl.q_heads, wl.kv_heads,
                             wl.seq_len, wl.window, wl.head_dim)
    scale = 1.0 / math.sqrt(d) if wl.kind == "gaussian" else 1.0
    qwin = _randn((R, Ly, Hq, W, d), gen, device) * scale
    k = _keys(wl, gen, device)
    v = _randn((R, Ly, H, N, d), gen, device) * scale
    planted = _plant_positions(wl, gen, device)
    if wl.planted:
        G = wl.group
        qlast = qwin[:, :, :, W - 1, :].reshape(R, Ly, H, G, d).mean(dim=3)
        qb = qlast.to(torch.bfloat16).float()
        kp = wl.plant_logit * math.sqrt(d) * qb / qb.pow(2).sum(-1, keepdim=True)
        idx = planted.unsqueeze(1).expand(R, Ly, H, wl.planted)
        k.scatter_(3, idx.unsqueeze(-1).expand(R, Ly, H, wl.planted, d),
                   kp.unsqueeze(3).expand(R, Ly, H, wl.planted, d).contiguous())
    return Inputs(qwin.to(torch.bfloat16).contiguous(), k.to(torch.bfloat16).contiguous(),
                  v.to(torch.bfloat16).contiguous(), planted)


def bf16_bits(t: torch.Tensor):
    """bf16 tensor -> numpy uint16 bit patterns (host copy)."""
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view("uint16")


# Hyper-parameter grid of the paper's ablation study (Sec. 5.3).  The
# component table switches E, L, T off in turn (all three off is the plain
# backbone score, all on the full method at m = 4, r = 5); the sensitivity
# tables take m in {0, 2, 4, 6, 8} at r = 5 and r in {0, 3, 5, 7, 9} at
# m = 4.  Those tables print for m = 0 the scores of the no-T row and for
# r = 0 those of the no-L row, so m = 0 and r = 0 are taken as those two
# component variants (by Eq. 6 read literally, r = 0 would give L = E
# instead).  Each distinct setting is listed once; fields not listed keep
# the context's values.
SWEEP_VARIANTS = (
    [dict(use_E=e, use_L=l, use_T=t, m=4, r=5)
     for e, l, t in ((1, 1, 1), (0, 0, 0), (1, 0, 1), (1, 1, 0), (0, 1, 1))]
    + [dict(m=m, r=5) for m in (2, 6, 8)]
    + [dict(m=4, r=r) for r in (3, 7, 9)]
)
