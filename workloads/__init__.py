"""Seeded synthetic workloads for the GreedyLore compression step.

This module only produces inputs: the shapes of the five benchmark
configurations and the per-worker gradients G_{i,t}.  It holds none of the
method's arithmetic, so both the CPU oracle (``oracle/``) and the CUDA path
(``paper_2507_08784_gb300``) can be fed from it without sharing any code.

Recipe (stands in for the paper's C4 / CIFAR / GLUE gradients, which are not
available): for every layer matrix of shape m x n

    G_{i,t} = S + c * Xi_{i,t} / sqrt(n),     S = U_b diag(s) V_b^T,

where U_b (m x rho) and V_b (n x rho) are orthonormal (QR of seeded Gaussian
matrices), s is the configuration's spectrum, S is shared by all workers and
steps, and Xi_{i,t} is i.i.d. N(0, 1), fresh per worker i and step t.  The
result is rounded to the configuration's gradient dtype (fp32 or bf16, round
to nearest even).  Shapes follow the paper's workloads: ResNet-18 conv
gradients reshaped out_ch x (in_ch*9) (Sec. 6.1, CIFAR pre-training) and
LLaMA-style decoder blocks (Sec. 6.1, C4 pre-training).
"""
from __future__ import annotations

import dataclasses
import math
from typing import Callable, List, Sequence, Tuple

import numpy as np

__all__ = [
    "Config", "CONFIGS", "config", "Problem", "make_problem",
    "gradients_numpy", "round_to_dtype_numpy", "gradients_torch",
]


@dataclasses.dataclass(frozen=True)
class Config:
    """One workload: the layer shapes and the compressor/optimizer settings."""
    name: str
    shapes: Tuple[Tuple[int, int], ...]   # (m, n) of each layer matrix, as the gradient is laid out
    N: int                                # simulated data-parallel workers
    r: int                                # compression rank
    basis_rank: int                       # k: 0 = full basis (paper-exact), else r <= k < min(m, n)
    tau: int                              # subspace refresh period
    steps: int
    grad_dtype: str                       # "f32" | "bf16"
    optimizer: str                        # "msgd" | "adam"
    lr: float
    beta1: float
    beta2: float
    eps: float
    spectrum: Callable[[int], float]      # s_k for k = 1..rho
    rho: int
    noise: float                          # c
    power_iters: int = 4
    master_seed: int = 0

    def matrix_elems(self) -> int:
        return sum(m * n for m, n in self.shapes)


def _resnet_stack():
    out = []
    for c in (64, 128, 256, 512):
        out += [(c, c * 9)] * 2
    return tuple(out)


def _decoder_stack(d, ffn, layers):
    per = [(d, d)] * 4 + [(ffn, d)] * 2 + [(d, ffn)]
    return tuple(per * layers)


CONFIGS = {
    # 1: one 256x128 fp32 matrix, N=4, r=4, refresh every 5 steps, MSGD.
    "cfg1_tiny": Config("cfg1_tiny", ((256, 128),), N=4, r=4, basis_rank=0, tau=5, steps=20,
                        grad_dtype="f32", optimizer="msgd", lr=0.01, beta1=0.9, beta2=0.0, eps=0.0,
                        spectrum=lambda k: 1.0 / k, rho=16, noise=0.05, master_seed=1001),
    # 2: ResNet-style conv-gradient stack, N=8, r=8, refresh every 50 steps, MSGD.
    "cfg2_resnet": Config("cfg2_resnet", _resnet_stack(), N=8, r=8, basis_rank=16, tau=50, steps=200,
                          grad_dtype="f32", optimizer="msgd", lr=0.01, beta1=0.9, beta2=0.0, eps=0.0,
                          spectrum=lambda k: k ** -1.5, rho=64, noise=0.02, master_seed=1002),
    # 3: 12-layer d=2048 / ffn=5632 decoder, bf16 gradients, N=8, r=32, Adam.
    "cfg3_llama_d2048": Config("cfg3_llama_d2048", _decoder_stack(2048, 5632, 12), N=8, r=32,
                               basis_rank=64, tau=100, steps=200, grad_dtype="bf16", optimizer="adam",
                               lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8,
                               spectrum=lambda k: 1.0 / k, rho=256, noise=0.01, master_seed=1003),
    # 4: one 4096x11008 bf16 matrix, refresh every step (refresh stress), N=8, r=128.
    "cfg4_refresh": Config("cfg4_refresh", ((4096, 11008),), N=8, r=128, basis_rank=128, tau=1, steps=50,
                           grad_dtype="bf16", optimizer="msgd", lr=0.01, beta1=0.9, beta2=0.0, eps=0.0,
                           spectrum=lambda k: math.exp(-k / 40.0), rho=512, noise=0.01, master_seed=1004),
    # 5: 8-layer d=4096 / ffn=11008 decoder, bf16 gradients, N=4, r=128, Adam.
    "cfg5_llama_d4096": Config("cfg5_llama_d4096", _decoder_stack(4096, 11008, 8), N=4, r=128,
                               basis_rank=256, tau=200, steps=100, grad_dtype="bf16", optimizer="adam",
                               lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8,
                               spectrum=lambda k: k ** -1.2, rho=512, noise=0.01, master_seed=1005),
}


def config(name: str, **overrides) -> Config:
    return dataclasses.replace(CONFIGS[name], **overrides)


@dataclasses.dataclass
class Problem:
    """The fixed low-rank part S of every layer matrix, as float64 factors."""
    cfg: Config
    Ub: List[np.ndarray]
    s: np.ndarray
    Vb: List[np.ndarray]
    seed: int

    def S(self, li: int) -> np.ndarray:
        return (self.Ub[li] * self.s[None, : self.Ub[li].shape[1]]) @ self.Vb[li].T


def _orthonormal(rng: np.random.Generator, rows: int, cols: int) -> np.ndarray:
    q, rr = np.linalg.qr(rng.standard_normal((rows, cols)))
    return q * np.sign(np.diag(rr))[None, :]


def make_problem(cfg: Config, seed: int | None = None) -> Problem:
    seed = cfg.master_seed if seed is None else seed
    Ub, Vb = [], []
    for li, (m, n) in enumerate(cfg.shapes):
        rng = np.random.default_rng([seed, 1, li])
        rho = min(cfg.rho, m, n)
        Ub.append(_orthonormal(rng, m, rho))
        Vb.append(_orthonormal(rng, n, rho))
    s = np.array([cfg.spectrum(k) for k in range(1, cfg.rho + 1)], dtype=np.float64)
    return Problem(cfg, Ub, s, Vb, seed)


def round_to_dtype_numpy(x: np.ndarray, dtype: str) -> np.ndarray:
    """Round to the gradient dtype (RNE) and return the exactly representable values as float64."""
    if dtype == "f32":
        return x.astype(np.float32).astype(np.float64)
    if dtype == "bf16":
        f = x.astype(np.float32)
        u = f.view(np.uint32).astype(np.uint64)
        lsb = (u >> 16) & 1
        u = ((u + 0x7FFF + lsb) >> 16) << 16
        return u.astype(np.uint32).view(np.float32).astype(np.float64)
    raise ValueError(dtype)


def gradients_numpy(prob: Problem, li: int, t: int, workers: Sequence[int] | None = None) -> np.ndarray:
    """G_{i,t} for layer li at step t, shape (N, m, n), float64 holding dtype-exact values."""
    cfg = prob.cfg
    m, n = cfg.shapes[li]
    S = prob.S(li)
    ws = range(cfg.N) if workers is None else workers
    out = np.empty((len(ws), m, n), dtype=np.float64)
    for slot, i in enumerate(ws):
        rng = np.random.default_rng([prob.seed, 2, li, t, i])
        out[slot] = S + cfg.noise * rng.standard_normal((m, n)) / math.sqrt(n)
    return round_to_dtype_numpy(out, cfg.grad_dtype)


def gradients_torch(prob: Problem, li: int, t: int, device="cuda", workers: Sequence[int] | None = None):
    """The same recipe generated on a torch device (for large benchmark inputs): a list of N
    tensors (m x n) in the configuration's dtype.  Uses torch's generator, so the noise
    differs from gradients_numpy; S is the same matrix."""
    import torch
    cfg = prob.cfg
    m, n = cfg.shapes[li]
    rho = prob.Ub[li].shape[1]
    Ub = torch.from_numpy(prob.Ub[li] * prob.s[None, :rho]).float().to(device)
    Vb = torch.from_numpy(prob.Vb[li]).float().to(device)
    S = Ub @ Vb.T
    dt = torch.float32 if cfg.grad_dtype == "f32" else torch.bfloat16
    gen = torch.Generator(device=device)
    out = []
    for i in (range(cfg.N) if workers is None else workers):
        gen.manual_seed((prob.seed * 1_000_003 + li * 10_007 + t * 101 + i) % (2 ** 63))
        noise = torch.randn(m, n, device=device, generator=gen)
        out.append((S + (cfg.noise / math.sqrt(n)) * noise).to(dt).contiguous())
    return out
