"""Seeded synthetic parameter sets shaped like the paper's merge workloads.

The paper merges RL experts of Qwen2.5-7B-Instruct and DeepSeek-R1-Distill-
Qwen-1.5B (App. F, backbones and experts); those checkpoints are not
available here, so these generators stand in for them with the same tensor
shapes and the update statistics the workload configurations state.  This
module draws random numbers and builds tensors; it holds none of the merge
method's arithmetic.  Both the CUDA tests and the oracle consume its output.

Recipes (all seeded; every tensor has its own generator seed):
* base weights        N(0, 0.02^2), rounded once to the base dtype
* RL update           N(0, std^2) with a Bernoulli(rate) subset replaced by
                      Laplace(0, b) (inverse-CDF sampling)
* checkpoint          bf16(theta_0 + delta): the fine-tuned weights as stored
* density-sweep delta bf16(N(0, 1e-3^2) + 1e-3 * t_3), t_3 = Z / sqrt(chi2_3 / 3),
                      plus 1000 entries moved onto the rho-threshold value
* merge experts       |N(0, std^2)| with sign + w.p. p_i ~ U(0.4, 0.6) per
                      expert, 0.5 % Laplace(0, 5e-3) outliers
"""
from __future__ import annotations

from typing import List, Tuple

import torch

# (rows, cols, is_1d) per tensor
Shape = Tuple[int, int, bool]

QWEN = {
    # DeepSeek-R1-Distill-Qwen-1.5B / Qwen2.5-1.5B geometry (tied embedding)
    "qwen1.5b": dict(layers=28, hidden=1536, kv=256, inter=8960, vocab=151936, lm_head=False),
    # Qwen2.5-7B geometry (separate lm_head)
    "qwen7b": dict(layers=28, hidden=3584, kv=512, inter=18944, vocab=152064, lm_head=True),
}


def qwen_shapes(name: str = "qwen1.5b", layers: int | None = None, scale: int = 1) -> List[Shape]:
    """Tensor list of a Qwen2-style decoder: embedding, then per layer
    q, k, v, o, gate, up, down and two RMSNorm vectors, then lm_head.
    ``scale`` divides every width (for small test sets)."""
    g = QWEN[name]
    h, kv, it, vocab = g["hidden"] // scale, g["kv"] // scale, g["inter"] // scale, g["vocab"] // scale
    L = g["layers"] if layers is None else layers
    out: List[Shape] = [(vocab, h, False)]
    for _ in range(L):
        out += [(h, h, False), (h, kv, False), (h, kv, False), (h, h, False),
                (h, it, False), (h, it, False), (it, h, False), (1, h, True), (1, h, True)]
    if g["lm_head"]:
        out.append((vocab, h, False))
    return out


def n_params(shapes: List[Shape]) -> int:
    return sum(r * c for r, c, _ in shapes)


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed & 0x7FFFFFFFFFFFFFFF)
    return g


def tensor_seed(seed: int, tensor_id: int, role: int) -> int:
    """Per-tensor seed; role 0 is the base, role 1 + i expert i."""
    return (seed * 1_000_003 + tensor_id * 9_176 + role * 7_919_911) & 0x7FFFFFFFFFFFFFFF


def _view(t: torch.Tensor, shape: Shape) -> torch.Tensor:
    r, c, one = shape
    return t.reshape(c) if one else t.reshape(r, c)


def normal(shape: Shape, std: float, gen: torch.Generator, device) -> torch.Tensor:
    r, c, _ = shape
    return torch.randn(r * c, generator=gen, device=device, dtype=torch.float32) * std


def laplace_(x: torch.Tensor, rate: float, b: float, gen: torch.Generator) -> torch.Tensor:
    """Replace a Bernoulli(rate) subset of x by Laplace(0, b) draws."""
    pick = torch.rand(x.numel(), generator=gen, device=x.device) < rate
    u = torch.rand(x.numel(), generator=gen, device=x.device) - 0.5
    # keep 2|u| < 1 so the inverse CDF stays finite (rand may return exactly 0)
    lap = -b * torch.sign(u) * torch.log1p(-(2.0 * u.abs()).clamp(max=1.0 - 2.0 ** -24))
    x[pick] = lap[pick]
    return x


def base_weights(shapes: List[Shape], seed: int, device="cpu", dtype=torch.bfloat16,
                 std: float = 0.02) -> List[torch.Tensor]:
    out = []
    for q, s in enumerate(shapes):
        g = _gen(tensor_seed(seed, q, 0), device)
        out.append(_view(normal(s, std, g, device).to(dtype), s))
    return out


def rl_delta(shape: Shape, gen: torch.Generator, device, std=5e-4, rate=0.005, b=5e-3) -> torch.Tensor:
    return laplace_(normal(shape, std, gen, device), rate, b, gen)


def rl_update_set(shapes: List[Shape], seed: int, device="cpu", std=5e-4, rate=0.005, b=5e-3,
                  base_dtype=torch.bfloat16):
    """(theta_0, theta_1): base weights and one RL checkpoint bf16(theta_0 + delta)."""
    th0 = base_weights(shapes, seed, device, base_dtype)
    th1 = []
    for q, (s, w) in enumerate(zip(shapes, th0)):
        g = _gen(tensor_seed(seed, q, 1), device)
        d = rl_delta(s, g, device, std, rate, b)
        th1.append(_view((w.reshape(-1).float() + d).to(base_dtype), s))
    return th0, th1


def tiny_set(seed: int = 0, device="cpu", rows=1024, cols=1024, K=2):
    """1024 x 1024 fp32 base ~ N(0, 0.02^2); K fp32 task vectors
    N(0, 1e-3^2) with 1 % Laplace(0, 1e-2) entries."""
    s = (rows, cols, False)
    th0 = base_weights([s], seed, device, torch.float32)
    taus = []
    for i in range(K):
        g = _gen(tensor_seed(seed, 0, 1 + i), device)
        taus.append([_view(rl_delta(s, g, device, 1e-3, 0.01, 1e-2), s)])
    return th0, taus


def merge_experts(shapes: List[Shape], seed: int, K: int = 8, device="cpu", std=5e-4,
                  rate=0.005, b=5e-3):
    """K fp32 task vectors with a per-expert sign bias p_i ~ U(0.4, 0.6)."""
    gp = _gen(tensor_seed(seed, 10_007, 99), "cpu")
    p = (0.4 + 0.2 * torch.rand(K, generator=gp)).tolist()
    taus = []
    for i in range(K):
        row = []
        for q, s in enumerate(shapes):
            g = _gen(tensor_seed(seed, q, 1 + i), device)
            mag = normal(s, std, g, device).abs_()
            sign = torch.where(torch.rand(mag.numel(), generator=g, device=device) < p[i], 1.0, -1.0)
            row.append(_view(laplace_(mag * sign, rate, b, g), s))
        taus.append(row)
    return taus, p


def density_sweep_delta(seed: int, rho: float, device="cpu", rows=4096, cols=14336,
                        n_ties: int = 1000):
    """bf16 delta N(0, 1e-3^2) + 1e-3 t_3 with n_ties entries moved onto the
    pre-injection rho-threshold magnitude (drawn among the entries below it,
    with a random sign), so the threshold is shared by >= n_ties + 1 entries."""
    s = (rows, cols, False)
    g = _gen(tensor_seed(seed, 0, 1), device)
    n = rows * cols
    z = torch.randn(n, generator=g, device=device)
    chi = (torch.randn(3, n, generator=g, device=device) ** 2).sum(0)
    t3 = torch.randn(n, generator=g, device=device) / torch.sqrt(chi / 3.0)
    d = (z * 1e-3 + 1e-3 * t3).to(torch.bfloat16).float()
    k = int(rho * n + 0.5)
    if 0 < k < n:
        mag = d.abs()
        thr = torch.topk(mag, k, sorted=False).values.min()
        below = torch.nonzero(mag < thr).flatten()
        if below.numel() >= n_ties:
            pick = below[torch.randperm(below.numel(), generator=g, device=device)[:n_ties]]
            sgn = torch.where(torch.rand(n_ties, generator=g, device=device) < 0.5, -1.0, 1.0)
            d[pick] = thr * sgn
    return _view(d.to(torch.bfloat16), s)
