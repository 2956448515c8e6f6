"""Seeded synthetic workloads shaped like the paper's long-context settings.

This module only draws inputs; it contains none of the method's arithmetic and
is shared by the CUDA path, the oracle-backed tests and the benchmark.  The
paper evaluates on LongBench-v2 and RULER with Llama-3.1-8B, Qwen3-8B and
Mistral-7B (§4 and the experimental-protocol appendix); neither the datasets
nor the checkpoints are available, so every tensor here is synthetic, with the
KV shapes of Llama-3-8B (32 layers, 32 query / 8 KV heads, d = 128) and
Llama-3-70B (80 layers, 64 / 8).

Every tensor slice (sequence, layer, tensor kind) is drawn from its own
``torch.Generator`` seeded by a fixed mix of (seed, config, kind, sequence,
layer), so a single layer can be regenerated alone with identical bytes on the
same device type.  CPU and CUDA generators produce different streams; tests
that compare the CUDA path with the oracle draw on one device and hand the
oracle the very bytes the GPU consumed.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import torch


@dataclass(frozen=True)
class Workload:
    name: str
    B: int          # sequences
    L: int          # layers
    Hq: int         # query heads
    H: int          # KV heads
    n: int          # context length
    d: int          # head dim
    w: int          # observation window
    keep: tuple     # kept fraction (num, den): B_live = H * floor(n * num / den)
    kind: str       # input recipe, see draw_layer
    decode_steps: int = 0
    description: str = ""
    keep_sweep: tuple = field(default_factory=tuple)

    @property
    def G(self) -> int:
        return self.Hq // self.H

    @property
    def units(self) -> int:
        return self.B * self.L * self.H

    @property
    def B_live(self) -> int:
        return self.H * ((self.n * self.keep[0]) // self.keep[1])

    def with_(self, **kw) -> "Workload":
        d = dict(self.__dict__)
        d.update(kw)
        return Workload(**d)


WORKLOADS = {
    "C1": Workload("C1", B=1, L=1, Hq=32, H=8, n=4096, d=128, w=32, keep=(1, 10),
                   kind="planted",
                   description="single layer, GQA 32/8, d=128, context 4096, window 32, "
                               "budget 10%; N(0,1) K/V/Q with 16 planted keys per head x4"),
    "C2": Workload("C2", B=1, L=32, Hq=32, H=8, n=32768, d=128, w=64, keep=(1, 10),
                   kind="lowrank",
                   description="Llama-3-8B-shaped KV, 32 layers, context 32768, window 64, "
                               "budget 1/10; planted retrieval keys and a rank-4 value "
                               "component whose strength varies across heads"),
    "C3": Workload("C3", B=1, L=32, Hq=32, H=8, n=131072, d=128, w=64, keep=(1, 10),
                   kind="zipf",
                   description="Llama-3-8B-shaped KV, 32 layers, context 131072, window 64, "
                               "budget 1/10; Gaussian keys mixed with 64 Zipf(1.1)-weighted "
                               "planted keys per head"),
    "C4": Workload("C4", B=8, L=32, Hq=32, H=8, n=32768, d=128, w=64, keep=(1, 10),
                   kind="lowrank", decode_steps=256,
                   description="batch 8 x context 32768, compression then 256 decode steps "
                               "with fresh N(0,1) queries, budget 1/10"),
    "C5": Workload("C5", B=1, L=80, Hq=64, H=8, n=131072, d=128, w=128, keep=(1, 10),
                   kind="student_t", keep_sweep=((1, 4), (1, 10), (1, 20)),
                   description="Llama-3-70B-shaped KV, 80 layers, 64/8 heads, context 131072, "
                               "window 128, Student-t(3) keys and values, budgets 1/4, 1/10, "
                               "1/20"),
}

_KIND_ID = {"K": 1, "V": 2, "Q": 3, "P": 4, "S": 5, "q": 6}
_LOWRANK_LEVELS = (0.0, 0.25, 0.5, 1.0, 2.0, 4.0, 8.0, 16.0)


def _gen(device, seed: int, wl: Workload, kind: str, b: int, l: int, extra: int = 0):
    g = torch.Generator(device=device)
    cfg_id = int(wl.name[1:]) if wl.name[1:].isdigit() else 0
    mix = (((seed * 1_000_003 + cfg_id) * 1_000_033 + _KIND_ID[kind]) * 1_000_037 + b)
    mix = (mix * 1_000_039 + l) * 1_000_081 + extra
    g.manual_seed(mix % (2 ** 63 - 1))
    return g


def _student_t(shape, g, device, nu: int = 3) -> torch.Tensor:
    z = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
    chi2 = torch.zeros(shape, device=device, dtype=torch.float32)
    for _ in range(nu):
        chi2 += torch.randn(shape, generator=g, device=device, dtype=torch.float32) ** 2
    return z / torch.sqrt(chi2 / nu)


def draw_layer(wl: Workload, b: int, l: int, seed: int = 0, device="cpu"):
    """K, V [H][n][d] and Q_obs [Hq][w][d] (bf16) of sequence b, layer l.

    Recipes (per KV head h; N(0,1) unless stated):
      planted   : 16 planted keys alpha*u_h with alpha = 4
      lowrank   : V += s_{l,h} * Z U_h (Z [n][4] ~ N(0,1), U_h [4][d] ~ N(0,1/4),
                  s in {0, .25, .5, 1, 2, 4, 8, 16} permuted per layer) and 16
                  planted keys with alpha = 4
      zipf      : 64 planted keys with alpha_i = 8 i^-1.1, i = 1..64
      student_t : K and V Student-t with 3 degrees of freedom, no planted keys
    u_h is the mean of the G*w observation query rows of KV head h rescaled to
    norm sqrt(d); planted keys sit at distinct positions drawn uniformly from
    [0, n - w).
    """
    H, n, d, w, G = wl.H, wl.n, wl.d, wl.w, wl.G
    gq = _gen(device, seed, wl, "Q", b, l)
    Q = torch.randn((wl.Hq, w, d), generator=gq, device=device, dtype=torch.float32)
    gk = _gen(device, seed, wl, "K", b, l)
    gv = _gen(device, seed, wl, "V", b, l)
    if wl.kind == "student_t":
        K = _student_t((H, n, d), gk, device)
        V = _student_t((H, n, d), gv, device)
    else:
        K = torch.randn((H, n, d), generator=gk, device=device, dtype=torch.float32)
        V = torch.randn((H, n, d), generator=gv, device=device, dtype=torch.float32)
    Qb = Q.to(torch.bfloat16)
    if wl.kind in ("planted", "lowrank", "zipf"):
        gp = _gen(device, seed, wl, "P", b, l)
        count = 64 if wl.kind == "zipf" else 16
        count = min(count, n - w)
        for h in range(H):
            u = Qb[h * G:(h + 1) * G].float().reshape(G * w, d).mean(0)
            u = u * (d ** 0.5) / u.norm().clamp_min(1e-30)
            pos = torch.randperm(n - w, generator=gp, device=device)[:count]
            if wl.kind == "zipf":
                alpha = 8.0 * torch.arange(1, count + 1, device=device,
                                           dtype=torch.float32) ** -1.1
            else:
                alpha = torch.full((count,), 4.0, device=device)
            K[h, pos] = alpha[:, None] * u[None, :]
    if wl.kind == "lowrank":
        gs = _gen(device, seed, wl, "S", b, l)
        levels = torch.tensor(_LOWRANK_LEVELS, device=device, dtype=torch.float32)
        strength = levels[torch.randperm(8, generator=gs, device=device)[
            torch.arange(H, device=device) % 8]]
        Z = torch.randn((H, n, 4), generator=gs, device=device, dtype=torch.float32)
        U = torch.randn((H, 4, d), generator=gs, device=device, dtype=torch.float32) * 0.5
        V += strength[:, None, None] * torch.bmm(Z, U)
    return K.to(torch.bfloat16), V.to(torch.bfloat16), Qb


def draw(wl: Workload, seed: int = 0, device="cpu", layers=None, batch=None):
    """Stacked inputs K, V [B'][L'][H][n][d], Q_obs [B'][L'][Hq][w][d] for the
    selected sequences (default all) and layers (default all)."""
    layers = list(range(wl.L)) if layers is None else list(layers)
    batch = list(range(wl.B)) if batch is None else list(batch)
    shp_kv = (len(batch), len(layers), wl.H, wl.n, wl.d)
    K = torch.empty(shp_kv, dtype=torch.bfloat16, device=device)
    V = torch.empty(shp_kv, dtype=torch.bfloat16, device=device)
    Q = torch.empty((len(batch), len(layers), wl.Hq, wl.w, wl.d), dtype=torch.bfloat16,
                    device=device)
    for bi, b in enumerate(batch):
        for li, l in enumerate(layers):
            k, v, q = draw_layer(wl, b, l, seed, device)
            K[bi, li].copy_(k)
            V[bi, li].copy_(v)
            Q[bi, li].copy_(q)
            del k, v, q
    return K, V, Q


def draw_decode_queries(wl: Workload, step: int, seed: int = 0, device="cpu", layers=None,
                        batch=None) -> torch.Tensor:
    """Fresh N(0,1) decode queries q [B'][L'][Hq][d] (bf16) for one decode step."""
    layers = list(range(wl.L)) if layers is None else list(layers)
    batch = list(range(wl.B)) if batch is None else list(batch)
    q = torch.empty((len(batch), len(layers), wl.Hq, wl.d), dtype=torch.bfloat16, device=device)
    for bi, b in enumerate(batch):
        for li, l in enumerate(layers):
            g = _gen(device, seed, wl, "q", b, l, extra=step)
            q[bi, li] = torch.randn((wl.Hq, wl.d), generator=g, device=device,
                                    dtype=torch.float32).to(torch.bfloat16)
    return q


def bf16_bits(t: torch.Tensor):
    """uint16 numpy view of a bf16 tensor's bytes (copied to host)."""
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view("uint16")
