"""Workload recipes and seeded generators.

Stand-ins for the paper's Qwen2.5 weights and captured activation statistics
(Sec. 4), which are not available here: every array is drawn from a seeded
torch generator on the requested device, with the shapes of the Qwen2.5
projections and the value distributions of the five workloads below.

Recipe (one module of shape rows x cols, out x in):
  * W ~ N(0, 0.02^2). A seed-chosen 1% of input channels (at least one) are
    outliers: x8 scaled Gaussians for the small single-matrix workload, and
    0.02*8*t_4 (Student-t, nu = 4) for the Qwen-shaped workloads.
  * W0 = RTN-INT4 symmetric, groups of 128 along the input dimension:
    s = fp16(max|w| / 7), q = clamp(rint(w / s), -8, 7), W0 = q*s (stored in
    the workload's weight dtype).
  * a_j = mean over 1024 tokens of x_j^2 with x_j ~ N(0, s_j^2),
    s_j ~ LogNormal(0, 1) (per input channel, Sec. 3.2 activation diagonal).
  * Fisher diagonal (PF workloads) F_ij ~ LogNormal(0, 1.5) per element;
    blend weights w_act = lam_a / mean(a), w_fisher = lam_F / mean(F).
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np
import torch

MODULE_ORDER = ("q_proj", "k_proj", "v_proj", "o_proj", "gate_proj", "up_proj", "down_proj")


def layer_shapes(hidden: int, inter: int, kv: int) -> List[Tuple[str, int, int]]:
    """(name, rows=out, cols=in) of the seven linear modules of a Qwen2.5 layer."""
    return [
        ("q_proj", hidden, hidden),
        ("k_proj", kv, hidden),
        ("v_proj", kv, hidden),
        ("o_proj", hidden, hidden),
        ("gate_proj", inter, hidden),
        ("up_proj", inter, hidden),
        ("down_proj", hidden, inter),
    ]


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    description: str
    layers: int
    shapes: Tuple[Tuple[str, int, int], ...]
    w_dtype: str            # "f32" | "bf16"
    C: int = 64
    P: int = 4
    b: int = 4
    S: int = 4096
    variant: int = 0        # 0 = U, 1 = PF
    scale_mode: int = 0     # 0 = power-of-two exponent, 1 = fp16 scale
    rates: Tuple[float, ...] = (0.162,)
    outlier: str = "t4"     # "x8" | "t4"
    blend: Tuple[float, float] = (1.0, 0.0)
    seed: int = 0

    @property
    def weights_per_layer(self) -> int:
        return sum(r * c for _, r, c in self.shapes)

    @property
    def tiles_per_layer(self) -> int:
        return self.weights_per_layer // self.C


_QWEN3B = tuple(layer_shapes(2048, 11008, 256))
_QWEN7B = tuple(layer_shapes(3584, 18944, 512))
_QWEN32B = tuple(layer_shapes(5120, 27648, 1024))

WORKLOADS: Dict[str, Workload] = {
    "single_256x512": Workload(
        name="single_256x512",
        description="single linear 256x512 FP32, 1% x8 outlier columns, RTN-INT4 g128, "
                    "C=64 P=4 b=4 S=256, FP16 scale, AWSRC-U at 0.162 bpw",
        layers=1, shapes=(("linear", 256, 512),), w_dtype="f32", S=256, scale_mode=1,
        outlier="x8"),
    "qwen2.5-3b_layer": Workload(
        name="qwen2.5-3b_layer",
        description="one Qwen2.5-3B-shaped layer (7 modules, 77,070,336 weights) BF16, "
                    "t4 outlier columns, RTN-INT4 g128, C=64 P=4 b=4 S=4096, AWSRC-U at 0.162 bpw",
        layers=1, shapes=_QWEN3B, w_dtype="bf16"),
    "qwen2.5-3b_stack": Workload(
        name="qwen2.5-3b_stack",
        description="36 Qwen2.5-3B-shaped layers, AWSRC-U at 0.162 bpw",
        layers=36, shapes=_QWEN3B, w_dtype="bf16"),
    "qwen2.5-7b_stack_pf": Workload(
        name="qwen2.5-7b_stack_pf",
        description="28 Qwen2.5-7B-shaped layers, AWSRC-P_F 0.5/0.5 blend, prefixes at "
                    "0.05/0.10/0.162/0.25 bpw",
        layers=28, shapes=_QWEN7B, w_dtype="bf16", variant=1,
        rates=(0.05, 0.10, 0.162, 0.25), blend=(0.5, 0.5)),
    "qwen2.5-32b_stack": Workload(
        name="qwen2.5-32b_stack",
        description="64 Qwen2.5-32B-shaped layers streamed one at a time, AWSRC-U at 0.162 bpw "
                    "plus AWSRC-P_F prefixes",
        layers=64, shapes=_QWEN32B, w_dtype="bf16"),
}


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed & 0x7FFF_FFFF_FFFF_FFFF)
    return g


def module_seed(base: int, layer: int, module: int) -> int:
    """Distinct, reproducible stream per (workload seed, layer, module)."""
    return (base * 1_000_003 + layer * 1009 + module * 7 + 12345) & 0x7FFF_FFFF


def rtn_int4_g128(W: torch.Tensor, group: int = 128) -> torch.Tensor:
    """RTN-INT4 symmetric backbone of Eq. 1, per (row, group of 128 inputs; the
    last group of a row may be shorter). Returns the float32 reconstruction q*s
    (exact in float32)."""
    rows, cols = W.shape
    ng = (cols + group - 1) // group
    w = torch.zeros(rows, ng * group, dtype=torch.float32, device=W.device)
    w[:, :cols] = W.float()
    w = w.reshape(rows, ng, group)
    amax = w.abs().amax(dim=-1, keepdim=True)
    s = (amax / 7.0).to(torch.float16).float()
    safe = torch.where(s > 0, s, torch.ones_like(s))
    q = torch.clamp(torch.round(w / safe), -8, 7)
    q = torch.where(s > 0, q, torch.zeros_like(q))
    return (q * s).reshape(rows, ng * group)[:, :cols].contiguous()


def activation_moments(cols: int, gen: torch.Generator, device, tokens: int = 1024,
                       chunk: int = 256) -> torch.Tensor:
    """a_j = mean over `tokens` draws of x_j^2, x_j ~ N(0, s_j^2), s_j ~ LogNormal(0, 1)."""
    s = torch.exp(torch.randn(cols, generator=gen, device=device, dtype=torch.float32))
    acc = torch.zeros(cols, device=device, dtype=torch.float64)
    for t0 in range(0, tokens, chunk):
        n = min(chunk, tokens - t0)
        x = torch.randn(n, cols, generator=gen, device=device, dtype=torch.float32) * s
        acc += (x.double() ** 2).sum(0)
    return (acc / tokens).float()


def make_module(rows: int, cols: int, *, seed: int, device="cpu", w_dtype: str = "bf16",
                outlier: str = "t4", fisher: bool = False,
                blend: Tuple[float, float] = (1.0, 0.0)) -> Dict[str, object]:
    """Draw one module's W, W0, activation moments (and Fisher diagonal)."""
    g = _gen(device, seed)
    W = torch.randn(rows, cols, generator=g, device=device, dtype=torch.float32) * 0.02
    n_out = max(1, int(round(0.01 * cols)))
    oc = torch.randperm(cols, generator=g, device=device)[:n_out]
    if outlier == "x8":
        W[:, oc] *= 8.0
    else:
        z = torch.randn(rows, n_out, generator=g, device=device, dtype=torch.float32)
        chi = (torch.randn(rows, n_out, 4, generator=g, device=device, dtype=torch.float32) ** 2).sum(-1)
        W[:, oc] = 0.02 * 8.0 * z / torch.sqrt(chi / 4.0)
    tdt = torch.float32 if w_dtype == "f32" else torch.bfloat16
    W = W.to(tdt)
    W0 = rtn_int4_g128(W).to(tdt)
    act = activation_moments(cols, g, device)
    out = {"W": W, "W0": W0, "act": act, "rows": rows, "cols": cols,
           "w_act": 1.0, "w_fisher": 0.0, "fisher": None}
    if fisher:
        F = torch.exp(1.5 * torch.randn(rows, cols, generator=g, device=device, dtype=torch.float32))
        out["fisher"] = F
        lam_a, lam_f = blend
        # normalisers computed in double, rounded once to the float the ABI carries
        out["w_act"] = float(np.float32(lam_a / act.double().mean().item()))
        out["w_fisher"] = float(np.float32(lam_f / F.double().mean().item()))
    return out


def make_layer(wl: Workload, layer: int = 0, device="cpu",
               modules: Optional[Sequence[int]] = None) -> List[Dict[str, object]]:
    """All (or the selected) modules of one layer of workload `wl`."""
    out = []
    for mi, (name, rows, cols) in enumerate(wl.shapes):
        if modules is not None and mi not in modules:
            continue
        m = make_module(rows, cols, seed=module_seed(wl.seed, layer, mi), device=device,
                        w_dtype=wl.w_dtype, outlier=wl.outlier, fisher=(wl.variant == 1),
                        blend=wl.blend)
        m["name"] = name
        out.append(m)
    return out


def total_weights(wl: Workload) -> int:
    return wl.layers * wl.weights_per_layer


def describe(wl: Workload) -> str:
    return f"{wl.name}: {wl.layers} layer(s) x {len(wl.shapes)} modules, " \
           f"{total_weights(wl):,} weights, {wl.layers * wl.tiles_per_layer:,} tiles, S={wl.S}"


__all__ = ["MODULE_ORDER", "Workload", "WORKLOADS", "layer_shapes", "make_module", "make_layer",
           "rtn_int4_g128", "activation_moments", "module_seed", "total_weights", "describe"]
