"""Seeded synthetic workloads for the structured-pruned CONV forward path.

This module holds the layer shapes of the benchmark workloads and the seeded
generators of their tensors.  It holds none of the pruning method's arithmetic:
the CUDA path and the CPU oracle both draw their inputs from here and from
nowhere else.

The paper measures on ImageNet-trained AlexNet / ResNet-50 layers (Sec. 5,
Tables 1-3); no dataset, weight or mask is available here, so seeded tensors
with the paper's layer shapes and these distributions stand in for them:

* W ~ N(0, 2/fan_in) (He init, variance 2/fan_in, fan_in = Cg*KT*KH*KW),
* x = ReLU(N(0, 1)) (about half zeros),
* bias ~ N(0, 0.01) read as variance 0.01 (std 0.1),

drawn in fp32 from one ``torch.Generator`` per layer in the order W, bias, x,
then rounded to bf16 (W, x); the bias stays fp32.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional

import torch

COL_NONE, COL_SHAPE, COL_CHANNEL = 0, 1, 2
COLKIND_NAMES = {COL_NONE: "none", COL_SHAPE: "shape", COL_CHANNEL: "channel"}


def retained(frac: float, groups: int) -> int:
    """Number of groups a retained fraction keeps: floor(frac*groups + 0.5)."""
    return int(math.floor(frac * groups + 0.5))


def pruning_rate(col_sparsity: float, row_sparsity: float = 0.0) -> float:
    """Weight pruning rate of a layer with the given GEMM column and row sparsity.

    Dense weights over kept weights: 1 / ((1 - col) * (1 - row)).  This is the
    bookkeeping behind the "pruning rate" rows of Tables 1 and 2.
    """
    return 1.0 / ((1.0 - col_sparsity) * (1.0 - row_sparsity))


@dataclasses.dataclass(frozen=True)
class ConvShape:
    """A CONV layer: input NCDHW (t=1 for 2-D), F filters in `groups` groups."""

    n: int
    c: int
    h: int
    w: int
    f: int
    kh: int
    kw: int
    sh: int = 1
    sw: int = 1
    ph: int = 0
    pw: int = 0
    groups: int = 1
    t: int = 1
    kt: int = 1
    st: int = 1
    pt: int = 0

    @property
    def cg(self) -> int:
        return self.c // self.groups

    @property
    def fg(self) -> int:
        return self.f // self.groups

    @property
    def taps(self) -> int:
        return self.kt * self.kh * self.kw

    @property
    def k(self) -> int:
        """GEMM columns: Cg * KT * KH * KW."""
        return self.cg * self.taps

    @property
    def ot(self) -> int:
        return (self.t + 2 * self.pt - self.kt) // self.st + 1

    @property
    def oh(self) -> int:
        return (self.h + 2 * self.ph - self.kh) // self.sh + 1

    @property
    def ow(self) -> int:
        return (self.w + 2 * self.pw - self.kw) // self.sw + 1

    @property
    def plane(self) -> int:
        """Output pixels per image and filter: OT*OH*OW."""
        return self.ot * self.oh * self.ow

    @property
    def m(self) -> int:
        """GEMM rows on the pixel side: N*OT*OH*OW."""
        return self.n * self.plane

    @property
    def is3d(self) -> bool:
        return self.t != 1 or self.kt != 1

    def desc16(self) -> List[int]:
        """n c t h w f groups kt kh kw st sh sw pt ph pw."""
        return [self.n, self.c, self.t, self.h, self.w, self.f, self.groups,
                self.kt, self.kh, self.kw, self.st, self.sh, self.sw,
                self.pt, self.ph, self.pw]

    def w_shape(self):
        if self.is3d:
            return (self.f, self.cg, self.kt, self.kh, self.kw)
        return (self.f, self.cg, self.kh, self.kw)

    def x_shape(self):
        if self.is3d:
            return (self.n, self.c, self.t, self.h, self.w)
        return (self.n, self.c, self.h, self.w)

    def y_shape(self):
        if self.is3d:
            return (self.n, self.f, self.ot, self.oh, self.ow)
        return (self.n, self.f, self.oh, self.ow)

    def with_batch(self, n: int) -> "ConvShape":
        return dataclasses.replace(self, n=n)


@dataclasses.dataclass(frozen=True)
class Layer:
    """A pruned layer: shape, retained filter fraction, column kind and fraction."""

    name: str
    shape: ConvShape
    filt_frac: float
    colkind: int
    col_frac: float
    seed: int

    @property
    def col_groups(self) -> int:
        """Number of column groups: K columns (shape-wise) or Cg channels."""
        if self.colkind == COL_CHANNEL:
            return self.shape.cg
        return self.shape.k

    @property
    def k_filters(self) -> int:
        return retained(self.filt_frac, self.shape.f)

    @property
    def k_cols(self) -> int:
        if self.colkind == COL_NONE:
            return self.col_groups
        return retained(self.col_frac, self.col_groups)

    @property
    def n_cols(self) -> int:
        """Retained GEMM columns K' after channel expansion."""
        if self.colkind == COL_CHANNEL:
            return self.k_cols * self.shape.taps
        return self.k_cols

    def retained_flops(self) -> float:
        """2 * M * K' * (retained filters): multiply-adds on retained weights.

        With groups, each retained filter sees K' columns, so the count is
        2 * M * F' * K' whatever the split of F' over conv groups.
        """
        return 2.0 * self.shape.m * self.k_filters * self.n_cols

    def dense_flops(self) -> float:
        return 2.0 * self.shape.m * self.shape.f * self.shape.k


def gen_tensors(shape: ConvShape, seed: int, device: str = "cpu") -> Dict[str, torch.Tensor]:
    """Seeded W (bf16), bias (fp32) and x (bf16) for one layer."""
    g = torch.Generator().manual_seed(int(seed))
    fan_in = shape.cg * shape.taps
    W = (torch.randn(shape.w_shape(), generator=g, dtype=torch.float32)
         * math.sqrt(2.0 / fan_in)).to(torch.bfloat16)
    bias = torch.randn((shape.f,), generator=g, dtype=torch.float32) * 0.1
    x = torch.relu(torch.randn(shape.x_shape(), generator=g, dtype=torch.float32)).to(torch.bfloat16)
    out = {"W": W, "bias": bias, "x": x}
    if device != "cpu":
        out = {k: v.to(device) for k, v in out.items()}
    return out


def gen_dual(shape: ConvShape, seed: int, scale: float = 0.01) -> torch.Tensor:
    """Seeded ADMM dual U (bf16), same shape as W, N(0, scale^2)."""
    g = torch.Generator().manual_seed(int(seed) + 7919)
    return (torch.randn(shape.w_shape(), generator=g, dtype=torch.float32) * scale).to(torch.bfloat16)


def gen_admm_state(shape: ConvShape, seed: int, dtype=torch.float32) -> Dict[str, torch.Tensor]:
    """Seeded ADMM state of one layer in training precision: W ~ N(0, 2/fan_in)
    and the scaled dual U ~ N(0, 0.1 * 2/fan_in), drawn in fp32 in that order
    (then cast to `dtype`)."""
    g = torch.Generator().manual_seed(int(seed) + 104729)
    fan_in = shape.cg * shape.taps
    sd = math.sqrt(2.0 / fan_in)
    W = torch.randn(shape.w_shape(), generator=g, dtype=torch.float32) * sd
    U = torch.randn(shape.w_shape(), generator=g, dtype=torch.float32) * (sd * math.sqrt(0.1))
    return {"W": W.to(dtype), "U": U.to(dtype)}


def gen_integer_weights(shape: ConvShape, seed: int, lo: int = -3, hi: int = 3) -> torch.Tensor:
    """Small-integer weights (exact in bf16; group sums exact in any order) for tie tests."""
    g = torch.Generator().manual_seed(int(seed))
    return torch.randint(lo, hi + 1, shape.w_shape(), generator=g).to(torch.bfloat16)


# ---------------------------------------------------------------------------
# The five workloads (layer shapes follow the paper's networks).
# ---------------------------------------------------------------------------

def single2d() -> List[Layer]:
    """One 2-D layer: N8 C64 32x32 F64 3x3 s1 p1, shape-wise keeping 50% of 576 columns."""
    s = ConvShape(n=8, c=64, h=32, w=32, f=64, kh=3, kw=3, ph=1, pw=1)
    return [Layer("single2d", s, 1.0, COL_SHAPE, 0.5, seed=0)]


def alexnet() -> List[Layer]:
    """AlexNet CONV1-5 at batch 128 (Tables 1-2 layer family), filter-wise plus
    shape-wise pruning at per-layer retained fractions 1.0/0.5/0.25/0.2/0.2,
    each applied to both filters and columns."""
    N = 128
    shapes = [
        ConvShape(n=N, c=3, h=227, w=227, f=96, kh=11, kw=11, sh=4, sw=4),
        ConvShape(n=N, c=96, h=27, w=27, f=256, kh=5, kw=5, ph=2, pw=2, groups=2),
        ConvShape(n=N, c=256, h=13, w=13, f=384, kh=3, kw=3, ph=1, pw=1),
        ConvShape(n=N, c=384, h=13, w=13, f=384, kh=3, kw=3, ph=1, pw=1, groups=2),
        ConvShape(n=N, c=384, h=13, w=13, f=256, kh=3, kw=3, ph=1, pw=1, groups=2),
    ]
    fracs = [1.0, 0.5, 0.25, 0.2, 0.2]
    return [Layer(f"conv{i + 1}", s, fr, COL_SHAPE, fr, seed=100 + i)
            for i, (s, fr) in enumerate(zip(shapes, fracs))]


def resnet50() -> List[Layer]:
    """ResNet-50 bottleneck CONV shapes (Table 3 family) at batch 64, stride 1,
    'same' padding; filter-wise 50% plus channel-wise 50%."""
    N = 64
    spec = []
    for hw, base in ((56, 64), (28, 128), (14, 256), (7, 512)):
        cin = 64 if base == 64 else base * 2
        spec += [(hw, cin, base, 1), (hw, base, base * 4, 1), (hw, base * 4, base, 1), (hw, base, base, 3)]
    layers = []
    for i, (hw, cin, cout, k) in enumerate(spec):
        p = k // 2
        s = ConvShape(n=N, c=cin, h=hw, w=hw, f=cout, kh=k, kw=k, ph=p, pw=p)
        layers.append(Layer(f"r{hw}_{cin}x{cout}_{k}x{k}", s, 0.5, COL_CHANNEL, 0.5, seed=200 + i))
    return layers


def c3d() -> List[Layer]:
    """C3D-style 3-D layer: N8 C128 T8 28x28 F256 3x3x3 p1, shape-wise keeping 30%."""
    s = ConvShape(n=8, c=128, t=8, h=28, w=28, f=256, kt=3, kh=3, kw=3, pt=1, ph=1, pw=1)
    return [Layer("c3d", s, 1.0, COL_SHAPE, 0.3, seed=300)]


SWEEP_COL_FRACS = (1.0, 0.5, 0.25, 0.1, 0.05)
SWEEP_FILT_FRACS = (1.0, 0.5)


def sweep(col_fracs=SWEEP_COL_FRACS, filt_fracs=SWEEP_FILT_FRACS) -> List[Layer]:
    """One large 2-D layer N128 C256 28x28 F512 3x3 p1 at several densities."""
    s = ConvShape(n=128, c=256, h=28, w=28, f=512, kh=3, kw=3, ph=1, pw=1)
    return [Layer(f"sweep_f{ff:g}_c{cf:g}", s, ff, COL_SHAPE, cf, seed=400)
            for ff in filt_fracs for cf in col_fracs]


WORKLOADS = {
    "single2d": single2d,
    "alexnet": alexnet,
    "resnet50": resnet50,
    "c3d": c3d,
    "sweep": sweep,
}


def get(name: str) -> List[Layer]:
    return WORKLOADS[name]()


def subset_layer(layer: Layer, n: int, name: Optional[str] = None) -> Layer:
    """Same layer at a smaller batch (for oracle-sized parity cases)."""
    return dataclasses.replace(layer, shape=layer.shape.with_batch(n), name=name or layer.name)
