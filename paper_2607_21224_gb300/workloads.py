"""Seeded synthetic workloads for the CPDP hot path.

Holds the parameter layouts of the paper's models (ResNet-50 with a 100- or
200-way head, ViT-S/16 with a 100-way head), their initialisations, and the
per-(worker, step) synthetic gradients. The paper trains on CIFAR-100 and
TinyImageNet (Sec. 5.2); only the parameter shapes matter to the optimizer and
reconcile path, so seeded random tensors of those shapes stand in for the real
models and data. None of CPDP's arithmetic lives here: both the CUDA path and
the CPU oracle receive the very same tensors from these generators.

Seeds: every tensor comes from its own torch.Generator seeded by
``seed_for(base, tag, a, b)``; the paper's seeds are 42, 123 and 777 (Sec. 5.1).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch

PAPER_SEEDS = (42, 123, 777)


@dataclass(frozen=True)
class TensorSpec:
    name: str
    shape: tuple[int, ...]
    init: str  # kaiming_fan_out | kaiming_fan_in | ones | zeros | normal | trunc_normal
    std: float = 0.0

    @property
    def numel(self) -> int:
        return math.prod(self.shape)


# ---------------------------------------------------------------------------
# model layouts
# ---------------------------------------------------------------------------
def resnet50_tensors(num_classes: int) -> list[TensorSpec]:
    """ResNet-50 (bottleneck blocks 3-4-6-3, 7x7 stem) parameters in
    registration order: convolutions, batch-norm scale/shift, classifier."""
    t: list[TensorSpec] = []

    def conv(name, cout, cin, k):
        t.append(TensorSpec(f"{name}.weight", (cout, cin, k, k), "kaiming_fan_out"))

    def bn(name, c):
        t.append(TensorSpec(f"{name}.weight", (c,), "ones"))
        t.append(TensorSpec(f"{name}.bias", (c,), "zeros"))

    conv("conv1", 64, 3, 7)
    bn("bn1", 64)
    inplanes = 64
    for li, (planes, blocks) in enumerate([(64, 3), (128, 4), (256, 6), (512, 3)], start=1):
        for b in range(blocks):
            p = f"layer{li}.{b}"
            conv(f"{p}.conv1", planes, inplanes, 1)
            bn(f"{p}.bn1", planes)
            conv(f"{p}.conv2", planes, planes, 3)
            bn(f"{p}.bn2", planes)
            conv(f"{p}.conv3", planes * 4, planes, 1)
            bn(f"{p}.bn3", planes * 4)
            if b == 0:
                conv(f"{p}.downsample.0", planes * 4, inplanes, 1)
                bn(f"{p}.downsample.1", planes * 4)
            inplanes = planes * 4
    t.append(TensorSpec("fc.weight", (num_classes, 2048), "kaiming_fan_in"))
    t.append(TensorSpec("fc.bias", (num_classes,), "zeros"))
    return t


def vit_s16_tensors(num_classes: int, tokens: int = 197, dim: int = 384, depth: int = 12,
                    mlp: int = 1536) -> list[TensorSpec]:
    """ViT-S/16 (12 blocks, width 384, 6 heads, MLP 1536, 196 patches + class
    token) parameters: class token, position embedding, patch projection,
    blocks, final norm, head."""
    tn = "trunc_normal"
    t = [TensorSpec("cls_token", (1, 1, dim), tn, 0.02),
         TensorSpec("pos_embed", (1, tokens, dim), tn, 0.02),
         TensorSpec("patch_embed.proj.weight", (dim, 3, 16, 16), tn, 0.02),
         TensorSpec("patch_embed.proj.bias", (dim,), "zeros")]
    for b in range(depth):
        p = f"blocks.{b}"
        t += [TensorSpec(f"{p}.norm1.weight", (dim,), "ones"),
              TensorSpec(f"{p}.norm1.bias", (dim,), "zeros"),
              TensorSpec(f"{p}.attn.qkv.weight", (3 * dim, dim), tn, 0.02),
              TensorSpec(f"{p}.attn.qkv.bias", (3 * dim,), "zeros"),
              TensorSpec(f"{p}.attn.proj.weight", (dim, dim), tn, 0.02),
              TensorSpec(f"{p}.attn.proj.bias", (dim,), "zeros"),
              TensorSpec(f"{p}.norm2.weight", (dim,), "ones"),
              TensorSpec(f"{p}.norm2.bias", (dim,), "zeros"),
              TensorSpec(f"{p}.mlp.fc1.weight", (mlp, dim), tn, 0.02),
              TensorSpec(f"{p}.mlp.fc1.bias", (mlp,), "zeros"),
              TensorSpec(f"{p}.mlp.fc2.weight", (dim, mlp), tn, 0.02),
              TensorSpec(f"{p}.mlp.fc2.bias", (dim,), "zeros")]
    t += [TensorSpec("norm.weight", (dim,), "ones"),
          TensorSpec("norm.bias", (dim,), "zeros"),
          TensorSpec("head.weight", (num_classes, dim), tn, 0.02),
          TensorSpec("head.bias", (num_classes,), "zeros")]
    return t


def flat_tensors(N: int, count: int = 1, std: float = 0.05) -> list[TensorSpec]:
    """`count` equal flat tensors (the last takes the remainder), N(0, std) init."""
    base = N // count
    sizes = [base] * (count - 1) + [N - base * (count - 1)]
    return [TensorSpec(f"p{k}", (n,), "normal", std) for k, n in enumerate(sizes)]


# ---------------------------------------------------------------------------
# workloads
# ---------------------------------------------------------------------------
@dataclass(frozen=True)
class Workload:
    name: str
    W: int
    tensors: tuple[TensorSpec, ...]
    K: int
    T: int                      # mini-batch steps per epoch
    grad_dtype: str = "f32"     # "f32" | "bf16"
    grad_std: float = 1e-3
    heavy_tail_p: float = 0.0   # probability that a gradient entry is scaled x100
    lr: float = 0.1
    momentum: float = 0.9
    weight_decay: float = 5e-4
    beta: float = 0.5
    alpha: float = 1.0
    optimizer: str = "sgd"      # "sgd" (momentum SGD) | "adamw"
    adam_beta1: float = 0.9
    adam_beta2: float = 0.999
    adam_eps: float = 1e-8
    notes: str = field(default="", compare=False)
    data: str = field(default="", compare=False)  # what the synthetic inputs stand in for

    @property
    def N(self) -> int:
        return sum(t.numel for t in self.tensors)

    @property
    def offsets(self) -> list[int]:
        o = [0]
        for t in self.tensors:
            o.append(o[-1] + t.numel)
        return o

    @property
    def torch_grad_dtype(self) -> torch.dtype:
        return torch.float32 if self.grad_dtype == "f32" else torch.bfloat16

    @property
    def grad_bytes(self) -> int:
        return 4 if self.grad_dtype == "f32" else 2

    @property
    def state_arrays(self) -> int:
        """[W][N] float32 arrays each optimizer step reads and writes: the
        replicas and the momentum buffers (SGD), plus the second moments (AdamW)."""
        return 3 if self.optimizer == "adamw" else 2

    def hyper(self) -> dict:
        return dict(lr=self.lr, momentum=self.momentum, weight_decay=self.weight_decay, K=self.K,
                    beta=self.beta, alpha=self.alpha)


def tiny() -> Workload:
    return Workload("tiny", W=2, tensors=tuple(flat_tensors(1 << 20, 8, 0.05)), K=2, T=4,
                    grad_std=0.01, notes="8 x 131072 flat tensors",
                    data="8 flat tensors of 131,072, init N(0, 0.05), gradients N(0, 0.01)")


def resnet50_cifar100() -> Workload:
    return Workload("resnet50_cifar100", W=8, tensors=tuple(resnet50_tensors(100)), K=4, T=16,
                    data="ResNet-50/CIFAR-100 parameter shapes (161 tensors), Kaiming init, gradients N(0, 1e-3)")


def vit_s16_cifar100() -> Workload:
    return Workload("vit_s16_cifar100", W=8, tensors=tuple(vit_s16_tensors(100)), K=4, T=16,
                    grad_dtype="bf16",
                    data="ViT-S/16/CIFAR-100 parameter shapes (152 tensors), truncated-normal init, "
                         "bf16 gradients N(0, 1e-3)")


def vit_s16_cifar100_adamw() -> Workload:
    """ViT-S/16 with the paper's own optimizer for it (Sec. 5.2, Table 3): AdamW,
    lr 5e-4, weight decay 0.05 (decoupled); PyTorch's default betas and eps."""
    return Workload("vit_s16_cifar100_adamw", W=8, tensors=tuple(vit_s16_tensors(100)), K=4, T=16,
                    grad_dtype="bf16", lr=5e-4, weight_decay=0.05, momentum=0.0, optimizer="adamw",
                    data="ViT-S/16/CIFAR-100 parameter shapes (152 tensors), truncated-normal init, "
                         "bf16 gradients N(0, 1e-3), AdamW")


def resnet50_tinyimagenet() -> Workload:
    return Workload("resnet50_tinyimagenet", W=16, tensors=tuple(resnet50_tensors(200)), K=2, T=32,
                    heavy_tail_p=0.01, beta=0.7,
                    data="ResNet-50/TinyImageNet parameter shapes (161 tensors), Kaiming init, gradients "
                         "N(0, 1e-3) with 1 % of entries x100")


def sweep_point(N: int, W: int, K: int) -> Workload:
    return Workload(f"sweep_N{N}_W{W}_K{K}", W=W, tensors=tuple(flat_tensors(N, 1, 0.05)), K=K, T=2 * K,
                    data="one flat tensor, init N(0, 0.05), gradients N(0, 1e-3)")


def flat_point(N: int, W: int, K: int, optimizer: str = "sgd", grad_dtype: str = "f32") -> Workload:
    """One flat tensor of N parameters like a sweep point, with either
    optimizer (AdamW at the ViT-S settings) and either gradient type."""
    kw = dict(lr=5e-4, weight_decay=0.05, momentum=0.0, optimizer="adamw") if optimizer == "adamw" else {}
    return Workload(f"flat_N{N}_W{W}_K{K}_{optimizer}_{grad_dtype}", W=W, tensors=tuple(flat_tensors(N, 1, 0.05)),
                    K=K, T=2 * K, grad_dtype=grad_dtype,
                    data=f"one flat tensor, init N(0, 0.05), {grad_dtype} gradients N(0, 1e-3), {optimizer}", **kw)


SWEEP_N = (1 << 20, 1 << 24, 1 << 26, 1 << 28)
SWEEP_W = (2, 4, 8, 16, 32)
SWEEP_K = (1, 2, 4, 8)
SWEEP_CAP_BYTES = 64 * 10**9  # replicas + gradients + momentum (12 bytes per element)


def sweep_points() -> list[tuple[int, int, int]]:
    return [(N, W, K) for N in SWEEP_N for W in SWEEP_W for K in SWEEP_K
            if 12 * W * N <= SWEEP_CAP_BYTES]


NAMED = {
    "tiny": tiny,
    "resnet50_cifar100": resnet50_cifar100,
    "vit_s16_cifar100": vit_s16_cifar100,
    "vit_s16_cifar100_adamw": vit_s16_cifar100_adamw,
    "resnet50_tinyimagenet": resnet50_tinyimagenet,
}


def get(name: str) -> Workload:
    if name in NAMED:
        return NAMED[name]()
    if name.startswith("sweep_"):
        kv = {p[0]: int(p[1:]) for p in name[len("sweep_"):].split("_")}
        return sweep_point(kv["N"], kv["W"], kv["K"])
    if name.startswith("flat_"):
        n, w, k, opt, gd = name[len("flat_"):].split("_")
        if opt not in ("sgd", "adamw") or gd not in ("f32", "bf16"):
            raise KeyError(name)
        return flat_point(int(n[1:]), int(w[1:]), int(k[1:]), opt, gd)
    raise KeyError(name)


# ---------------------------------------------------------------------------
# seeded generators
# ---------------------------------------------------------------------------
_TAGS = {"init": 1, "grad": 2}


def seed_for(base: int, tag: str, a: int = 0, b: int = 0) -> int:
    """A 63-bit seed from (base seed, what is drawn, two indices)."""
    x = (base * 0x9E3779B97F4A7C15 + _TAGS[tag] * 0xBF58476D1CE4E5B9
         + (a + 1) * 0x94D049BB133111EB + (b + 1) * 0xD6E8FEB86659FD93)
    x ^= x >> 31
    return x & ((1 << 63) - 1)


def _generator(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _init_tensor(spec: TensorSpec, gen: torch.Generator, device) -> torch.Tensor:
    n = spec.numel
    if spec.init == "ones":
        return torch.ones(n, device=device)
    if spec.init == "zeros":
        return torch.zeros(n, device=device)
    if spec.init == "kaiming_fan_out":      # conv weight (cout, cin, kh, kw)
        std = math.sqrt(2.0 / (spec.shape[0] * math.prod(spec.shape[2:])))
    elif spec.init == "kaiming_fan_in":     # linear weight (out, in)
        std = math.sqrt(2.0 / spec.shape[1])
    elif spec.init in ("normal", "trunc_normal"):
        std = spec.std
    else:
        raise ValueError(spec.init)
    x = torch.randn(n, generator=gen, device=device)
    if spec.init == "trunc_normal":         # resample outside +-2 sigma
        bad = x.abs() > 2.0
        while bool(bad.any()):
            x[bad] = torch.randn(int(bad.sum()), generator=gen, device=device)
            bad = x.abs() > 2.0
    return x.mul_(std)


def make_theta0(wl: Workload, seed: int = 42, device="cpu") -> torch.Tensor:
    """Initial parameters theta0, float32 [N], tensor by tensor in layout order."""
    parts = [_init_tensor(s, _generator(device, seed_for(seed, "init", k)), device)
             for k, s in enumerate(wl.tensors)]
    return torch.cat(parts).contiguous()


def make_grads(wl: Workload, step: int, seed: int = 42, device="cpu", out: torch.Tensor | None = None,
               columns: slice | None = None) -> torch.Tensor:
    """Gradients of mini-batch `step` (1-based) for all W workers, [W][N] in the
    workload's gradient dtype: N(0, grad_std) per entry, from one generator per
    (worker, step); with heavy_tail_p > 0 each entry is independently scaled by
    100 with that probability. `columns` returns only that slice of every row
    (drawn in full, then sliced, so the values equal the full tensor's)."""
    N = wl.N
    cols = slice(0, N) if columns is None else columns
    width = len(range(N)[cols])
    if out is None:
        out = torch.empty((wl.W, width), dtype=wl.torch_grad_dtype, device=device)
    for i in range(wl.W):
        gen = _generator(device, seed_for(seed, "grad", i, step))
        row = torch.randn(N, generator=gen, device=device).mul_(wl.grad_std)
        if wl.heavy_tail_p > 0:
            hit = torch.rand(N, generator=gen, device=device) < wl.heavy_tail_p
            row = torch.where(hit, row * 100.0, row)
        out[i].copy_(row[cols])
    return out
