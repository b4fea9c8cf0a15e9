"""The seeded input generators: model layouts match the paper's models, seeds
are deterministic, column slices equal the full tensors, and the value
distributions are the configured ones."""
import math

import pytest
import torch

from paper_2607_21224_gb300 import workloads as wls


def test_model_layouts():
    r = wls.resnet50_cifar100()
    assert (r.N, len(r.tensors), r.W, r.K, r.T) == (23_712_932, 161, 8, 4, 16)
    t = wls.resnet50_tinyimagenet()
    assert (t.N, len(t.tensors), t.W, t.K, t.T, t.beta) == (23_917_832, 161, 16, 2, 32, 0.7)
    v = wls.vit_s16_cifar100()
    assert (v.N, len(v.tensors), v.grad_dtype) == (21_704_164, 152, "bf16")
    tiny = wls.tiny()
    assert (tiny.N, len(tiny.tensors), tiny.W, tiny.K, tiny.T) == (1 << 20, 8, 2, 2, 4)
    for wl in (r, t, v, tiny):
        assert all(s.numel % 4 == 0 for s in wl.tensors)
        offs = wl.offsets
        assert offs[0] == 0 and offs[-1] == wl.N and all(b > a for a, b in zip(offs, offs[1:]))


def test_resnet50_backbone_count():
    # the 1000-way ImageNet ResNet-50 has 25,557,032 parameters; swapping the
    # head to 100 classes removes (1000-100) * (2048+1) of them
    assert wls.Workload("x", 1, tuple(wls.resnet50_tensors(1000)), 1, 1).N == 25_557_032
    assert 25_557_032 - 900 * 2049 == 23_712_932


def test_sweep_points_respect_cap():
    pts = wls.sweep_points()
    assert len(pts) == 76
    assert (1 << 28, 32, 1) not in pts and (1 << 28, 16, 8) in pts
    assert all(12 * W * N <= wls.SWEEP_CAP_BYTES for N, W, _ in pts)
    assert wls.get("sweep_N1048576_W4_K2").W == 4


def test_theta0_deterministic_and_inits():
    wl = wls.resnet50_cifar100()
    a = wls.make_theta0(wl, 42)
    b = wls.make_theta0(wl, 42)
    assert torch.equal(a, b) and a.dtype == torch.float32 and a.numel() == wl.N
    assert not torch.equal(a, wls.make_theta0(wl, 123))
    offs = wl.offsets
    for k, s in enumerate(wl.tensors):
        x = a[offs[k]:offs[k + 1]]
        if s.init == "ones":
            assert torch.all(x == 1)
        elif s.init == "zeros":
            assert torch.all(x == 0)
        elif s.init == "kaiming_fan_out" and s.numel > 100_000:
            std = math.sqrt(2.0 / (s.shape[0] * s.shape[2] * s.shape[3]))
            assert abs(float(x.std()) / std - 1) < 0.02


def test_vit_truncated_normal():
    wl = wls.vit_s16_cifar100()
    a = wls.make_theta0(wl, 7)
    offs = wl.offsets
    for k, s in enumerate(wl.tensors):
        if s.init == "trunc_normal":
            x = a[offs[k]:offs[k + 1]]
            assert float(x.abs().max()) <= 0.04 + 1e-7


def test_grads_seeded_per_worker_and_step():
    wl = wls.tiny()
    g1 = wls.make_grads(wl, 1)
    assert torch.equal(g1, wls.make_grads(wl, 1))
    assert not torch.equal(g1, wls.make_grads(wl, 2))
    assert not torch.equal(g1[0], g1[1])
    assert abs(float(g1.std()) / 0.01 - 1) < 0.01
    part = wls.make_grads(wl, 3, columns=slice(1000, 1017))
    assert torch.equal(part, wls.make_grads(wl, 3)[:, 1000:1017])


def test_heavy_tail_fraction():
    wl = wls.Workload("ht", 2, tuple(wls.flat_tensors(400_000)), 2, 2, heavy_tail_p=0.01)
    g = wls.make_grads(wl, 1)
    frac = float((g.abs() > 0.02).float().mean())  # |N(0,1e-3)| > 20 sigma only if scaled
    assert 0.006 < frac < 0.012


def test_bf16_gradients():
    wl = wls.vit_s16_cifar100()
    g = wls.make_grads(wl, 1, columns=slice(0, 4096))
    assert g.dtype == torch.bfloat16 and g.shape == (8, 4096)


def test_seed_for_distinct():
    seeds = {wls.seed_for(42, "grad", i, t) for i in range(32) for t in range(1, 65)}
    assert len(seeds) == 32 * 64
    assert wls.seed_for(42, "init", 0) != wls.seed_for(42, "grad", 0)


def test_flat_points_by_name():
    wl = wls.get("flat_N1024_W3_K2_adamw_bf16")
    assert (wl.N, wl.W, wl.K, wl.T, wl.optimizer, wl.grad_dtype) == (1024, 3, 2, 4, "adamw", "bf16")
    assert wl.lr == 5e-4 and wl.weight_decay == 0.05 and wl.momentum == 0.0 and wl.state_arrays == 3
    sgd = wls.get("flat_N4096_W1_K4_sgd_f32")
    assert (sgd.N, sgd.W, sgd.optimizer, sgd.grad_dtype, sgd.momentum) == (4096, 1, "sgd", "f32", 0.9)
    for bad in ("flat_N4096_W1_K4_adam_f32", "flat_N4096_W1_K4_sgd_f16"):
        with pytest.raises(KeyError):
            wls.get(bad)
