"""Host logic of bench.py that runs without a GPU: algorithmic byte counts, the
clock summary, the max-over-ranks reduction (2 gloo ranks on CPU), and the
reference arm (the fp64 oracle timed on the metric's workload)."""
import argparse
import json
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
from paper_2607_21224_gb300 import workloads as wls


def test_byte_counts_resnet50_w8():
    wl = wls.resnet50_cifar100()
    N = 23_712_932
    assert wl.N == N
    # per parameter and worker: theta, buf, g read (12 B); theta, buf written (8 B)
    assert bench.local_step_bytes(8, N, 4) == 20 * 8 * N == 3_794_069_120
    # per parameter: 20 B per worker + theta_ref and v read and written (16 B)
    assert bench.reconcile_bytes(8, N, 4) == (20 * 8 + 16) * N == 4_173_476_032
    assert bench.cycle_bytes(8, N, 4, 4) == 3 * 3_794_069_120 + 4_173_476_032


def test_byte_counts_bf16_gradients():
    assert bench.local_step_bytes(8, 100, 2) == 18 * 8 * 100
    assert bench.reconcile_bytes(8, 100, 2) == (18 * 8 + 16) * 100
    assert bench.cycle_bytes(2, 10, 1, 4) == bench.reconcile_bytes(2, 10, 4)


def test_summarize_clocks_window_and_reasons():
    rows = [
        "2026/12/02 10:00:00.000, 1000, 2070, 300.0, 0x0, Not Active, Not Active, Not Active, Not Active",
        "2026/12/02 10:00:01.000, 1900, 2070, 900.0, 0x4, Not Active, Not Active, Not Active, Active",
        "2026/12/02 10:00:01.100, 1950, 2070, 950.0, 0x0, Not Active, Not Active, Not Active, Not Active",
        "2026/12/02 10:00:05.000, 800, 2070, 200.0, 0x0, Active, Not Active, Not Active, Not Active",
    ]
    from datetime import datetime
    t0 = datetime(2026, 12, 2, 10, 0, 0, 900000).timestamp()
    t1 = datetime(2026, 12, 2, 10, 0, 1, 200000).timestamp()
    s = bench.summarize_clocks("\n".join(rows), t0, t1)
    assert s["samples"] == 2 and s["window"] == "timed region"
    assert s["sm_mhz"] == 1925.0 and s["sm_max_mhz"] == 2070.0
    assert s["reasons"] == ["sw_power_cap"]
    whole = bench.summarize_clocks("\n".join(rows), None, None)
    assert whole["samples"] == 4 and "hw_slowdown" in whole["reasons"]
    assert bench.summarize_clocks("", None, None)["samples"] == 0


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench.barrier(None)
        got = bench.max_over_ranks(10.0 + rank, None)
        assert bench.dist_env() == (rank, world, rank)
        out[rank] = got
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_gloo_two_ranks():
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(2, port, out), nprocs=2, join=True)
        assert dict(out) == {0: 11.0, 1: 11.0}


def test_max_over_ranks_single_process_is_identity():
    assert bench.max_over_ranks(3.5) == 3.5


def test_reference_arm_prints_contract_line(capsys):
    bench.main(["--impl", "reference", "--workload", "tiny", "--steps", "2", "--warmup", "3",
                "--ref-step-seconds", "0.02"])
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in line, key
    assert line["impl"] == "reference" and line["unit"] == "GB/s" and line["value"] > 0
    assert line["steps"] == 2 and line["warmup"] == 3 and line["config"]["workload"] == "tiny"
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] == 1
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["value"] == line["value"]
    # the GPU arm prints the same config for the same arguments
    args = argparse.Namespace(method="cpdp", state_reconcile=False, no_pdl=False, reconcile_staging=0,
                              reconcile_shuffle=False)
    assert line["config"] == bench.arm_config(wls.get("tiny"), args)


@pytest.mark.parametrize("method,ss", [("localsgd", True), ("ddp", False)])
def test_reference_arm_follows_method(capsys, method, ss):
    argv = ["--impl", "reference", "--workload", "tiny", "--steps", "1", "--warmup", "3", "--ref-step-seconds",
            "0.01", "--method", method] + (["--state-reconcile"] if ss else [])
    bench.main(argv)
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["config"]["method"] == method and line["config"]["state_reconcile"] == ss
    wl = wls.get("tiny")
    assert line["config"]["bytes_per_step"] == bench.cycle_bytes(wl.W, wl.N, wl.K, 4, method)


def test_reference_arm_silent_on_nonzero_rank(capsys, monkeypatch):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    bench.main(["--impl", "reference", "--workload", "tiny", "--steps", "1", "--warmup", "3"])
    assert capsys.readouterr().out == ""


def test_warmup_floor(monkeypatch):
    seen = {}
    monkeypatch.setattr(bench, "run_reference", lambda a: seen.setdefault("w", a.warmup))
    bench.main(["--impl", "reference", "--warmup", "1"])
    assert seen["w"] == 3


def test_ncu_traffic_requires_matching_source(tmp_path, monkeypatch):
    assert bench.ncu_traffic("no_such_kernel") is None


def test_floor_skips_what_the_floor_kernel_cannot_move():
    """No floor (rather than a failed launch after the timed region) for other
    methods or for N not a multiple of 4; decided before any device work."""
    import argparse
    for name, method in (("flat_N1027_W2_K2_sgd_f32", "cpdp"), ("flat_N1024_W2_K2_sgd_f32", "ddp")):
        args = argparse.Namespace(method=method, warmup=3, steps=4)
        assert bench.run_floor(args, wls.get(name), None, None, None, None, None) is None


def test_kernel_source_hash_ignores_comments_not_code(tmp_path, monkeypatch):
    """The committed traffic figures are keyed on the kernels' code: a comment
    or layout edit keeps the key, a code edit changes it."""
    csrc = tmp_path / "paper_2607_21224_gb300" / "csrc"
    csrc.mkdir(parents=True)
    real = bench.ROOT / "paper_2607_21224_gb300" / "csrc"
    for name in ("cpdp_kernels.cuh", "cpdp_shapes.cuh"):
        (csrc / name).write_text((real / name).read_text())
    monkeypatch.setattr(bench, "ROOT", tmp_path)
    base = bench.kernel_source_sha()
    shapes = csrc / "cpdp_shapes.cuh"
    text = shapes.read_text()
    shapes.write_text("// a new comment\n/* and a\n block */\n" + text.replace("\n", "\n  ", 3))
    assert bench.kernel_source_sha() == base
    shapes.write_text(text.replace("kGradChunksManyWorkers = 8", "kGradChunksManyWorkers = 9"))
    assert bench.kernel_source_sha() != base
    assert bench.strip_comments("a // c\nb /* x\ny */ c") == "a b c"


def test_l2_note_is_truthful():
    assert bench.workload_config(wls.resnet50_cifar100())["l2"].startswith("inputs larger than L2")
    assert bench.workload_config(wls.tiny())["l2"].startswith("working set") and bench.needs_l2_flush(wls.tiny())
    assert not bench.needs_l2_flush(wls.resnet50_cifar100())


def test_method_byte_counts():
    W, N = 8, 1000
    assert bench.sync_bytes(W, N, 4, "cpdp") == (20 * W + 16) * N
    assert bench.sync_bytes(W, N, 4, "localsgd") == 20 * W * N == bench.sync_bytes(W, N, 4, "ddp")
    assert bench.cycle_bytes(W, N, 4, 4, "ddp") == 4 * 20 * W * N
    assert bench.cycle_bytes(W, N, 4, 4, "localsgd") == 4 * 20 * W * N
    assert bench.cycle_bytes(W, N, 4, 4) == 3 * 20 * W * N + (20 * W + 16) * N


def test_adamw_byte_counts():
    W, N = 8, 1000
    assert bench.local_step_bytes(W, N, 4, 3) == 28 * W * N
    assert bench.reconcile_bytes(W, N, 2, 3) == ((24 + 2) * W + 16) * N
    wl = wls.vit_s16_cifar100_adamw()
    assert wl.state_arrays == 3 and wl.optimizer == "adamw" and wl.lr == 5e-4 and wl.weight_decay == 0.05


def test_cpu_baseline_splits_local_and_reconcile():
    """The CPU baseline reports the oracle's seconds per local step and per
    reconcile (scaled to the full N) beside the K-cycle figure."""
    wl = wls.get("tiny")
    cb = bench.cpu_baseline(wl, target_s=0.2)
    assert cb["kind"] == "oracle" and cb["cores"] == 1 and cb["value"] > 0
    ps = cb["per_step"]
    assert set(ps) == {"local_step", "reconcile"}
    for v in ps.values():
        assert v["s_full_N"] > 0 and v["GB_s"] > 0


def test_sweep_cpu_baseline_scales_a_window_to_the_full_point():
    """A sweep point's oracle figure comes from an instance of at most 2^18
    columns with its seconds scaled to the point's N."""
    wl = wls.sweep_point(1 << 20, 2, 2)
    cb = bench.sweep_cpu_baseline(wl, 0.1)
    assert cb["kind"] == "oracle" and cb["cores"] == 1 and cb["value"] > 0
    want = bench.cycle_bytes(2, 1 << 20, 2, 4) / (cb["value"] * 1e9)
    assert abs(cb["s_per_cycle_full_N"] - want) <= 1e-3 * want + 1e-4
    assert "262144 of its 1048576 columns" in cb["sample"]


@pytest.mark.parametrize("gd", ["f32", "bf16"])
@pytest.mark.parametrize("opt", ["sgd", "adamw"])
@pytest.mark.parametrize("W", [1, 3, 8])
def test_floor_rows_move_the_launch_bytes(opt, W, gd):
    """The floor kernel, given the rows floor_rows picks, moves exactly the
    algorithmic bytes of the launch it stands for (n elements per row, each
    input row read once and each output row written once), in place, with
    the gradient rows, and only those, read as bf16 where they are bf16."""
    import types
    N = 64
    wl = wls.get(f"flat_N{N}_W{W}_K2_{opt}_{gd}")
    S, gb = wl.state_arrays, wl.grad_bytes
    st = types.SimpleNamespace(params=torch.zeros(W, N), mom=torch.zeros(W, N), exp_avg_sq=torch.zeros(W, N),
                               anchor=torch.zeros(N), slow_v=torch.zeros(N))
    g = torch.zeros(W, N, dtype=torch.bfloat16 if gd == "bf16" else torch.float32)
    for kind, want in (("local", bench.local_step_bytes(W, N, gb, S)), ("sync", bench.reconcile_bytes(W, N, gb, S))):
        ins, ins16, outs, n = bench.floor_rows(wl, st, g, kind)
        assert 4 * n * (len(ins) + len(outs)) + 2 * n * len(ins16) == want
        assert all(x.dtype == torch.float32 for x in ins + outs) and all(x.dtype == torch.bfloat16 for x in ins16)
        assert len(ins16) == (0 if gd == "f32" else 1 if kind == "local" else W)
        assert all(any(o.data_ptr() == i.data_ptr() for i in ins) for o in outs)  # outputs among the inputs
