"""bench.py on the GPU, at small sizes: the JSON line carries what the
measurement promises (roofline, floors for L2-sized workloads and, on
request, for larger ones, the e2e leg with the host link measured around it,
the staged-reconcile option), and the bounded kernel waits never ran out."""
import contextlib
import io
import json

import pytest

import bench

pytestmark = pytest.mark.gpu


def _line(argv) -> dict:
    buf = io.StringIO()
    with contextlib.redirect_stdout(buf):
        bench.main(argv)
    return json.loads(buf.getvalue().strip().splitlines()[-1])


def test_tiny_line_has_floor_e2e_and_graph():
    d = _line(["--workload", "tiny", "--steps", "6", "--warmup", "3", "--no-cpu-baseline", "--graph",
               "--e2e-steps", "4"])
    assert d["value"] > 0 and d["unit"] == "GB/s" and d["gpu_launches"] == 6 * 2
    assert d["roofline"]["bound"] == "hbm" and d["roofline"]["achieved"] > 0
    assert d["kernel_wait_timeouts"] == 0
    f = d["floor"]
    assert f["stream_GB_s"] > 0 and f["empty_ms_per_step"] > 0 and f["frac_of_stream_floor"] > 0
    e = d["e2e"]
    assert e["h2d_bytes_per_step"] == 2 * 2 * (1 << 20) * 4 and e["d2h_bytes_per_step"] == (1 << 20) * 4
    assert e["link_h2d_GB_s"] == max(e["link_h2d_before_GB_s"], e["link_h2d_after_GB_s"]) > 0
    assert 0 < e["frac_of_link"] and e["ms_per_step_median"] <= e["ms_per_step_max"]
    assert d["graph_replay"]["value"] > 0
    assert d["config"]["reconcile_staging"] == 0 and d["config"]["workload"] == "tiny"


def test_staged_reconcile_option_reports_its_kernel():
    d = _line(["--workload", "sweep_N1048576_W4_K2", "--steps", "4", "--warmup", "3", "--no-cpu-baseline",
               "--no-e2e", "--reconcile-staging", "3"])
    kernels = {d["roofline"]["kernel"], d["roofline_other"]["kernel"]}
    assert "reconcile_tma_kernel" in kernels and d["config"]["reconcile_staging"] == 3
    assert d["kernel_wait_timeouts"] == 0


def test_adamw_graph_is_reported_unavailable():
    d = _line(["--workload", "flat_N65536_W2_K2_adamw_bf16", "--steps", "4", "--warmup", "3", "--no-cpu-baseline",
               "--no-e2e", "--graph"])
    assert "unavailable" in d["graph_replay"] and d["value"] > 0
    # bf16 gradients have their floor too (the gradient rows read as bf16)
    assert d["floor"]["stream_reconcile_GB_s"] > 0 and d["floor"]["stream_local_GB_s"] > 0


def test_floor_option_above_l2_reports_each_kernel_against_its_floor():
    d = _line(["--workload", "flat_N16777216_W4_K2_adamw_bf16", "--steps", "4", "--warmup", "3",
               "--no-cpu-baseline", "--no-e2e", "--floor"])
    f = d["floor"]
    assert "larger than L2" in d["config"]["l2"] and f["scrub"].startswith("none")
    for r in (d["roofline"], d["roofline_other"]):
        key = "stream_local_GB_s" if r["kernel"] == "local_step_kernel" else "stream_reconcile_GB_s"
        assert r["floor_GB_s"] == f[key] > 0 and r["frac_of_floor"] == round(r["achieved"] / f[key], 4)
    rr = d["roofline"] if d["roofline"]["kernel"] != "local_step_kernel" else d["roofline_other"]
    assert rr["column_walk_GB_s"] == f["columns_reconcile_GB_s"] > 0 and "blocks per SM" in f["columns_shape"]


def test_floor_kernel_sums_float_and_bf16_rows():
    """The floor kernel's arithmetic: each output row receives the sum of the
    float32 rows and the widened bf16 rows, column by column."""
    import torch
    from paper_2607_21224_gb300 import cpdp
    n = 4 * 1000
    a = torch.randn(n, device="cuda")
    b = torch.randn(n, device="cuda").to(torch.bfloat16)
    c = torch.randn(n, device="cuda").to(torch.bfloat16)
    out = torch.empty(2, n, device="cuda")
    cpdp.cpdp_floor_stream([a], [out[0], out[1]], n, 0, torch.cuda.current_stream().cuda_stream, inputs_bf16=[b, c])
    torch.cuda.synchronize()
    want = (b.float() + c.float()) + a
    assert torch.equal(out[0], want) and torch.equal(out[1], want)


def test_odd_n_workload_reports_the_scalar_kernel_and_no_floor():
    d = _line(["--workload", "flat_N1027_W3_K2_sgd_f32", "--steps", "4", "--warmup", "3", "--no-cpu-baseline",
               "--no-e2e"])
    assert "floor" not in d and d["value"] > 0
    assert {d["roofline"]["kernel"], d["roofline_other"]["kernel"]} == {"local_step_kernel", "reconcile_scalar_kernel"}


@pytest.mark.parametrize("rows,blocks", [(2, 4), (3, 3), (4, 2)])
@pytest.mark.parametrize("gd", ["f32", "bf16"])
def test_floor_columns_kernel_arithmetic(rows, blocks, gd):
    """The column-walk floor's arithmetic, for every compiled shape and a worker
    count that leaves a partial chunk: each state row gains its gradient row,
    theta_ref gains v, and nothing else changes."""
    import torch
    from paper_2607_21224_gb300 import cpdp
    W, N = 5, 4 * 777
    g32 = torch.randn(W, N, device="cuda")
    g = g32.to(torch.bfloat16) if gd == "bf16" else g32
    p0, m0, s0 = (torch.randn(W, N, device="cuda") for _ in range(3))
    ref0, vel0 = torch.randn(N, device="cuda"), torch.randn(N, device="cuda")
    p, m, sq, ref, vel = p0.clone(), m0.clone(), s0.clone(), ref0.clone(), vel0.clone()
    dt = cpdp.CPDP_BF16 if gd == "bf16" else cpdp.CPDP_F32
    cpdp.cpdp_floor_columns(p, m, sq, g, dt, ref, vel, W, N, rows, blocks, torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    gf = g.float()
    assert torch.equal(p, p0 + gf) and torch.equal(m, m0 + gf) and torch.equal(sq, s0 + gf)
    assert torch.equal(ref, ref0 + vel0) and torch.equal(vel, vel0)
    p2, m2 = p0.clone(), m0.clone()  # two state arrays
    cpdp.cpdp_floor_columns(p2, m2, None, g, dt, ref, vel, W, N, rows, blocks, torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    assert torch.equal(p2, p0 + gf) and torch.equal(m2, m0 + gf)
