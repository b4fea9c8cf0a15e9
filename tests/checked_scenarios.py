"""Runs every kernel variant of the library once through a short epoch and
prints one JSON line: a digest of all state arrays per configuration, and the
out-of-range index count the library reports after each (cpdp_bad_index_count:
-1 from a release build). tests/test_checked_build_gpu.py runs it against the
release library and against the index-checked debug build (CPDP_LIBRARY) and
compares the two. Not a test module itself."""
import hashlib
import itertools
import json
import sys
from pathlib import Path

sys.path.insert(0, str(Path(__file__).resolve().parents[1]))

import torch  # noqa: E402

from paper_2607_21224_gb300 import cpdp  # noqa: E402
from paper_2607_21224_gb300.pipeline import HostGradientPipeline  # noqa: E402
from paper_2607_21224_gb300.state import CPDPState, grad_dtype_code  # noqa: E402


def digest(st: CPDPState) -> str:
    h = hashlib.sha256()
    for x in (st.params, st.mom, st.anchor, st.slow_v, getattr(st, "exp_avg_sq", None)):
        if x is not None:
            h.update(x.cpu().numpy().tobytes())
    return h.hexdigest()[:16]


def main() -> None:
    dev = torch.device("cuda")
    out, bad = {}, {}
    combos = [("cpdp", False), ("cpdp", True), ("localsgd", False), ("localsgd", True), ("ddp", False)]
    for (method, ss), opt, gdt, N, W in itertools.product(combos, ("sgd", "adamw"), (torch.float32, torch.bfloat16),
                                                          (4 * (256 * 3 + 5), 1027), (1, 2, 3, 4, 5, 6, 8)):
        name = f"{method}{'+ss' if ss else ''}/{opt}/{str(gdt)[6:]}/N{N}/W{W}"
        gen = torch.Generator(device=dev).manual_seed(N * 10 + W)
        theta0 = torch.randn(N, device=dev, generator=gen) * 0.05
        grads = [(torch.randn(W, N, device=dev, generator=gen) * 1e-3).to(gdt) for _ in range(3)]
        lr = 1e-3 if opt == "adamw" else 0.1
        with CPDPState(W, N, lr=lr, momentum=0.9, weight_decay=5e-4, K=2, beta=0.5) as st:
            if opt == "adamw":
                st.set_adamw()
            st.set_method(method)
            st.set_state_reconcile(ss)
            st.init_params(theta0)
            for t in range(1, 4):
                st.step(grads[t - 1], t, 3)
            torch.cuda.synchronize()
            out[name] = digest(st)
            bad[name] = cpdp.cpdp_bad_index_count(st.ctx)
    # the reconcile staged through shared memory by bulk copies (its segment
    # offsets go through the same checks), with a ragged last tile
    for W in (1, 2, 3, 5, 6, 8):
        N = 4 * (256 * 3 + 5)
        gen = torch.Generator(device=dev).manual_seed(N * 10 + W + 1)
        theta0 = torch.randn(N, device=dev, generator=gen) * 0.05
        grads = [torch.randn(W, N, device=dev, generator=gen) * 1e-3 for _ in range(3)]
        with CPDPState(W, N, lr=0.1, momentum=0.9, weight_decay=5e-4, K=2, beta=0.5) as st:
            st.set_reconcile_staging(2)
            st.init_params(theta0)
            for t in range(1, 4):
                st.step(grads[t - 1], t, 3)
            torch.cuda.synchronize()
            out[f"staged/W{W}"] = digest(st)
            bad[f"staged/W{W}"] = cpdp.cpdp_bad_index_count(st.ctx)
    # the reconcile with worker rows across a warp's lanes and shuffle sums,
    # with a partial last warp tile
    for W in (1, 3, 4, 8):
        N = 4 * (8 * 37 + 3)
        gen = torch.Generator(device=dev).manual_seed(N * 10 + W + 2)
        theta0 = torch.randn(N, device=dev, generator=gen) * 0.05
        grads = [torch.randn(W, N, device=dev, generator=gen) * 1e-3 for _ in range(3)]
        with CPDPState(W, N, lr=0.1, momentum=0.9, weight_decay=5e-4, K=2, beta=0.5) as st:
            st.set_reconcile_shuffle(True)
            st.init_params(theta0)
            for t in range(1, 4):
                st.step(grads[t - 1], t, 3)
            torch.cuda.synchronize()
            out[f"shuffle/W{W}"] = digest(st)
            bad[f"shuffle/W{W}"] = cpdp.cpdp_bad_index_count(st.ctx)
    # the host-fed paths, which stage gradients before the same kernels
    N, W = 4 * 1000, 4
    gen = torch.Generator(device="cpu").manual_seed(3)
    host = [(torch.randn(W, N, generator=gen) * 1e-3).pin_memory() for _ in range(2)]
    for path in ("staged", "noalloc"):
        with CPDPState(W, N, lr=0.1, momentum=0.9, weight_decay=5e-4, K=2, beta=0.5) as st:
            st.init_params(torch.zeros(N, device=dev))
            feed = HostGradientPipeline(st) if path == "staged" else None
            for t in (1, 2):
                if feed is not None:
                    feed.step(host[t - 1], t, 2)
                else:
                    cpdp.cpdp_step_host_noalloc(st.ctx, host[t - 1], grad_dtype_code(host[t - 1]), t, 2)
            torch.cuda.synchronize()
            out[f"host/{path}"] = digest(st)
            bad[f"host/{path}"] = cpdp.cpdp_bad_index_count(st.ctx)
    print(json.dumps({"library": str(cpdp.library_path().name), "digests": out, "bad": bad}))


if __name__ == "__main__":
    main()
