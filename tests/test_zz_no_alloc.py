"""flarepp_route_fwd_noalloc, the entry point for callers that cannot allocate device memory
at call time (a plugin whose host application owns all device memory, a latency-critical
loop where cudaMalloc/cudaFree would synchronise the device). It runs the chain with the
library's fixed 64 MiB scratch array instead of a caller workspace.

Checked through the C ABI. The no-allocation call runs the same plan and the same
deterministic kernels as flarepp_route_fwd, so their outputs must be bit-identical. Two
calls in a row run per shape, the larger shape first: the second call finds the first
call's contents in the shared scratch, so a read of a stale slot would show. One float32
case is also checked against the oracle (1e-5, the float32 parity tolerance). This file is
collected last on purpose.
"""
import pytest
import torch

from paper_2608_11519_gb300 import flarepp, inputs

pytestmark = pytest.mark.gpu

# larger workspaces first, so that each later call finds more scratch written than it uses
SHAPES = [
    inputs.get("pde2d").with_(B=2, N=9000),
    inputs.Workload("ragged", 1, 3, 1001, 300, 64, "bf16"),
    inputs.get("tiny"),
]


def test_noalloc_bit_identical_to_route_fwd():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    for w in SHAPES:
        for seed in (11, 12):
            x = inputs.make_inputs(w, seed=seed, device="cuda")
            args = (x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"])
            ref = flarepp.route_fwd(*args, w.scale)
            got = flarepp.route_fwd_noalloc(*args, w.scale)
            torch.cuda.synchronize()
            assert torch.equal(got, ref), \
                f"{w.describe()} seed {seed}: max|noalloc - route_fwd| = " \
                f"{float((got.double() - ref.double()).abs().max())}"


def test_noalloc_matches_oracle_f32():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import oracle
    torch.cuda.set_device(0)
    w = inputs.get("tiny")
    x = inputs.make_inputs(w, seed=5)
    xd = {k: v.cuda() for k, v in x.items()}
    got = flarepp.route_fwd_noalloc(xd["seeds"], xd["Kt"], xd["Vt"], xd["K"], xd["V"], w.scale)
    torch.cuda.synchronize()
    f = inputs.to_f64_numpy(x)
    _, _, Yo = oracle.route(f["seeds"], f["Kt"], f["Vt"], f["K"], f["V"], w.scale)
    err = float(abs(got.double().cpu().numpy() - Yo).max())
    assert err <= 1e-5, f"max|noalloc - oracle| = {err}"


def test_noalloc_rejects_shapes_beyond_its_scratch():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    lib = flarepp.load()
    shape = flarepp.make_shape(1, 8, 262144, 2048, 64, flarepp.BF16)
    assert flarepp.workspace_bytes(1, 8, 262144, 2048, 64, flarepp.BF16) > (64 << 20)
    import ctypes
    rc = lib.flarepp_route_fwd_noalloc(ctypes.byref(shape), None, None, None, None, None,
                                       ctypes.c_float(0.125), None, None)
    assert rc == flarepp.ERR_WORKSPACE
