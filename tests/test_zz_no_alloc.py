"""flarepp_route_fwd_noalloc, the entry point for callers that cannot allocate device memory
at call time (a plugin whose host application owns all device memory, a latency-critical
loop where cudaMalloc/cudaFree would synchronise the device). It runs the chain with the
library's fixed 64 MiB scratch array instead of a caller workspace.

Checked through the C ABI: two calls in a row (the second finds the first call's contents
in the shared scratch) must each match flarepp_route_fwd within the parity tolerances used
elsewhere (1e-5 float32, 2e-2 bf16). This file is collected last on purpose.
"""
import pytest
import torch

from paper_2608_11519_gb300 import flarepp, inputs

pytestmark = pytest.mark.gpu

TOL = {"f32": 1e-5, "bf16": 2e-2}


@pytest.mark.parametrize("w", [
    inputs.get("tiny"),
    inputs.get("pde2d").with_(B=2, N=9000),
    inputs.Workload("ragged", 1, 3, 1001, 300, 64, "bf16"),
], ids=lambda w: w.name)
def test_noalloc_matches_route_fwd_twice(w):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    xs = [inputs.make_inputs(w, seed=s, device="cuda") for s in (11, 12)]
    for x in xs:
        args = (x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"])
        ref = flarepp.route_fwd(*args, w.scale)
        got = flarepp.route_fwd_noalloc(*args, w.scale)
        torch.cuda.synchronize()
        err = float((got.double() - ref.double()).abs().max())
        assert err <= TOL[w.dtype], f"{w.describe()}: max|noalloc - route_fwd| = {err}"


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
