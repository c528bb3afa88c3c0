"""Failure detection on the GPU without a fault: a bounded wait inside a tensor-core kernel
is made to run out, and the library must report it and stay usable.

flarepp_test_wait_fault makes CTA 0's load warp skip one item of its ring of tiles in one
launch of the chain and bounds every wait of that launch at 1 ms. The consumers of that item
then wait for a copy that never comes: their waits give up, the kernel records
FLAREPP_ERR_TIMEOUT in the workspace's status word, every role leaves its loops, the copies
in flight are awaited and TMEM is freed. Nothing traps or faults. The call must return, the
status word must read the timeout, and the next ordinary call on the same workspace must pass
oracle parity (the GPU context is intact).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_11519_gb300 import flarepp, inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    flarepp.load()
    torch.cuda.set_device(0)


@pytest.mark.parametrize("kernel,name", [(1, "encode of call 1"), (2, "encode of call 2"),
                                         (3, "decode")])
def test_bounded_wait_runs_out_and_call_recovers(kernel, name):
    lib = flarepp.load()
    w = inputs.Workload("timeout", 1, 2, 700, 96, 32, "bf16")
    x = inputs.make_inputs(w, seed=21)
    xd = {k: v.cuda() for k, v in x.items()}
    args = (xd["seeds"], xd["Kt"], xd["Vt"], xd["K"], xd["V"])
    ws = flarepp.Workspace()
    lib.flarepp_test_wait_fault(kernel, 0, 1_000_000)  # item 0 of CTA 0, 1 ms waits
    try:
        flarepp.route_fwd(*args, w.scale, workspace=ws)
        torch.cuda.synchronize()
        status = flarepp.device_status(args, ws)
    finally:
        lib.flarepp_test_wait_fault(0, -1, 0)
    assert status == flarepp.ERR_TIMEOUT, f"{name}: status {status} after a withheld item"
    # the same workspace, an ordinary call: status cleared, results match the oracle
    Y = flarepp.route_fwd(*args, w.scale, workspace=ws)
    torch.cuda.synchronize()
    assert flarepp.device_status(args, ws) == flarepp.OK
    f = inputs.to_f64_numpy(x)
    _, _, Yo = oracle.route(f["seeds"], f["Kt"], f["Vt"], f["K"], f["V"], w.scale)
    err = float(np.abs(Y.double().cpu().numpy() - Yo).max())
    assert err <= 2e-2, f"after the timeout in the {name}: max|Y - oracle| = {err}"


@pytest.mark.parametrize("pass_index,name", [(0, "route pass of call 3"),
                                             (4, "token pass of call 1")])
def test_backward_pass_wait_runs_out_and_recovers(pass_index, name):
    """The same for one tensor-core pass of the chain's backward (kernel 4 + pass): the call
    returns with FLAREPP_ERR_TIMEOUT in the backward workspace's status word, and a second
    backward on that workspace matches the oracle's gradients (2e-2 of each gradient's scale,
    the backward parity tolerance)."""
    lib = flarepp.load()
    w = inputs.Workload("timeout", 1, 2, 700, 96, 32, "bf16")
    x = inputs.make_inputs(w, seed=22)
    dY = inputs.make_output_grad(w, 22)
    xd = {k: v.cuda() for k, v in x.items()}
    args = (xd["seeds"], xd["Kt"], xd["Vt"], xd["K"], xd["V"])
    Y, saved = flarepp.route_fwd_train(*args, w.scale)
    wsb = flarepp.Workspace()
    lib.flarepp_test_wait_fault(4 + pass_index, 0, 1_000_000)
    try:
        flarepp.route_bwd(*args, Y, dY.cuda(), saved, w.scale, workspace=wsb)
        torch.cuda.synchronize()
        status = flarepp.device_status(args, wsb)
    finally:
        lib.flarepp_test_wait_fault(0, -1, 0)
    assert status == flarepp.ERR_TIMEOUT, f"{name}: status {status} after a withheld item"
    grads = flarepp.route_bwd(*args, Y, dY.cuda(), saved, w.scale, workspace=wsb)
    torch.cuda.synchronize()
    assert flarepp.device_status(args, wsb) == flarepp.OK
    f = inputs.to_f64_numpy(x)
    want = oracle.route_bwd(f["seeds"], f["Kt"], f["Vt"], f["K"], f["V"], w.scale,
                            dY.double().numpy())
    for gname, g, r in zip(("dseeds", "dKt", "dVt", "dK", "dV"), grads, want):
        bound = 2e-2 * max(1.0, float(np.abs(r).max()))
        err = float(np.abs(g.double().cpu().numpy() - r).max())
        assert err <= bound, f"after the timeout in the {name}: {gname} {err} > {bound}"
