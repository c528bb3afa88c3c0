"""GPU parity of the routing chain against the float64 oracle, through the C ABI.

Tolerances (max abs error, after upcasting Y to float64):
  * float32 inputs: 1e-5 on Q, Z and Y
  * bf16 inputs, float32 accumulation: 2e-2 on Q, Z and Y
Inputs come from paper_2608_11519_gb300.inputs (seeded); the oracle sees the exact input
values the GPU sees. Full-size workloads are checked on whole (b, h) slices (slices are
independent, Sec. 3.2) or, for the largest, on sampled tokens of one slice, plus the
convex-hull property on every output.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_11519_gb300 import flarepp, inputs

pytestmark = pytest.mark.gpu

TOL = {"f32": 1e-5, "bf16": 2e-2}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    flarepp.load()
    torch.cuda.set_device(0)


def _np(t):
    return t.detach().to("cpu", torch.float64).numpy()


def _run(x, scale, stream=None):
    xd = {k: v.cuda() for k, v in x.items()}
    Y, Q, Z = flarepp.route_fwd_debug(xd["seeds"], xd["Kt"], xd["Vt"], xd["K"], xd["V"], scale,
                                      stream=stream)
    torch.cuda.synchronize()
    return _np(Y), _np(Q), _np(Z)


def _check(name, got, want, tol):
    err = float(np.abs(got - want).max()) if got.size else 0.0
    assert err <= tol and not math.isnan(err), f"{name}: max|err| {err} > {tol}"
    return err


def _full_check(w, seed=0, scale=None, x=None, tol=None):
    x = x if x is not None else inputs.make_inputs(w, seed)
    s = w.scale if scale is None else scale
    Y, Q, Z = _run(x, s)
    f = inputs.to_f64_numpy(x)
    Qo, Zo, Yo = oracle.route(f["seeds"], f["Kt"], f["Vt"], f["K"], f["V"], s)
    tol = TOL[w.dtype] if tol is None else tol
    return {n: _check(n, g, o, tol) for n, g, o in (("Q", Q, Qo), ("Z", Z, Zo), ("Y", Y, Yo))}


def _hull_check(Y, V, slack):
    lo = V.min(axis=2, keepdims=True)
    hi = V.max(axis=2, keepdims=True)
    assert np.all(Y >= lo - slack) and np.all(Y <= hi + slack)


def _slice_check(w, slices, seed=0, sample_tokens=None):
    """Full-size run; oracle on the listed (b, h) slices (all tokens, or a token sample)."""
    x = inputs.make_inputs(w, seed, device="cuda")
    Y, Q, Z = _run(x, w.scale)
    tol = TOL[w.dtype]
    V = x["V"]
    for (b, h) in slices:
        f = {k: _np(v[h:h + 1] if k == "seeds" else v[b:b + 1, h:h + 1]) for k, v in x.items()}
        if sample_tokens is None:
            Qo, Zo, Yo = oracle.route(f["seeds"], f["Kt"], f["Vt"], f["K"], f["V"], w.scale)
            _check(f"Y[{b},{h}]", Y[b:b + 1, h:h + 1], Yo, tol)
        else:
            seeds_b = f["seeds"][None]
            Qo, _ = oracle.sdpa(seeds_b, f["Kt"], f["Vt"], w.scale)
            Zo, _ = oracle.sdpa(Qo, f["K"], f["V"], w.scale)
            rng = np.random.default_rng(b * 131 + h)
            rows = np.unique(np.concatenate([rng.integers(0, w.N, sample_tokens), [0, w.N - 1]]))
            Yo, _ = oracle.sdpa(f["K"][:, :, rows], Qo, Zo, w.scale)
            _check(f"Y[{b},{h}] sampled", Y[b:b + 1, h:h + 1][:, :, rows], Yo, tol)
        _check(f"Q[{b},{h}]", Q[b:b + 1, h:h + 1], Qo, tol)
        _check(f"Z[{b},{h}]", Z[b:b + 1, h:h + 1], Zo, tol)
    _hull_check(Y, _np(V), 1e-2 if w.dtype == "bf16" else 1e-6)


# ------------------------------------------------------------------ the stated workloads

def test_tiny_f32_full():
    _full_check(inputs.get("tiny"), seed=0)


def test_golden_fixture_f32():
    import json
    import os
    with open(os.path.join(os.path.dirname(__file__), "golden", "route_small.json")) as fh:
        doc = json.load(fh)
    x = {k: torch.tensor(v, dtype=torch.float32) for k, v in doc["inputs"].items()}
    Y, Q, Z = _run(x, doc["scale"])
    for name, got in (("Q", Q), ("Z", Z), ("Y", Y)):
        _check(name, got, np.array(doc["expected"][name]), 1e-5)


def test_pde2d_full_size():
    _slice_check(inputs.get("pde2d"), [(0, 0), (1, 3), (2, 6), (3, 7)])


def test_longseq_full_size():
    _slice_check(inputs.get("longseq"), [(0, 0), (17, 4), (31, 7)])


def test_mesh3d_full_size_sampled():
    """The largest workload at full size: Q and Z of three heads in full, Y on 4096 sampled
    tokens of each (plus the first and last)."""
    _slice_check(inputs.get("mesh3d"), [(0, 0), (0, 5), (0, 7)], sample_tokens=4096)


SWEEP = [(m, d) for m in (16, 32, 64, 128, 256, 512, 1024, 2048) for d in (16, 32, 64)]


@pytest.mark.parametrize("M,D", SWEEP)
def test_sweep_full_size(M, D):
    """Every point of the M x D sweep at its full size (N = 262,144): one (b, h) slice of Q,
    Z and Y in full against the oracle, the hull bound on every output."""
    _slice_check(inputs.get(f"sweep_M{M}_D{D}"), [(0, 3)])


@pytest.mark.parametrize("M,D", [(512, 32), (1024, 64), (2048, 16), (2048, 64)])
def test_sweep_large_M_reduced_N(M, D):
    w = inputs.get(f"sweep_M{M}_D{D}").with_(H=2, N=8192)
    _full_check(w)


# ------------------------------------------------------------------ edge cases

@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("N,M,D", [(1, 1, 16), (2, 3, 32), (31, 5, 64), (127, 32, 16),
                                   (129, 100, 32), (1000, 130, 64), (4097, 300, 32),
                                   (257, 1, 32), (5000, 17, 16)])
def test_ragged_shapes(dtype, N, M, D):
    w = inputs.Workload("ragged", 2, 3, N, M, D, dtype)
    _full_check(w, seed=N + M + D)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_clustered_peaked_small(dtype):
    w = inputs.Workload("peaked", 1, 2, 3000, 64, 32, dtype, n_centres=16)
    _full_check(w, seed=3)


def test_scale_zero_and_large():
    w = inputs.Workload("s", 1, 2, 700, 24, 32, "f32")
    _full_check(w, scale=0.0)
    # scale 2 gives logits of order +-30, which exercises the running max. The chain then
    # amplifies float32 rounding: an error dQ in a routing query moves call-2 logits by
    # s*|k|*dQ (s|k| ~ 2*8) and Z by that times the spread of V (~6), so the float32 bound
    # here is ~1e-6 * 16 * 6 ~ 1e-4 rather than the 1e-5 of the paper's scale 1/sqrt(D).
    _full_check(w, scale=2.0, tol=2e-4)


def test_m_zero_writes_zero():
    w = inputs.Workload("m0", 1, 2, 100, 0, 32, "bf16")
    x = {k: v.cuda() for k, v in inputs.make_inputs(w).items()}
    Y = torch.full_like(x["K"], 7.0)
    flarepp.route_fwd(x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"], Y=Y)
    torch.cuda.synchronize()
    assert torch.all(Y == 0)


def test_n_zero_and_b_zero_are_noops():
    for (B, N) in [(2, 0), (0, 50)]:
        w = inputs.Workload("e", B, 2, N, 8, 16, "f32")
        x = {k: v.cuda() for k, v in inputs.make_inputs(w).items()}
        Y, Q, Z = flarepp.route_fwd_debug(x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"])
        torch.cuda.synchronize()
        assert Y.numel() == 0 or B == 0
        assert torch.all(Q == 0) and torch.all(Z == 0)


def test_constant_values_give_constant_output():
    w = inputs.get("pde2d").with_(B=1, N=20000)
    x = inputs.make_inputs(w, seed=1, device="cuda")
    c = torch.randn(1, w.H, 1, w.D, device="cuda").to(torch.bfloat16)
    x["V"] = c.expand_as(x["V"]).contiguous()
    Y = flarepp.route_fwd(x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"])
    torch.cuda.synchronize()
    assert float((Y.float() - x["V"].float()).abs().max()) <= 2e-2


@pytest.mark.parametrize("shape", [
    dict(B=2, N=9000),                  # pde2d's routes: one route tile, four token parities
    dict(B=1, H=8, N=65536, M=16),      # 19 chunks x 4 parities: the merge splits slots over lanes
])
def test_deterministic_bitwise(shape):
    w = inputs.get("pde2d").with_(**shape)
    x = inputs.make_inputs(w, seed=4, device="cuda")
    a = flarepp.route_fwd(x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"])
    b = flarepp.route_fwd(x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"])
    torch.cuda.synchronize()
    assert torch.equal(a, b)


def test_guard_bands_untouched():
    """Canaries right after Y and after the workspace must survive a call."""
    w = inputs.get("pde2d").with_(B=1, N=5000)
    x = inputs.make_inputs(w, seed=5, device="cuda")
    nY = x["K"].numel()
    ybuf = torch.full((nY + 4096,), 1234.0, dtype=torch.bfloat16, device="cuda")
    Y = ybuf[:nY].view_as(x["K"])
    nws = flarepp.workspace_bytes(w.B, w.H, w.N, w.M, w.D, flarepp.BF16)
    wsbuf = torch.full((nws + 65536,), 0xA5, dtype=torch.uint8, device="cuda")
    flarepp.route_fwd(x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"], Y=Y, workspace=wsbuf)
    torch.cuda.synchronize()
    assert torch.all(ybuf[nY:] == 1234.0)
    assert torch.all(wsbuf[nws:] == 0xA5)


def test_side_stream_and_host_entry():
    w = inputs.get("tiny")
    x = inputs.make_inputs(w, seed=9)
    f = inputs.to_f64_numpy(x)
    _, _, Yo = oracle.route(f["seeds"], f["Kt"], f["Vt"], f["K"], f["V"], w.scale)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        Y, _, _ = _run(x, w.scale, stream=s)
    _check("Y side stream", Y, Yo, 1e-5)
    xh = {k: v.pin_memory() for k, v in x.items()}
    Yh = flarepp.route_fwd_host(xh["seeds"], xh["Kt"], xh["Vt"], xh["K"], xh["V"], w.scale)
    _check("Y host entry", _np(Yh), Yo, 1e-5)


@pytest.mark.parametrize("B,H,N,M,D,dtype", [
    (1, 8, 5000, 128, 32, "bf16"),   # eight groups of one head
    (1, 16, 2000, 64, 32, "bf16"),   # eight groups of two heads
    (9, 2, 3000, 100, 16, "bf16"),   # groups of two batch elements, a shorter last group
    (3, 3, 2000, 64, 64, "bf16"),    # one batch element per group
    (1, 4, 700, 20, 16, "f32"),      # one head per group, CUDA-core path
])
def test_host_entry_pipelined_groups(B, H, N, M, D, dtype):
    """flarepp_route_fwd_host splits the heads into groups and overlaps copies with compute;
    every group shape must give the oracle's Y."""
    w = inputs.Workload("host", B, H, N, M, D, dtype)
    x = inputs.make_inputs(w, seed=4)
    f = inputs.to_f64_numpy(x)
    _, _, Yo = oracle.route(f["seeds"], f["Kt"], f["Vt"], f["K"], f["V"], w.scale)
    xh = {k: v.pin_memory() for k, v in x.items()}
    ws = flarepp.Workspace()
    for _ in range(2):  # the second call reuses the device buffer
        Yh = flarepp.route_fwd_host(xh["seeds"], xh["Kt"], xh["Vt"], xh["K"], xh["V"], w.scale,
                                    workspace=ws)
        _check("Y host pipelined", _np(Yh), Yo, TOL[dtype])
    st = flarepp.device_status((x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"]), ws)
    assert st == 0


@pytest.mark.parametrize("B,H,N,M,D,dtype,scale", [
    (1, 2, 3000, 128, 32, "bf16", None),
    (2, 3, 2000, 100, 16, "bf16", -0.3),    # negative scale: negated query operands
    (1, 2, 5000, 700, 64, "bf16", None),    # two route groups, 32-route items
    (1, 1, 64, 512, 32, "bf16", None),      # one token item
    (2, 2, 700, 20, 16, "f32", None),       # CUDA-core path
])
def test_flare_fixed_queries(B, H, N, M, D, dtype, scale):
    """FLARE (Sec. 3, eq. prelim_flare_sdpa): Z = SDPA(Q_h, K, V), Y = SDPA(K, Q_h, Z)."""
    w = inputs.Workload("flare", B, H, N, M, D, dtype)
    s = w.scale if scale is None else scale
    x = inputs.make_inputs(w, seed=5)
    f = inputs.to_f64_numpy(x)
    Zo, Yo = oracle.flare(f["seeds"], f["K"], f["V"], s)
    xd = {k: v.cuda() for k, v in x.items()}
    Z = torch.empty((B, H, M, D), dtype=torch.float32, device="cuda")
    Y = flarepp.flare_fwd(xd["seeds"], xd["K"], xd["V"], s, Z_out=Z)
    torch.cuda.synchronize()
    _check("Z", _np(Z), Zo, TOL[dtype])
    _check("Y", _np(Y), Yo, TOL[dtype])


@pytest.mark.parametrize("D,M", [(16, 300), (32, 520), (64, 130)])
def test_bf16_logits_far_above_reference(D, M):
    """Scores far above a row's running reference. The bf16 kernels take each unit's first
    score as the reference and overwrite S with P as they go; a row whose later scores
    exceed the reference by tens of base-2 units is recomputed exactly. With scale 3, the
    base-2 logits have a spread of about 25 per standard deviation, so nearly every encode
    and decode row takes that path at least once. FLARE's queries are exact bf16 inputs, so
    the softmaxes (nearly one-hot) are compared without the chain's amplification of
    operand rounding."""
    w = inputs.Workload("flare", 1, 3, 2000, M, D, "bf16")
    s = 3.0
    x = inputs.make_inputs(w, seed=9)
    f = inputs.to_f64_numpy(x)
    Zo, Yo = oracle.flare(f["seeds"], f["K"], f["V"], s)
    xd = {k: v.cuda() for k, v in x.items()}
    Z = torch.empty((1, 3, M, D), dtype=torch.float32, device="cuda")
    Y = flarepp.flare_fwd(xd["seeds"], xd["K"], xd["V"], s, Z_out=Z)
    torch.cuda.synchronize()
    _check("Z", _np(Z), Zo, TOL["bf16"])
    # The decode's rows are nearly one-hot here, so the bf16 rounding of its P (relative
    # 2^-9 per probability) no longer averages out over many routes: between two close
    # routes it moves Y by up to 2^-8 |Z_a - Z_b| (|Z| <= max|V| ~ 4: 0.031), and the bf16
    # operand copy of Z adds 2^-9 |Z| (0.008). An exact-path mistake (a wrong reference,
    # a sum counted twice) moves Y by O(1).
    _check("Y", _np(Y), Yo, 4e-2)


@pytest.mark.parametrize("B,H,N,M,D,dtype,scale", [
    (1, 8, 5000, 128, 32, "bf16", None),   # eight head groups
    (2, 3, 1500, 40, 16, "bf16", -0.3),    # groups of whole batch elements, negative scale
    (1, 4, 700, 20, 16, "f32", None),      # CUDA-core path
])
def test_flare_host_entry(B, H, N, M, D, dtype, scale):
    """FLARE on host buffers (flarepp_flare_fwd_host, copies overlapped by head groups)
    against the oracle; a group's plan may chunk its tokens differently from the whole
    call's, so the comparison with the device entry is the oracle's tolerance, not bits. A
    second call on the same device buffer gives the same bits and leaves the status clear."""
    w = inputs.Workload("flare", B, H, N, M, D, dtype)
    s = w.scale if scale is None else scale
    x = inputs.make_inputs(w, seed=8)
    f = inputs.to_f64_numpy(x)
    _, Yo = oracle.flare(f["seeds"], f["K"], f["V"], s)
    xh = {k: v.pin_memory() for k, v in x.items()}
    ws = flarepp.Workspace()
    Yh = flarepp.flare_fwd_host(xh["seeds"], xh["K"], xh["V"], s, workspace=ws).clone()
    _check("Y host", _np(Yh), Yo, TOL[dtype])
    Yh2 = flarepp.flare_fwd_host(xh["seeds"], xh["K"], xh["V"], s, workspace=ws)
    assert torch.equal(Yh, Yh2)
    assert flarepp.device_status((x["seeds"], x["K"], x["V"], x["K"], x["V"]), ws) == 0


def test_shared_projection():
    """The shared-projection variant ties Kt, Vt to K, V (App. cost_model): the chain on
    aliased inputs, on device buffers and through the host entry (which copies K, V once)."""
    w = inputs.get("pde2d").with_(B=1, H=2, N=6000)
    x = inputs.make_inputs(w, seed=6)
    f = inputs.to_f64_numpy(x)
    Qo, Zo, Yo = oracle.route(f["seeds"], f["K"], f["V"], f["K"], f["V"], w.scale)
    xd = {k: v.cuda() for k, v in x.items()}
    Y, Q, Z = flarepp.route_fwd_debug(xd["seeds"], xd["K"], xd["V"], xd["K"], xd["V"], w.scale)
    torch.cuda.synchronize()
    for n, g, o in (("Q", Q, Qo), ("Z", Z, Zo), ("Y", Y, Yo)):
        _check(n, _np(g), o, TOL["bf16"])
    xh = {k: v.pin_memory() for k, v in x.items()}
    Yh = flarepp.route_fwd_host(xh["seeds"], xh["K"], xh["V"], xh["K"], xh["V"], w.scale)
    _check("Y host shared", _np(Yh), Yo, TOL["bf16"])


def test_profiled_entry_records_stages():
    w = inputs.get("pde2d").with_(B=1, N=8192)
    x = inputs.make_inputs(w, seed=2, device="cuda")
    ev = flarepp.StageEvents()
    Y = flarepp.route_fwd_profiled(x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"], ev)
    ms = ev.stage_ms()
    assert set(ms) == set(flarepp.STAGES) and all(v >= 0 for v in ms.values())
    Y2 = flarepp.route_fwd(x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"])
    torch.cuda.synchronize()
    assert torch.equal(Y, Y2)


def test_binding_rejects_tensors_on_another_device():
    """A host tensor among device tensors is refused before anything is launched: the
    library takes raw pointers and would read host memory as device memory."""
    w = inputs.get("tiny").with_(dtype="bf16")
    x = inputs.make_inputs(w, seed=3, device="cuda")
    for name in ("seeds", "Kt", "V"):
        y = dict(x)
        y[name] = y[name].cpu()
        with pytest.raises(ValueError, match=name):
            flarepp.route_fwd(y["seeds"], y["Kt"], y["Vt"], y["K"], y["V"])
    with pytest.raises(ValueError, match="Y"):
        flarepp.route_fwd(x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"], Y=torch.empty_like(
            x["K"], device="cpu"))
    with pytest.raises(ValueError, match="saved"):
        flarepp.route_bwd(x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"], x["K"], x["V"],
                          torch.empty(16, dtype=torch.uint8))
