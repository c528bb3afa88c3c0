"""GPU parity of the chain's backward (App. A.5) against the float64 oracle, through the C ABI.

The training forward (``flarepp_route_fwd_train``) runs first and its Y and saved state
feed ``flarepp_route_bwd``; the oracle recomputes everything from the same input values.

Tolerance, per gradient tensor G (max abs error after upcasting to float64):
    max|G - G_ref| <= tol * max(1, max|G_ref|),  tol = 1e-5 (float32), 2e-2 (bf16 inputs)
i.e. the forward's tolerances taken relative to the gradient's own scale: a gradient sums
N (or M, or B*N) unit-scale products, so its magnitude is not 1. On the bf16 path the forward
multiplies bf16 copies of Q and Z and stores Y in bf16; the backward differentiates that
function, while the oracle differentiates the exact one, so the gap is of the order of the
forward's own bf16 error.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_11519_gb300 import flarepp, inputs

pytestmark = pytest.mark.gpu

TOL = {"f32": 1e-5, "bf16": 2e-2}
NAMES = ("dseeds", "dKt", "dVt", "dK", "dV")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    flarepp.load()
    torch.cuda.set_device(0)


def _np(t):
    return t.detach().to("cpu", torch.float64).numpy()


def _gpu_grads(x, dY, scale):
    xd = {k: v.cuda() for k, v in x.items()}
    args = (xd["seeds"], xd["Kt"], xd["Vt"], xd["K"], xd["V"])
    Y, saved = flarepp.route_fwd_train(*args, scale)
    grads = flarepp.route_bwd(*args, Y, dY.cuda(), saved, scale)
    torch.cuda.synchronize()
    return [_np(g) for g in grads], Y


def _check_grads(got, want, tol, where=""):
    errs = {}
    for name, g, r in zip(NAMES, got, want):
        bound = tol * max(1.0, float(np.abs(r).max()) if r.size else 0.0)
        err = float(np.abs(g - r).max()) if g.size else 0.0
        assert err <= bound and not math.isnan(err), f"{name}{where}: {err} > {bound}"
        errs[name] = err
    return errs


SHAPES = [
    # B, H, N, M, D, dtype, scale (None: 1/sqrt(D))
    (1, 4, 1024, 32, 16, "f32", None),   # the tiny float32 configuration
    (2, 3, 300, 40, 16, "f32", None),
    (3, 2, 257, 7, 64, "f32", -0.5),
    (1, 1, 1, 1, 32, "f32", None),
    (2, 2, 3000, 128, 32, "bf16", None),
    (1, 2, 1000, 600, 32, "bf16", None),  # more than one 512-route group
    (1, 3, 777, 100, 16, "bf16", None),
    (1, 2, 500, 64, 64, "bf16", None),
    (2, 2, 600, 50, 32, "bf16", -0.3),
    (1, 2, 130, 513, 32, "bf16", None),   # ragged route tile
    (1, 1, 50, 10, 32, "bf16", None),     # one partial tile each way
    (2, 1, 129, 257, 64, "bf16", 0.2),    # tails of both 256-row groups
]


@pytest.mark.parametrize("shape", SHAPES, ids=[str(s) for s in SHAPES])
def test_bwd_matches_oracle(shape):
    B, H, N, M, D, dt, scale = shape
    w = inputs.Workload("case", B, H, N, M, D, dt)
    scale = 1.0 / math.sqrt(D) if scale is None else scale
    x = inputs.make_inputs(w, 3)
    dY = inputs.make_output_grad(w, 3)
    got, _ = _gpu_grads(x, dY, scale)
    f = inputs.to_f64_numpy(x)
    want = oracle.route_bwd(f["seeds"], f["Kt"], f["Vt"], f["K"], f["V"], scale, _np(dY))
    _check_grads(got, want, TOL[dt])


@pytest.mark.parametrize("D", [32, 64])
def test_training_forward_matches_forward(D):
    """The training forward writes Y as the plain forward does and saves the log-normalisers
    of the oracle's calls. At D = 64 it runs the plain forward's kernels: Y bit for bit. At
    D <= 32 its calls 2 and 3 take Q as a hi/lo pair of bf16 operands (the plain forward: bf16
    Q alone), so Y differs from the plain forward's by bf16 rounding only, and both match the
    oracle."""
    w = inputs.Workload("case", 2, 2, 2000, 96, D, "bf16")
    x = {k: v.cuda() for k, v in inputs.make_inputs(w, 5).items()}
    args = (x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"])
    s = 1.0 / math.sqrt(w.D)
    Y0 = flarepp.route_fwd(*args, s)
    Y1, saved = flarepp.route_fwd_train(*args, s)
    torch.cuda.synchronize()
    if D > 32:
        assert torch.equal(Y0, Y1)
    else:
        assert not torch.equal(Y0, Y1)  # the hi/lo operands did run
        f = inputs.to_f64_numpy({k: v.cpu() for k, v in x.items()})
        _, _, Yo = oracle.route(f["seeds"], f["Kt"], f["Vt"], f["K"], f["V"], s)
        for Yg in (Y0, Y1):
            err = float(np.abs(_np(Yg) - Yo).max())
            assert err <= TOL["bf16"], err
    BH, M, N, D = w.B * w.H, w.M, w.N, w.D
    qz = BH * M * D * 4
    al = lambda n: (n + 255) // 256 * 256
    off_l1 = 2 * al(qz)
    off_l2 = off_l1 + al(BH * M * 4)
    off_l3 = off_l2 + al(BH * M * 4)
    raw = saved.cpu()
    L = lambda off, n: raw[off:off + 4 * n].view(torch.float32).double().numpy()
    ln2 = math.log(2.0)
    f = inputs.to_f64_numpy({k: v.cpu() for k, v in x.items()})
    Qs = np.broadcast_to(f["seeds"], (w.B,) + f["seeds"].shape)
    Q, L1 = oracle.sdpa(Qs, f["Kt"], f["Vt"], s)
    Z, L2 = oracle.sdpa(Q, f["K"], f["V"], s)
    _, L3 = oracle.sdpa(f["K"], Q, Z, s)
    for got, want in ((L(off_l1, BH * M), L1), (L(off_l2, BH * M), L2), (L(off_l3, BH * N), L3)):
        np.testing.assert_allclose(got * ln2, want.reshape(-1), rtol=0, atol=2e-2)


@pytest.mark.parametrize("name", ["pde2d", "longseq"])
def test_bwd_full_size_slices(name):
    """Full-size workloads: the backward of the whole batch on the GPU, each sampled (b, h)
    slice checked against the oracle run on that slice alone (slices are independent, and
    the seeds' gradient of a slice is its batch element's share)."""
    w = inputs.get(name)
    s = w.scale
    x = inputs.make_inputs(w, 0)
    dY = inputs.make_output_grad(w, 0)
    got, _ = _gpu_grads(x, dY, s)
    f = inputs.to_f64_numpy(x)
    dYn = _np(dY)
    rng = np.random.default_rng(0)
    picks = [(0, 0), (w.B - 1, w.H - 1)] + [(int(rng.integers(w.B)), int(rng.integers(w.H)))]
    # the seeds' gradient sums over the batch: check it on a batch of one element per head
    for b, h in picks:
        sl = lambda a: a[b:b + 1, h:h + 1]
        want = oracle.route_bwd(f["seeds"][h:h + 1], sl(f["Kt"]), sl(f["Vt"]), sl(f["K"]),
                                sl(f["V"]), s, sl(dYn))
        tol = TOL[w.dtype]
        for name_, g, r in zip(NAMES[1:], got[1:], want[1:]):
            gg = g[b:b + 1, h:h + 1]
            bound = tol * max(1.0, float(np.abs(r).max()))
            err = float(np.abs(gg - r).max())
            assert err <= bound, f"{name_}[{b},{h}]: {err} > {bound}"
    # dseeds over the whole batch, checked head by head through the oracle on all b
    h = picks[0][1]
    want = oracle.route_bwd(f["seeds"][h:h + 1], f["Kt"][:, h:h + 1], f["Vt"][:, h:h + 1],
                            f["K"][:, h:h + 1], f["V"][:, h:h + 1], s, dYn[:, h:h + 1])
    r = want[0][0]
    bound = TOL[w.dtype] * max(1.0, float(np.abs(r).max()))
    assert float(np.abs(got[0][h] - r).max()) <= bound


def test_bwd_identities_at_mesh3d_size():
    """The largest workload (one head of 1,048,576 tokens per head, M = 512, bf16): the
    oracle is too slow there, so the identities that hold at any size are checked on the
    GPU's gradients (in float64 on the host): call 1's keys sum to zero gradient over the
    tokens, the values' gradients sum to those of Y, <dV, V> = <dY, Y> and
    <dseeds, seeds> = <dKt, Kt>. Each sum is compared with the sum of the magnitudes of its
    terms."""
    w = inputs.get("mesh3d")
    s = w.scale
    x = inputs.make_inputs(w, 0)
    dY = inputs.make_output_grad(w, 0)
    got, Y = _gpu_grads(x, dY, s)
    dseeds, dKt, dVt, dK, dV = got
    f = inputs.to_f64_numpy(x)
    dYn, Yn = _np(dY), _np(Y)
    for v in got:
        assert np.all(np.isfinite(v))
    rel = 1e-2
    lhs = dKt.sum(axis=2)
    assert np.all(np.abs(lhs) <= rel * np.abs(dKt).sum(axis=2) + 1e-6)
    lhs = dV.sum(axis=2) - dYn.sum(axis=2)
    assert np.all(np.abs(lhs) <= rel * (np.abs(dV).sum(axis=2) + np.abs(dYn).sum(axis=2)))
    a, b = np.sum(dV * f["V"]), np.sum(dYn * Yn)
    assert abs(a - b) <= rel * (np.abs(dV * f["V"]).sum() + np.abs(dYn * Yn).sum())
    a, b = np.sum(dseeds * f["seeds"]), np.sum(dKt * f["Kt"])
    assert abs(a - b) <= rel * (np.abs(dseeds * f["seeds"]).sum() + np.abs(dKt * f["Kt"]).sum())


def test_bwd_degenerate_shapes():
    """N = 0, M = 0 or B = 0: every existing gradient is zero."""
    for (B, H, N, M, D, dt) in [(2, 2, 0, 8, 32, "bf16"), (1, 2, 64, 0, 16, "f32"),
                                (0, 2, 64, 8, 32, "bf16")]:
        w = inputs.Workload("case", B, H, N, M, D, dt)
        x = {k: v.cuda() for k, v in inputs.make_inputs(w, 1).items()}
        args = (x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"])
        Y, saved = flarepp.route_fwd_train(*args)
        dY = inputs.make_output_grad(w, 1).cuda()
        grads = [torch.full_like(t, 7.0) for t in args]
        flarepp.route_bwd(*args, Y, dY, saved, grads=grads)
        torch.cuda.synchronize()
        for g in grads:
            assert not torch.any(g != 0)


def test_bwd_is_deterministic():
    w = inputs.Workload("case", 1, 2, 5000, 128, 32, "bf16")
    x = inputs.make_inputs(w, 9)
    dY = inputs.make_output_grad(w, 9)
    a, _ = _gpu_grads(x, dY, w.scale)
    b, _ = _gpu_grads(x, dY, w.scale)
    for u, v in zip(a, b):
        assert np.array_equal(u, v)


@pytest.mark.parametrize("shape", [(1, 2, 700, 2048, 16, "bf16"), (1, 1, 500, 2048, 64, "bf16"),
                                   (1, 1, 300, 1024, 32, "f32")],
                         ids=["M2048_D16", "M2048_D64", "M1024_f32"])
def test_bwd_largest_route_counts(shape):
    """The largest supported M (2048) with the smallest and largest head widths."""
    B, H, N, M, D, dt = shape
    w = inputs.Workload("case", B, H, N, M, D, dt)
    x = inputs.make_inputs(w, 4)
    dY = inputs.make_output_grad(w, 4)
    got, _ = _gpu_grads(x, dY, w.scale)
    f = inputs.to_f64_numpy(x)
    want = oracle.route_bwd(f["seeds"], f["Kt"], f["Vt"], f["K"], f["V"], w.scale, _np(dY))
    _check_grads(got, want, TOL[dt])


def test_bwd_guard_bands_untouched():
    """The gradients are written inside their tensors only: each output is a view into a
    larger buffer whose bands before and after keep their sentinel value."""
    w = inputs.Workload("case", 2, 2, 777, 100, 32, "bf16")
    x = {k: v.cuda() for k, v in inputs.make_inputs(w, 6).items()}
    args = (x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"])
    Y, saved = flarepp.route_fwd_train(*args, w.scale)
    dY = inputs.make_output_grad(w, 6).cuda()
    band = 4096
    grads, bufs = [], []
    for t in args:
        buf = torch.full((t.numel() + 2 * band,), 7.0, dtype=t.dtype, device="cuda")
        bufs.append(buf)
        grads.append(buf[band:band + t.numel()].view(t.shape))
    flarepp.route_bwd(*args, Y, dY, saved, w.scale, grads=tuple(grads))
    torch.cuda.synchronize()
    for buf in bufs:
        assert torch.all(buf[:band] == 7.0) and torch.all(buf[-band:] == 7.0)
    for g in grads:
        assert torch.isfinite(g.float()).all()


def _stat_spread(f, scale):
    """Per (b, h): max_n L3 - min_m L2 of the chain's calls 2 and 3 (base-2 log-normalisers
    of the scores x = scale log2(e) <Q_m, K_n>, over tokens per route and over routes per
    token), computed in float64 from the oracle's Q."""
    c = scale / math.log(2)
    out = []
    B, H = f["K"].shape[:2]
    for b in range(B):
        for h in range(H):
            x1 = c * f["seeds"][h] @ f["Kt"][b, h].T
            a1 = np.exp2(x1 - x1.max(1, keepdims=True))
            Q = (a1 / a1.sum(1, keepdims=True)) @ f["Vt"][b, h]
            x2 = c * Q @ f["K"][b, h].T  # [M, N]
            m2 = x2.max(1, keepdims=True)
            L2 = m2[:, 0] + np.log2(np.exp2(x2 - m2).sum(1))
            m3 = x2.max(0, keepdims=True)
            L3 = m3[0] + np.log2(np.exp2(x2 - m3).sum(0))
            out.append(max(L3.max() - L2.min(), L2.max() - L2.min()))
    return out


@pytest.mark.parametrize("D,fac,flagged", [(32, 8, False), (16, 8, False), (32, 16, True),
                                           (16, 16, True)])
def test_bwd_wide_score_ranges(D, fac, flagged):
    """Sharp routes (seeds x 10) and, on heads 1 and 3, keys scaled by `fac` spread the
    log-normalisers L2, L3 over tens of binary orders. The merged pass of calls 3 and 2
    scales V and dZ by 2^(L3 - R) and 2^(R - L2); up to a spread of 60 it serves every head
    (fac 8: spreads near 50), beyond it those heads run the unmerged pass while the others
    stay merged (fac 16: spreads above 80 on heads 1 and 3). Both must match the oracle, every
    gradient at the bf16 tolerance.

    On heads this sharp, the softmaxes of calls 2 and 3 react to Q's bf16 rounding (a score
    moves by 2^-9 of its size, which here is tens of binary orders): with bf16 Q alone, dQ is
    off by up to 4 % of its scale, and the gradients of call 1 and dK by up to 6 %. The
    training forward and the backward therefore take Q as a hi/lo pair of bf16 operands in
    the scores of calls 2 and 3 (D <= 32)."""
    scale = 1.0 / math.sqrt(D)
    w = inputs.Workload("case", 1, 4, 2000, 200, D, "bf16")
    x = inputs.make_inputs(w, 5)
    x["seeds"] = (x["seeds"].float() * 10).to(torch.bfloat16)
    K = x["K"].float()
    K[:, 1] *= fac
    K[:, 3] *= fac
    x["K"] = K.to(torch.bfloat16)
    dY = inputs.make_output_grad(w, 5)
    f = inputs.to_f64_numpy(x)
    spread = _stat_spread(f, scale)
    wide = [s > 60.0 for s in spread]
    assert wide == [False, flagged, False, flagged], spread
    assert max(spread) > 30.0, spread
    got, _ = _gpu_grads(x, dY, scale)
    want = oracle.route_bwd(f["seeds"], f["Kt"], f["Vt"], f["K"], f["V"], scale, _np(dY))
    _check_grads(got, want, TOL["bf16"], f" (D={D}, fac={fac})")


def test_golden_bwd_fixture_f32():
    """The float32 backward on the stored case (tests/golden/route_small.json inputs,
    route_bwd_small.json's dY and oracle gradients)."""
    import json
    import os
    here = os.path.join(os.path.dirname(__file__), "golden")
    with open(os.path.join(here, "route_small.json")) as fh:
        fwd = json.load(fh)
    with open(os.path.join(here, "route_bwd_small.json")) as fh:
        bwd = json.load(fh)
    x = {k: torch.tensor(v, dtype=torch.float32) for k, v in fwd["inputs"].items()}
    dY = torch.tensor(bwd["dY"], dtype=torch.float32)
    got, _ = _gpu_grads(x, dY, fwd["scale"])
    want = [np.array(bwd["expected"][n]) for n in NAMES]
    _check_grads(got, want, TOL["f32"], " (stored case)")
