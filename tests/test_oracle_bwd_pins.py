"""Pins for the oracle's backward pass (App. A.5), against facts the oracle does not restate.

Each check is one of:
  * central finite differences of the oracle's own forward chain (itself pinned in
    ``test_oracle_pins.py``), in float64 on tiny shapes, for every input element;
  * torch's float64 CPU autograd through its own scaled_dot_product_attention, in the
    paper's three-call form (Sec. 3.2) and for one SDPA;
  * identities of the chain: the keys of call 1 enter only through a softmax over the
    tokens (so their gradients sum to zero over the tokens); Y is linear in V with rows of
    two stochastic matrices in front (so the gradients of V sum to those of Y, and
    <dV, V> = <dY, Y>); call 1's logits are bilinear in the seeds and Kt (so
    <dseeds, seeds> = <dKt, Kt>);
  * a closed form for one route (M = 1), where call 3 is the identity on Z.

``test_bwd_pins_reject_planted_mistakes`` rebuilds the oracle with one deliberate mistake in
the backward at a time and checks that at least one pin fails for each.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle as oracle_pkg


def _rand(rng, *shape, scale=1.0):
    return rng.standard_normal(shape) * scale


def _inputs(B, H, N, M, D, rng, key_scale=1.0):
    seeds = _rand(rng, H, M, D)
    Kt = _rand(rng, B, H, N, D, scale=key_scale)
    Vt = _rand(rng, B, H, N, D)
    K = _rand(rng, B, H, N, D, scale=key_scale)
    V = _rand(rng, B, H, N, D)
    return seeds, Kt, Vt, K, V


def _torch_chain_grads(seeds, Kt, Vt, K, V, s, dY):
    """The chain as three torch SDPA calls (Sec. 3.2) differentiated by torch autograd."""
    t = lambda a: torch.tensor(np.asarray(a), dtype=torch.float64, requires_grad=True)
    ts, tKt, tVt, tK, tV = (t(a) for a in (seeds, Kt, Vt, K, V))
    B = K.shape[0]
    Qs = ts.unsqueeze(0).expand(B, *ts.shape)
    Q = F.scaled_dot_product_attention(Qs, tKt, tVt, scale=s)
    Z = F.scaled_dot_product_attention(Q, tK, tV, scale=s)
    Y = F.scaled_dot_product_attention(tK, Q, Z, scale=s)
    Y.backward(torch.from_numpy(np.asarray(dY, dtype=np.float64)))
    return tuple(a.grad.numpy() for a in (ts, tKt, tVt, tK, tV)), Y.detach().numpy()


# ---------------------------------------------------------------------------- pins

def pin_bwd_finite_differences(o):
    """Every gradient element equals a central difference of the forward chain."""
    rng = np.random.default_rng(11)
    for (B, H, N, M, D, s) in [(2, 2, 5, 3, 4, 0.45), (1, 1, 7, 2, 3, -0.8)]:
        x = list(_inputs(B, H, N, M, D, rng))
        W = _rand(rng, B, H, N, D)
        grads = o.route_bwd(*x, s, W)
        loss = lambda xs: float(np.sum(W * o.route(*xs, s)[2]))
        h = 1e-5
        for which in range(5):
            fd = np.zeros_like(x[which])
            flat = x[which].reshape(-1)
            for i in range(flat.size):
                keep = flat[i]
                flat[i] = keep + h
                lp = loss(x)
                flat[i] = keep - h
                lm = loss(x)
                flat[i] = keep
                fd.reshape(-1)[i] = (lp - lm) / (2 * h)
            g = grads[which]
            assert g.shape == fd.shape
            np.testing.assert_allclose(g, fd, rtol=0, atol=1e-7 * max(1.0, np.abs(fd).max()))


def pin_sdpa_bwd_vs_torch(o):
    """One SDPA's backward from the saved output and L equals torch autograd."""
    rng = np.random.default_rng(12)
    for (G, nq, nk, D, s) in [(3, 5, 17, 4, 0.5), (2, 33, 7, 16, 0.25), (1, 1, 1, 3, 1.3),
                              (2, 9, 40, 8, -0.6)]:
        q, k, v = _rand(rng, G, nq, D), _rand(rng, G, nk, D), _rand(rng, G, nk, D)
        dout = _rand(rng, G, nq, D)
        out, lse = o.sdpa(q, k, v, s)
        dq, dk, dv = o.sdpa_bwd(q, k, v, out, lse, dout, s)
        tq, tk, tv = (torch.tensor(a, requires_grad=True) for a in (q, k, v))
        F.scaled_dot_product_attention(tq, tk, tv, scale=s).backward(torch.from_numpy(dout))
        for mine, ref in ((dq, tq.grad), (dk, tk.grad), (dv, tv.grad)):
            np.testing.assert_allclose(mine, ref.numpy(), rtol=0, atol=1e-12)


def pin_route_bwd_vs_torch(o):
    """The chain's gradients equal torch autograd through three torch SDPA calls."""
    rng = np.random.default_rng(13)
    for (B, H, N, M, D, s, ks) in [(2, 3, 40, 6, 8, 1.0 / math.sqrt(8), 1.0),
                                   (1, 2, 100, 16, 4, 0.5, 2.0),
                                   (3, 1, 9, 12, 16, 0.25, 1.0),
                                   (1, 1, 33, 5, 8, -0.35, 1.5)]:
        x = _inputs(B, H, N, M, D, rng, key_scale=ks)
        dY = _rand(rng, B, H, N, D)
        mine = o.route_bwd(*x, s, dY)
        ref, _ = _torch_chain_grads(*x, s, dY)
        for a, b in zip(mine, ref):
            np.testing.assert_allclose(a, b, rtol=0, atol=1e-11 * max(1.0, np.abs(b).max()))


def pin_bwd_identities(o):
    """Shift invariance of call 1's softmax over tokens, linearity of Y in V, and the
    bilinear logits of call 1."""
    rng = np.random.default_rng(14)
    for (B, H, N, M, D, s) in [(2, 2, 50, 7, 8, 0.35), (1, 3, 17, 33, 4, 0.9)]:
        x = _inputs(B, H, N, M, D, rng)
        seeds, Kt, Vt, K, V = x
        dY = _rand(rng, B, H, N, D)
        dseeds, dKt, dVt, dK, dV = o.route_bwd(*x, s, dY)
        _, _, Y = o.route(*x, s)
        tol = 1e-10
        # adding a constant vector to every key of call 1 leaves Q unchanged
        np.testing.assert_allclose(dKt.sum(axis=2), 0.0, atol=tol * np.abs(dKt).max())
        # adding a constant vector a to every value row adds a to every Y row
        np.testing.assert_allclose(dV.sum(axis=2), dY.sum(axis=2), atol=tol * N)
        # Y(lambda V) = lambda Y
        assert abs(np.sum(dV * V) - np.sum(dY * Y)) <= tol * N * B * H
        # S1 = s seeds Kt^T is bilinear: scaling either factor scales S1 alike
        assert abs(np.sum(dseeds * seeds) - np.sum(dKt * Kt)) <= tol * N * B * H


def pin_bwd_one_route(o):
    """M = 1: call 3 returns Z for every token, so dZ = sum_n dY_n, the decoder adds
    nothing to dK, and dV_n = p_n dZ with p the softmax of call 2 over the tokens."""
    rng = np.random.default_rng(15)
    B, H, N, D, s = 2, 2, 23, 6, 0.7
    x = _inputs(B, H, N, 1, D, rng)
    seeds, Kt, Vt, K, V = x
    dY = _rand(rng, B, H, N, D)
    dseeds, dKt, dVt, dK, dV = o.route_bwd(*x, s, dY)
    for b in range(B):
        for h in range(H):
            l1 = s * Kt[b, h] @ seeds[h, 0]
            p1 = np.exp(l1 - l1.max())
            p1 /= p1.sum()
            q = p1 @ Vt[b, h]
            l2 = s * K[b, h] @ q
            p2 = np.exp(l2 - l2.max())
            p2 /= p2.sum()
            z = p2 @ V[b, h]
            dz = dY[b, h].sum(axis=0)
            np.testing.assert_allclose(dV[b, h], np.outer(p2, dz), atol=1e-12)
            ds2 = p2 * (V[b, h] @ dz - dz @ z)
            np.testing.assert_allclose(dK[b, h], s * np.outer(ds2, q), atol=1e-12)


BWD_PINS = [pin_bwd_finite_differences, pin_sdpa_bwd_vs_torch, pin_route_bwd_vs_torch,
            pin_bwd_identities, pin_bwd_one_route]


@pytest.mark.parametrize("pin", BWD_PINS, ids=[p.__name__ for p in BWD_PINS])
def test_bwd_pin(pin):
    pin(oracle_pkg.default())


def test_bwd_degenerate_shapes():
    """No tokens or no routes: every gradient is zero and nothing is NaN."""
    o = oracle_pkg.default()
    rng = np.random.default_rng(16)
    for (B, H, N, M, D) in [(2, 2, 0, 3, 4), (1, 2, 5, 0, 4), (0, 2, 5, 3, 4)]:
        x = _inputs(B, H, N, M, D, rng)
        g = o.route_bwd(*x, 0.5, _rand(rng, B, H, N, D))
        for a in g:
            assert np.all(a == 0.0)


@pytest.mark.parametrize("plant", [7, 8, 9, 10])
def test_bwd_pins_reject_planted_mistakes(plant, tmp_path):
    """Plants: the <dO, O> correction dropped, the key gradient taken through k instead of q,
    call 1 given only the decoder's query gradient, the seeds' gradient from one batch
    element. Each must fail at least one backward pin."""
    o = oracle_pkg.Oracle(plant=plant, build_dir=str(tmp_path))
    failed = []
    for pin in BWD_PINS:
        try:
            pin(o)
        except AssertionError:
            failed.append(pin.__name__)
    assert failed, f"plant {plant} passed every backward pin"


def test_golden_bwd_fixture_regression():
    """The oracle's backward still reproduces the stored small case
    (tests/golden/route_bwd_small.json, on the inputs of route_small.json), whose values the
    pins above were green for when it was written."""
    import json
    import os
    here = os.path.join(os.path.dirname(__file__), "golden")
    with open(os.path.join(here, "route_small.json")) as f:
        fwd = json.load(f)
    with open(os.path.join(here, "route_bwd_small.json")) as f:
        bwd = json.load(f)
    x = {k: np.array(v) for k, v in fwd["inputs"].items()}
    got = oracle_pkg.route_bwd(x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"], fwd["scale"],
                               np.array(bwd["dY"]))
    for name, g in zip(("dseeds", "dKt", "dVt", "dK", "dV"), got):
        want = np.array(bwd["expected"][name])
        assert g.shape == want.shape
        np.testing.assert_allclose(g, want, rtol=0, atol=1e-13, err_msg=name)
