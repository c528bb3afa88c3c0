"""Pins for the float64 oracle, against facts fixed by the paper and by mathematics.

None of these re-runs the oracle's own formula. Each check is one of:
  * a library routine (torch's float64 CPU scaled_dot_product_attention, scipy softmax /
    logsumexp) applied in the paper's own three-call form (Fig. 1; Sec. 3.2),
  * brute force: the explicit N x M routing matrices and W_eff = W_dec W_enc (Sec. 2,
    eq. prelim_flare_operator; Sec. 3.2),
  * invariants: rank(W_eff) <= M, row-stochastic W_eff probed through the oracle itself,
    convex-hull bounds, constant values, token-permutation equivariance, route-order
    invariance, independent (b, h) slices,
  * closed forms: scale 0, one token, one route, a two-token example worked by hand,
  * the shard merge of App. A.3 against the unsharded encoder and scipy's logsumexp.

``test_pins_reject_planted_mistakes`` rebuilds the oracle with one deliberate mistake at
a time and checks that at least one pin fails for each.
"""
import math

import numpy as np
import pytest
import scipy.special as sps
import torch
import torch.nn.functional as F

import oracle as oracle_pkg

RNG = np.random.default_rng(1234)


def _rand(*shape, scale=1.0, rng=None):
    rng = RNG if rng is None else rng
    return rng.standard_normal(shape) * scale


def _torch_sdpa(q, k, v, s):
    t = lambda a: torch.from_numpy(np.array(a, dtype=np.float64, order="C", copy=True))
    return F.scaled_dot_product_attention(t(q), t(k), t(v), scale=s).numpy()


def _chain_inputs(B, H, N, M, D, rng, key_scale=1.0):
    seeds = _rand(H, M, D, rng=rng)
    Kt = _rand(B, H, N, D, scale=key_scale, rng=rng)
    Vt = _rand(B, H, N, D, rng=rng)
    K = _rand(B, H, N, D, scale=key_scale, rng=rng)
    V = _rand(B, H, N, D, rng=rng)
    return seeds, Kt, Vt, K, V


# ---------------------------------------------------------------------------- pins
# Each pin takes an Oracle instance and raises AssertionError when it fails.

def pin_sdpa_vs_torch(o):
    """SDPA (eq. sdpa_definition) equals torch's float64 SDPA, N_q != N_k allowed."""
    rng = np.random.default_rng(1)
    for (G, nq, nk, D, s) in [(3, 5, 17, 4, 0.5), (2, 33, 7, 16, 0.25), (1, 1, 1, 3, 1.3),
                              (4, 8, 64, 8, 1.0 / math.sqrt(8))]:
        q, k, v = _rand(G, nq, D, rng=rng), _rand(G, nk, D, rng=rng), _rand(G, nk, D, rng=rng)
        out, lse = o.sdpa(q, k, v, s)
        np.testing.assert_allclose(out, _torch_sdpa(q, k, v, s), rtol=0, atol=1e-13)
        ref_lse = sps.logsumexp(s * np.einsum("gid,gjd->gij", q, k), axis=-1)
        np.testing.assert_allclose(lse, ref_lse, rtol=1e-14, atol=1e-13)


def pin_route_vs_torch_three_calls(o):
    """The chain equals three library SDPA calls in the paper's order (Fig. 1, Sec. 3.2)."""
    rng = np.random.default_rng(2)
    for (B, H, N, M, D) in [(2, 3, 37, 5, 4), (1, 2, 130, 16, 8), (1, 1, 9, 12, 3)]:
        s = 1.0 / math.sqrt(D)
        seeds, Kt, Vt, K, V = _chain_inputs(B, H, N, M, D, rng)
        Q, Z, Y = o.route(seeds, Kt, Vt, K, V, s)
        seeds_b = np.broadcast_to(seeds, (B, H, M, D))
        Qr = _torch_sdpa(seeds_b, Kt, Vt, s)
        Zr = _torch_sdpa(Qr, K, V, s)
        Yr = _torch_sdpa(K, Qr, Zr, s)
        np.testing.assert_allclose(Q, Qr, rtol=0, atol=1e-13)
        np.testing.assert_allclose(Z, Zr, rtol=0, atol=1e-13)
        np.testing.assert_allclose(Y, Yr, rtol=0, atol=1e-12)


def _softmax_rows(x):
    return sps.softmax(x, axis=-1)


def pin_brute_force_matrices(o):
    """Explicit A1, A2 in R^{MxN}, A3 in R^{NxM}: Q = A1 Vt and Y = (A3 A2) V (Sec. 2-3.2)."""
    rng = np.random.default_rng(3)
    for (N, M, D) in [(64, 6, 4), (200, 16, 8), (31, 40, 2)]:
        s = 0.7
        seeds, Kt, Vt, K, V = (a[0, 0] if a.ndim == 4 else a[0]
                               for a in _chain_inputs(1, 1, N, M, D, rng))
        Q, Z, Y = o.route(seeds[None], Kt[None, None], Vt[None, None], K[None, None],
                          V[None, None], s)
        Q, Z, Y = Q[0, 0], Z[0, 0], Y[0, 0]
        A1 = _softmax_rows(s * seeds @ Kt.T)          # M x N, over tokens
        Qb = A1 @ Vt
        A2 = _softmax_rows(s * Qb @ K.T)              # M x N, over tokens
        A3 = _softmax_rows(s * K @ Qb.T)              # N x M, over routes
        W = A3 @ A2                                   # N x N
        np.testing.assert_allclose(Q, Qb, rtol=0, atol=1e-13)
        np.testing.assert_allclose(Z, A2 @ V, rtol=0, atol=1e-13)
        np.testing.assert_allclose(Y, W @ V, rtol=0, atol=1e-13)


def _probe_weff(o, seeds, Kt, Vt, K):
    """Recover W_eff (N x N) from the oracle alone: Y is linear in V (eq. prelim_flare_operator),
    so feeding unit vectors in V reads off columns, D of them per call."""
    H, M, D = seeds.shape
    N = K.shape[2]
    W = np.zeros((N, N))
    for j0 in range(0, N, D):
        V = np.zeros((1, 1, N, D))
        cols = list(range(j0, min(N, j0 + D)))
        for d, j in enumerate(cols):
            V[0, 0, j, d] = 1.0
        _, _, Y = o.route(seeds, Kt, Vt, K, V, 1.0 / math.sqrt(D))
        for d, j in enumerate(cols):
            W[:, j] = Y[0, 0, :, d]
    return W


def pin_rank_and_stochastic(o):
    """W_eff = W_dec W_enc has rank <= M and is row-stochastic (Sec. 3.2; Fig. 1)."""
    rng = np.random.default_rng(4)
    for (N, M, D) in [(96, 5, 8), (128, 12, 16)]:
        seeds, Kt, Vt, K, _ = _chain_inputs(1, 1, N, M, D, rng)
        W = _probe_weff(o, seeds, Kt, Vt, K)
        sv = np.linalg.svd(W, compute_uv=False)
        assert sv[M] / sv[0] < 1e-12, (sv[M] / sv[0])
        assert sv[M - 1] / sv[0] > 1e-9  # the bound is attained for generic inputs
        assert W.min() > 0.0
        np.testing.assert_allclose(W.sum(axis=1), 1.0, rtol=0, atol=1e-14)


def pin_convex_hull(o):
    """Every softmax row is a convex weight vector, so Q lies in the hull of Vt and Z, Y
    in the hull of V, per channel."""
    rng = np.random.default_rng(5)
    B, H, N, M, D = 2, 2, 300, 20, 8
    seeds, Kt, Vt, K, V = _chain_inputs(B, H, N, M, D, rng, key_scale=3.0)
    Q, Z, Y = o.route(seeds, Kt, Vt, K, V, 1.0 / math.sqrt(D))
    for out, src in ((Q, Vt), (Z, V), (Y, V)):
        lo = src.min(axis=2, keepdims=True)
        hi = src.max(axis=2, keepdims=True)
        assert np.all(out >= lo - 1e-13) and np.all(out <= hi + 1e-13)


def pin_constant_values(o):
    """Constant V per channel gives Y == V; constant Vt gives equal Q rows, a uniform
    decode, and Y[n] = SDPA(q, K, V) for every token n."""
    rng = np.random.default_rng(6)
    B, H, N, M, D = 1, 2, 50, 7, 4
    s = 0.5
    seeds, Kt, Vt, K, V = _chain_inputs(B, H, N, M, D, rng)
    Vc = np.broadcast_to(rng.standard_normal((B, H, 1, D)), (B, H, N, D)).copy()
    _, _, Y = o.route(seeds, Kt, Vt, K, Vc, s)
    np.testing.assert_allclose(Y, Vc, rtol=0, atol=1e-14)
    Vtc = np.broadcast_to(rng.standard_normal((B, H, 1, D)), (B, H, N, D)).copy()
    Q, Z, Y = o.route(seeds, Kt, Vtc, K, V, s)
    np.testing.assert_allclose(Q, np.broadcast_to(Vtc[:, :, :1], Q.shape), rtol=0, atol=1e-14)
    z0 = _torch_sdpa(Vtc[:, :, :1], K, V, s)  # [B,H,1,D]
    np.testing.assert_allclose(Y, np.broadcast_to(z0, Y.shape), rtol=0, atol=1e-13)


def pin_closed_forms(o):
    """scale 0 -> every softmax uniform: Q = mean(Vt), Z = Y = mean(V).
    N = 1 -> Q = Vt[0], Z = V[0], Y = V[0].  M = 1 -> Y[n] = SDPA(SDPA(q, Kt, Vt), K, V)."""
    rng = np.random.default_rng(7)
    B, H, N, M, D = 2, 3, 41, 6, 5
    seeds, Kt, Vt, K, V = _chain_inputs(B, H, N, M, D, rng)
    Q, Z, Y = o.route(seeds, Kt, Vt, K, V, 0.0)
    np.testing.assert_allclose(Q, np.broadcast_to(Vt.mean(2, keepdims=True), Q.shape), atol=1e-14)
    np.testing.assert_allclose(Z, np.broadcast_to(V.mean(2, keepdims=True), Z.shape), atol=1e-14)
    np.testing.assert_allclose(Y, np.broadcast_to(V.mean(2, keepdims=True), Y.shape), atol=1e-14)

    seeds1, Kt1, Vt1, K1, V1 = _chain_inputs(B, H, 1, M, D, rng)
    Q, Z, Y = o.route(seeds1, Kt1, Vt1, K1, V1, 0.9)
    np.testing.assert_array_equal(Q, np.broadcast_to(Vt1, Q.shape))
    np.testing.assert_array_equal(Z, np.broadcast_to(V1, Z.shape))
    np.testing.assert_allclose(Y, V1, rtol=1e-15, atol=1e-15)

    s = 0.45
    seedsm, Ktm, Vtm, Km, Vm = _chain_inputs(B, H, N, 1, D, rng)
    _, _, Y = o.route(seedsm, Ktm, Vtm, Km, Vm, s)
    q = _torch_sdpa(np.broadcast_to(seedsm, (B, H, 1, D)), Ktm, Vtm, s)
    z = _torch_sdpa(q, Km, Vm, s)
    np.testing.assert_allclose(Y, np.broadcast_to(z, Y.shape), rtol=0, atol=1e-13)


def pin_two_token_hand_example(o):
    """A hand-worked case, D = 1, N = 2, M = 2, s = 1 (eqs. flarepp_dynamic_query, flarepp_mixer).

    seeds (ln 3, 0), Kt (0, 1), Vt (2, 6):
      route 0 logits (0, ln 3) -> weights (1/4, 3/4) -> Q0 = 2/4 + 18/4 = 5
      route 1 logits (0, 0)    -> weights (1/2, 1/2) -> Q1 = 4
    K (0, k) with k = ln(2)/5, V (3, 9):
      route 0 logits (0, ln 2)   -> weights (1/3, 2/3) -> Z0 = 1 + 6 = 7
      route 1 logits (0, 4k)     -> w = 2^0.8 / (1 + 2^0.8) -> Z1 = 3 + 6 w
    decode, token 0 (key 0): all logits 0 -> Y0 = (Z0 + Z1) / 2
    decode, token 1 (key k): logits (5k, 4k) = (ln 2, 0.8 ln 2) -> weights proportional to
      (2, 2^0.8) -> Y1 = (2 Z0 + 2^0.8 Z1) / (2 + 2^0.8)
    """
    k = math.log(2.0) / 5.0
    seeds = np.array([[[math.log(3.0)], [0.0]]])
    Kt = np.array([[[[0.0], [1.0]]]])
    Vt = np.array([[[[2.0], [6.0]]]])
    K = np.array([[[[0.0], [k]]]])
    V = np.array([[[[3.0], [9.0]]]])
    Q, Z, Y = o.route(seeds, Kt, Vt, K, V, 1.0)
    w = 2 ** 0.8 / (1 + 2 ** 0.8)
    z0, z1 = 7.0, 3.0 + 6.0 * w
    np.testing.assert_allclose(Q.ravel(), [5.0, 4.0], rtol=1e-15, atol=1e-15)
    np.testing.assert_allclose(Z.ravel(), [z0, z1], rtol=1e-15, atol=1e-15)
    np.testing.assert_allclose(Y.ravel(), [(z0 + z1) / 2, (2 * z0 + 2 ** 0.8 * z1) / (2 + 2 ** 0.8)],
                               rtol=1e-15, atol=1e-14)


def pin_symmetries(o):
    """Token permutation equivariance (no token order, App. A.1), invariance to the order of
    the seed rows, and independent (b, h) slices."""
    rng = np.random.default_rng(8)
    B, H, N, M, D = 2, 2, 77, 9, 4
    s = 0.5
    seeds, Kt, Vt, K, V = _chain_inputs(B, H, N, M, D, rng)
    _, _, Y = o.route(seeds, Kt, Vt, K, V, s)
    p = rng.permutation(N)
    _, _, Yp = o.route(seeds, Kt[:, :, p], Vt[:, :, p], K[:, :, p], V[:, :, p], s)
    np.testing.assert_allclose(Yp, Y[:, :, p], rtol=0, atol=1e-13)
    r = rng.permutation(M)
    _, _, Yr = o.route(seeds[:, r], Kt, Vt, K, V, s)
    np.testing.assert_allclose(Yr, Y, rtol=0, atol=1e-13)
    for b in range(B):
        for h in range(H):
            _, _, Ys = o.route(seeds[h:h + 1], Kt[b:b + 1, h:h + 1], Vt[b:b + 1, h:h + 1],
                               K[b:b + 1, h:h + 1], V[b:b + 1, h:h + 1], s)
            np.testing.assert_array_equal(Ys[0, 0], Y[b, h])


def pin_sharded_merge(o):
    """Sharded encode + stable LSE merge equals the encoder on the whole sequence (App. A.2-A.3),
    with shards that do not divide N and extra empty shards (L_r = -inf, O_r = 0)."""
    rng = np.random.default_rng(9)
    G, nq, nk, D, s = 3, 6, 101, 4, 0.8
    q, k, v = _rand(G, nq, D, rng=rng), _rand(G, nk, D, scale=3.0, rng=rng), _rand(G, nk, D, rng=rng)
    ref = _torch_sdpa(q, k, v, s)
    ref_lse = sps.logsumexp(s * np.einsum("gid,gjd->gij", q, k), axis=-1)
    for chunk, n_empty in [(1, 0), (7, 0), (10, 2), (100, 1), (101, 0), (500, 3)]:
        out, lse = o.encode_sharded(q, k, v, s, chunk, n_empty)
        np.testing.assert_allclose(out, ref, rtol=0, atol=1e-13)
        np.testing.assert_allclose(lse, ref_lse, rtol=1e-14, atol=1e-12)


def pin_large_logits(o):
    """Stable softmax: logits of order 10^3 must not overflow (torch's SDPA is stable)."""
    rng = np.random.default_rng(10)
    B, H, N, M, D = 1, 2, 40, 5, 4
    seeds, Kt, Vt, K, V = _chain_inputs(B, H, N, M, D, rng, key_scale=30.0)
    s = 10.0
    Q, Z, Y = o.route(seeds * 10.0, Kt, Vt, K, V, s)
    assert np.all(np.isfinite(Y))
    seeds_b = np.broadcast_to(seeds * 10.0, (B, H, M, D))
    Qr = _torch_sdpa(seeds_b, Kt, Vt, s)
    Zr = _torch_sdpa(Qr, K, V, s)
    np.testing.assert_allclose(Q, Qr, rtol=0, atol=1e-12)
    np.testing.assert_allclose(Z, Zr, rtol=0, atol=1e-10)


def pin_flare_brute_force(o):
    """FLARE (Sec. 3, eqs. prelim_flare_sdpa and prelim_flare_operator): explicit
    W_enc = softmax(s Q K^T) (M x N, over tokens) and W_dec = softmax(s K Q^T) (N x M, over
    routes) give Z = W_enc V and Y = W_dec W_enc V, with rank(W_dec W_enc) <= M; also two
    torch float64 SDPA calls in the paper's order."""
    rng = np.random.default_rng(21)
    for (N, M, D, s) in [(64, 6, 4, 0.7), (150, 16, 8, 0.35), (29, 40, 2, 1.1)]:
        Q, K, V = _rand(1, M, D, rng=rng), _rand(1, 1, N, D, rng=rng), _rand(1, 1, N, D, rng=rng)
        Z, Y = o.flare(Q, K, V, s)
        Wenc = _softmax_rows(s * Q[0] @ K[0, 0].T)
        Wdec = _softmax_rows(s * K[0, 0] @ Q[0].T)
        np.testing.assert_allclose(Z[0, 0], Wenc @ V[0, 0], rtol=0, atol=1e-13)
        np.testing.assert_allclose(Y[0, 0], Wdec @ Wenc @ V[0, 0], rtol=0, atol=1e-13)
        sv = np.linalg.svd(Wdec @ Wenc, compute_uv=False)
        if M < N:
            assert sv[M] / sv[0] < 1e-12
        Zr = _torch_sdpa(Q[None], K, V, s)
        np.testing.assert_allclose(Y, _torch_sdpa(K, Q[None], Zr, s), rtol=0, atol=1e-12)


def pin_flare_is_the_chain_without_call_one(o):
    """FLARE++ is FLARE whose queries come from call 1 (Sec. 3.2): the chain's Z and Y equal
    FLARE's on the chain's own Q; for B > 1 the learned Q is shared by the batch."""
    rng = np.random.default_rng(22)
    for (N, M, D) in [(70, 8, 4), (33, 3, 8)]:
        s = 1.0 / math.sqrt(D)
        seeds, Kt, Vt, K, V = _chain_inputs(1, 2, N, M, D, rng)
        Q, Z, Y = o.route(seeds, Kt, Vt, K, V, s)
        Zf, Yf = o.flare(Q[0], K, V, s)
        np.testing.assert_allclose(Zf, Z, rtol=0, atol=1e-14)
        np.testing.assert_allclose(Yf, Y, rtol=0, atol=1e-14)
    Qh = _rand(2, 5, 4, rng=rng)
    K, V = _rand(3, 2, 20, 4, rng=rng), _rand(3, 2, 20, 4, rng=rng)
    Z, Y = o.flare(Qh, K, V, 0.5)
    for b in range(3):
        Zb, Yb = o.flare(Qh, K[b:b + 1], V[b:b + 1], 0.5)
        np.testing.assert_allclose(Z[b:b + 1], Zb, rtol=0, atol=0)
        np.testing.assert_allclose(Y[b:b + 1], Yb, rtol=0, atol=0)


def pin_flare_closed_forms(o):
    """scale 0: every route and token averages V uniformly; one route: every token gets Z."""
    rng = np.random.default_rng(23)
    Q, K, V = _rand(2, 6, 4, rng=rng), _rand(1, 2, 25, 4, rng=rng), _rand(1, 2, 25, 4, rng=rng)
    Z, Y = o.flare(Q, K, V, 0.0)
    mean = V.mean(axis=2, keepdims=True)
    np.testing.assert_allclose(Z, np.broadcast_to(mean, Z.shape), rtol=0, atol=1e-14)
    np.testing.assert_allclose(Y, np.broadcast_to(mean, Y.shape), rtol=0, atol=1e-14)
    Z, Y = o.flare(Q[:, :1], K, V, 0.8)
    np.testing.assert_allclose(Y, np.broadcast_to(Z, Y.shape), rtol=0, atol=1e-14)


PINS = [pin_sdpa_vs_torch, pin_route_vs_torch_three_calls, pin_brute_force_matrices,
        pin_rank_and_stochastic, pin_convex_hull, pin_constant_values, pin_closed_forms,
        pin_two_token_hand_example, pin_symmetries, pin_sharded_merge, pin_large_logits,
        pin_flare_brute_force, pin_flare_is_the_chain_without_call_one, pin_flare_closed_forms]


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_pin(pin):
    pin(oracle_pkg.default())


def test_empty_rows():
    """A row with no keys gives output 0 and L = -inf, never NaN (App. A.3); N = 0 tokens
    gives zero Q and Z and an empty Y."""
    o = oracle_pkg.default()
    out, lse = o.sdpa(np.ones((2, 3, 4)), np.zeros((2, 0, 4)), np.zeros((2, 0, 4)), 0.5)
    assert np.all(out == 0.0) and np.all(np.isneginf(lse))
    Q, Z, Y = o.route(np.ones((2, 3, 4)), *(np.zeros((1, 2, 0, 4)),) * 4, 0.5)
    assert np.all(Q == 0) and np.all(Z == 0) and Y.shape == (1, 2, 0, 4)


def test_thread_count_invariance():
    """Rows are independent, so the thread count never changes a bit of the result."""
    o = oracle_pkg.default()
    rng = np.random.default_rng(11)
    args = _chain_inputs(2, 2, 500, 24, 8, rng)
    n0 = o.max_threads()
    try:
        o.set_threads(1)
        a = o.route(*args, 0.35)
        o.set_threads(max(2, n0))
        b = o.route(*args, 0.35)
    finally:
        o.set_threads(n0)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)


@pytest.mark.parametrize("plant", [1, 2, 3, 4, 5, 6])
def test_pins_reject_planted_mistakes(plant, tmp_path):
    """Build the oracle with one planted mistake (no max subtraction, wrong decode queries,
    decode against the seeds, scale applied twice, a shard lost in the merge, the last key
    dropped) and check that some pin fails."""
    o = oracle_pkg.Oracle(plant=plant, build_dir=str(tmp_path))
    failed = []
    for pin in PINS:
        try:
            with np.errstate(all="ignore"):
                pin(o)
        except AssertionError:
            failed.append(pin.__name__)
    assert failed, f"plant {plant} passed every pin"


def test_golden_fixture_regression():
    """The oracle still reproduces the stored small case (tests/golden/route_small.json)."""
    import json
    import os
    path = os.path.join(os.path.dirname(__file__), "golden", "route_small.json")
    with open(path) as f:
        doc = json.load(f)
    x = {k: np.array(v) for k, v in doc["inputs"].items()}
    Q, Z, Y = oracle_pkg.route(x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"], doc["scale"])
    for name, got in (("Q", Q), ("Z", Z), ("Y", Y)):
        np.testing.assert_allclose(got, np.array(doc["expected"][name]), rtol=0, atol=1e-14)
