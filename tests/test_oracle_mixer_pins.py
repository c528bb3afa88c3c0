"""Pins for the oracle's FLARE++ mixer layer (Fig. 1; eqs. flarepp_query_synthesis and
flarepp_mixer), against facts the oracle does not restate:
  * torch float64 in the paper's own pseudocode form (Fig. 1): four nn.functional.linear
    projections, three scaled_dot_product_attention calls, a head merge and an output linear;
  * channel-permutation weights turn the layer into the bare chain on permuted copies of X (a
    closed form through the pinned chain);
  * O is linear in Wo and in the value projection (Y is linear in V, Sec. 3.2);
  * the shared-projection variant (App. C.2) equals the four-projection layer with the K~, V~
    blocks set to copies of the K, V blocks.
"""
import math

import numpy as np
import torch
import torch.nn.functional as F

import oracle


def _case(B, H, N, M, D, rng, P=4):
    C = H * D
    X = rng.standard_normal((B, N, C))
    W_in = rng.standard_normal((P * C, C)) / math.sqrt(C)
    Wo = rng.standard_normal((C, C)) / math.sqrt(C)
    seeds = rng.standard_normal((H, M, D))
    return X, W_in, Wo, seeds


def _torch_mixer(X, W_in, Wo, seeds, s):
    t = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    X, W_in, Wo, seeds = t(X), t(W_in), t(Wo), t(seeds)
    B, N, C = X.shape
    H, M, D = seeds.shape
    proj = [F.linear(X, W_in[i * C:(i + 1) * C]) for i in range(W_in.shape[0] // C)]
    split = lambda T: T.reshape(B, N, H, D).transpose(1, 2)
    K, V = split(proj[0]), split(proj[1])
    Kt, Vt = (split(proj[2]), split(proj[3])) if len(proj) == 4 else (K, V)
    Qs = seeds.unsqueeze(0).expand(B, H, M, D)
    Q = F.scaled_dot_product_attention(Qs, Kt, Vt, scale=s)
    Z = F.scaled_dot_product_attention(Q, K, V, scale=s)
    Y = F.scaled_dot_product_attention(K, Q, Z, scale=s)
    return F.linear(Y.transpose(1, 2).reshape(B, N, C), Wo).numpy()


def test_mixer_vs_torch_pseudocode():
    rng = np.random.default_rng(21)
    for (B, H, N, M, D, P) in [(2, 2, 40, 6, 8, 4), (1, 4, 33, 5, 4, 4), (2, 3, 17, 9, 4, 2)]:
        X, W_in, Wo, seeds = _case(B, H, N, M, D, rng, P)
        s = 1.0 / math.sqrt(D)
        np.testing.assert_allclose(oracle.mixer(X, W_in, Wo, seeds, s),
                                   _torch_mixer(X, W_in, Wo, seeds, s), rtol=0, atol=1e-12)


def test_mixer_with_permutation_weights_is_the_chain():
    """W_in made of four channel permutations and Wo = I: the projections are permuted copies
    of X, so the layer is the chain on those copies, merged (written out by hand here)."""
    rng = np.random.default_rng(22)
    B, H, N, M, D = 2, 2, 30, 5, 4
    C = H * D
    X = rng.standard_normal((B, N, C))
    perms = [rng.permutation(C) for _ in range(4)]
    W_in = np.concatenate([np.eye(C)[p] for p in perms])  # row j of block i picks channel p_i[j]
    seeds = rng.standard_normal((H, M, D))
    s = 0.5
    split = lambda T: np.ascontiguousarray(T.reshape(B, N, H, D).transpose(0, 2, 1, 3))
    K, V, Kt, Vt = (split(X[..., p]) for p in perms)
    _, _, Y = oracle.route(seeds, Kt, Vt, K, V, s)
    want = Y.transpose(0, 2, 1, 3).reshape(B, N, C)
    np.testing.assert_allclose(oracle.mixer(X, W_in, np.eye(C), seeds, s), want, atol=1e-13)


def test_mixer_linearity():
    rng = np.random.default_rng(23)
    B, H, N, M, D = 1, 2, 25, 4, 8
    C = H * D
    X, W_in, Wo, seeds = _case(B, H, N, M, D, rng)
    s = 1.0 / math.sqrt(D)
    base = oracle.mixer(X, W_in, Wo, seeds, s)
    np.testing.assert_allclose(oracle.mixer(X, W_in, -2.5 * Wo, seeds, s), -2.5 * base,
                               atol=1e-12)
    W2 = W_in.copy()
    W2[C:2 * C] *= 3.0  # the value projection: Y is linear in V
    np.testing.assert_allclose(oracle.mixer(X, W2, Wo, seeds, s), 3.0 * base, atol=1e-11)


def test_shared_projection_layer():
    rng = np.random.default_rng(24)
    B, H, N, M, D = 2, 2, 20, 4, 4
    X, W2, Wo, seeds = _case(B, H, N, M, D, rng, P=2)
    W4 = np.concatenate([W2, W2])
    s = 0.4
    np.testing.assert_allclose(oracle.mixer(X, W2, Wo, seeds, s),
                               oracle.mixer(X, W4, Wo, seeds, s), atol=0)


def _torch_mixer_grads(X, W_in, Wo, seeds, s, dO):
    t = lambda a: torch.tensor(np.asarray(a, dtype=np.float64), requires_grad=True)
    tX, tW, tWo, ts = t(X), t(W_in), t(Wo), t(seeds)
    B, N, C = tX.shape
    H, M, D = ts.shape
    P = tW.shape[0] // C
    proj = [F.linear(tX, tW[i * C:(i + 1) * C]) for i in range(P)]
    split = lambda T: T.reshape(B, N, H, D).transpose(1, 2)
    K, V = split(proj[0]), split(proj[1])
    Kt, Vt = (split(proj[2]), split(proj[3])) if P == 4 else (K, V)
    Qs = ts.unsqueeze(0).expand(B, H, M, D)
    Q = F.scaled_dot_product_attention(Qs, Kt, Vt, scale=s)
    Z = F.scaled_dot_product_attention(Q, K, V, scale=s)
    Y = F.scaled_dot_product_attention(K, Q, Z, scale=s)
    O = F.linear(Y.transpose(1, 2).reshape(B, N, C), tWo)
    O.backward(torch.from_numpy(np.asarray(dO, dtype=np.float64)))
    return tuple(a.grad.numpy() for a in (tX, tW, tWo, ts))


def test_mixer_bwd_vs_torch_autograd():
    rng = np.random.default_rng(31)
    for (B, H, N, M, D, P) in [(2, 2, 30, 5, 4, 4), (1, 3, 25, 7, 4, 2), (2, 2, 17, 4, 8, 4)]:
        X, W_in, Wo, seeds = _case(B, H, N, M, D, rng, P)
        dO = rng.standard_normal(X.shape)
        s = 1.0 / math.sqrt(D)
        mine = oracle.mixer_bwd(X, W_in, Wo, seeds, s, dO)
        ref = _torch_mixer_grads(X, W_in, Wo, seeds, s, dO)
        for a, b in zip(mine, ref):
            np.testing.assert_allclose(a, b, rtol=0, atol=1e-11 * max(1.0, np.abs(b).max()))


def test_mixer_bwd_finite_differences():
    rng = np.random.default_rng(32)
    B, H, N, M, D, P = 1, 2, 6, 3, 2, 4
    X, W_in, Wo, seeds = _case(B, H, N, M, D, rng, P)
    dO = rng.standard_normal(X.shape)
    s = 0.6
    grads = oracle.mixer_bwd(X, W_in, Wo, seeds, s, dO)
    ins = [X, W_in, Wo, seeds]
    loss = lambda xs: float(np.sum(dO * oracle.mixer(*xs, s)))
    h = 1e-5
    for which in range(4):
        fd = np.zeros_like(ins[which])
        flat = ins[which].reshape(-1)
        for i in range(flat.size):
            keep = flat[i]
            flat[i] = keep + h
            lp = loss(ins)
            flat[i] = keep - h
            lm = loss(ins)
            flat[i] = keep
            fd.reshape(-1)[i] = (lp - lm) / (2 * h)
        np.testing.assert_allclose(grads[which], fd, rtol=0,
                                   atol=1e-7 * max(1.0, np.abs(fd).max()))
