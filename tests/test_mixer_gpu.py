"""GPU parity of the FLARE++ mixer layer (Fig. 1: projections, chain, head merge, output
projection) against the float64 oracle, through the C ABI.

Tolerance: max|O - O_ref| <= 2e-2 * max(1, max|O_ref|) (bf16 inputs, float32 accumulation;
the projections are stored in bf16 before the chain reads them, as the chain's own inputs are).
With permutation weights every projection output is one input value (a sum with one nonzero
term), so there the layer must equal the chain on the permuted copies bit for bit.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_11519_gb300 import flarepp

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    flarepp.load()
    torch.cuda.set_device(0)


def _np(t):
    return t.detach().to("cpu", torch.float64).numpy()


def _case(B, H, N, M, D, P, seed):
    g = torch.Generator().manual_seed(seed)
    C = H * D
    X = torch.randn(B, N, C, generator=g).to(torch.bfloat16)
    W_in = (torch.randn(P * C, C, generator=g) / math.sqrt(C)).to(torch.bfloat16)
    Wo = (torch.randn(C, C, generator=g) / math.sqrt(C)).to(torch.bfloat16)
    seeds = torch.randn(H, M, D, generator=g).to(torch.bfloat16)
    return X, W_in, Wo, seeds


SHAPES = [
    # B, H, N, M, D, P
    (1, 8, 3000, 128, 32, 4),
    (2, 2, 500, 64, 32, 4),
    (2, 4, 300, 40, 16, 4),
    (1, 2, 129, 20, 64, 4),
    (1, 8, 1000, 96, 32, 2),
    (3, 3, 200, 30, 16, 2),   # C = 48: one head per tile
    (1, 4, 600, 1024, 64, 4),  # D = 64 and a large route count
]


@pytest.mark.parametrize("shape", SHAPES, ids=[str(s) for s in SHAPES])
def test_mixer_matches_oracle(shape):
    B, H, N, M, D, P = shape
    X, W_in, Wo, seeds = _case(B, H, N, M, D, P, 7)
    s = 1.0 / math.sqrt(D)
    O = flarepp.mixer_fwd(X.cuda(), W_in.cuda(), Wo.cuda(), seeds.cuda(), s)
    torch.cuda.synchronize()
    want = oracle.mixer(_np(X), _np(W_in), _np(Wo), _np(seeds), s)
    got = _np(O)
    bound = 2e-2 * max(1.0, float(np.abs(want).max()))
    assert float(np.abs(got - want).max()) <= bound


def test_mixer_with_permutation_weights_is_the_chain_exactly():
    B, H, N, M, D = 2, 4, 700, 64, 32
    C = H * D
    g = torch.Generator().manual_seed(3)
    X = torch.randn(B, N, C, generator=g).to(torch.bfloat16)
    perms = [torch.randperm(C, generator=g) for _ in range(4)]
    W_in = torch.cat([torch.eye(C)[p] for p in perms]).to(torch.bfloat16)
    Wo = torch.eye(C).to(torch.bfloat16)
    seeds = torch.randn(H, M, D, generator=g).to(torch.bfloat16)
    s = 1.0 / math.sqrt(D)
    O = flarepp.mixer_fwd(X.cuda(), W_in.cuda(), Wo.cuda(), seeds.cuda(), s)
    split = lambda T: T.reshape(B, N, H, D).transpose(1, 2).contiguous().cuda()
    K, V, Kt, Vt = (split(X[..., p]) for p in perms)
    Y = flarepp.route_fwd(seeds.cuda(), Kt, Vt, K, V, s)
    torch.cuda.synchronize()
    merged = Y.transpose(1, 2).reshape(B, N, C)
    assert torch.equal(O, merged)


def test_mixer_degenerate_shapes():
    X, W_in, Wo, seeds = _case(1, 2, 50, 0, 16, 4, 1)  # M = 0: Y = 0, so O = 0
    O = torch.full_like(X, 3.0).cuda()
    flarepp.mixer_fwd(X.cuda(), W_in.cuda(), Wo.cuda(), seeds.cuda(), O=O)
    torch.cuda.synchronize()
    assert not torch.any(O != 0)
    X, W_in, Wo, seeds = _case(2, 2, 0, 8, 16, 4, 1)  # N = 0: nothing to do
    O = flarepp.mixer_fwd(X.cuda(), W_in.cuda(), Wo.cuda(), seeds.cuda())
    assert O.numel() == 0


def test_mixer_guard_bands_untouched():
    """O is written inside its tensor only (the TMA stores clip rows beyond N)."""
    X, W_in, Wo, seeds = _case(2, 4, 333, 48, 32, 4, 9)
    band = 4096
    buf = torch.full((X.numel() + 2 * band,), 5.0, dtype=X.dtype, device="cuda")
    O = buf[band:band + X.numel()].view(X.shape)
    flarepp.mixer_fwd(X.cuda(), W_in.cuda(), Wo.cuda(), seeds.cuda(), O=O)
    torch.cuda.synchronize()
    assert torch.all(buf[:band] == 5.0) and torch.all(buf[-band:] == 5.0)
    assert torch.isfinite(O.float()).all()


BWD_SHAPES = [
    # B, H, N, M, D, P
    (1, 8, 2000, 128, 32, 4),
    (2, 2, 500, 64, 32, 4),
    (1, 4, 300, 40, 16, 2),
    (2, 2, 257, 20, 64, 4),
    (1, 1, 130, 16, 32, 2),   # C = D: one head
    (1, 6, 300, 32, 32, 4),   # C = 192: weight-gradient row tiles cross projections mid-tile
]


@pytest.mark.parametrize("shape", BWD_SHAPES, ids=[str(s) for s in BWD_SHAPES])
def test_mixer_bwd_matches_oracle(shape):
    """The layer's gradients (App. A.5 through the projections) against the oracle; each
    tensor within 2e-2 of its own scale, as for the chain's backward."""
    B, H, N, M, D, P = shape
    X, W_in, Wo, seeds = _case(B, H, N, M, D, P, 13)
    g = torch.Generator().manual_seed(14)
    dO = torch.randn(X.shape, generator=g).to(torch.bfloat16)
    s = 1.0 / math.sqrt(D)
    dev = [t.cuda() for t in (X, W_in, Wo, seeds)]
    O, saved = flarepp.mixer_fwd_train(*dev, s)
    grads = flarepp.mixer_bwd(*dev, saved, dO.cuda(), s)
    torch.cuda.synchronize()
    O_plain = flarepp.mixer_fwd(*dev, s)
    torch.cuda.synchronize()
    if D > 32:
        assert torch.equal(O, O_plain)
    else:
        # the training forward's calls 2 and 3 take Q as a hi/lo operand pair: O differs from
        # the plain forward's by bf16 rounding only
        a, b = O.float(), O_plain.float()
        assert float((a - b).abs().max()) <= 2e-2 * max(1.0, float(b.abs().max()))
    want = oracle.mixer_bwd(_np(X), _np(W_in), _np(Wo), _np(seeds), s, _np(dO))
    for name, got, ref in zip(("dX", "dW_in", "dWo", "dseeds"), grads, want):
        got = _np(got)
        assert got.shape == ref.shape, name
        bound = 2e-2 * max(1.0, float(np.abs(ref).max()))
        err = float(np.abs(got - ref).max())
        assert err <= bound, f"{name}: {err} > {bound}"


def test_mixer_full_size_pde2d():
    """The mixer layer and its backward at the pde2d workload's full size (B = 4, H = 8,
    N = 16,384, M = 128, D = 32), inputs from the shared input recipe."""
    from paper_2608_11519_gb300 import inputs
    w = inputs.get("pde2d")
    m = inputs.make_mixer_inputs(w, 2)
    md = {k: v.cuda() for k, v in m.items()}
    args = (md["X"], md["W_in"], md["Wo"], md["seeds"])
    g = torch.Generator().manual_seed(3)
    dO = torch.randn(md["X"].shape, generator=g).to(torch.bfloat16)
    O, saved = flarepp.mixer_fwd_train(*args, w.scale)
    grads = flarepp.mixer_bwd(*args, saved, dO.cuda(), w.scale)
    torch.cuda.synchronize()
    f = inputs.to_f64_numpy(m)
    want_O = oracle.mixer(f["X"], f["W_in"], f["Wo"], f["seeds"], w.scale)
    want = oracle.mixer_bwd(f["X"], f["W_in"], f["Wo"], f["seeds"], w.scale, _np(dO))
    for name, got, ref in zip(("O", "dX", "dW_in", "dWo", "dseeds"), (O,) + tuple(grads),
                              (want_O,) + tuple(want)):
        bound = 2e-2 * max(1.0, float(np.abs(ref).max()))
        err = float(np.abs(_np(got) - ref).max())
        assert err <= bound, f"{name}: {err} > {bound}"
