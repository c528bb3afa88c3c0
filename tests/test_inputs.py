"""The seeded workload generators: determinism, shapes, dtypes and the stated distributions."""
import math

import torch

from paper_2608_11519_gb300 import inputs


def test_workload_table():
    w = inputs.get("mesh3d")
    assert (w.B, w.H, w.N, w.M, w.D, w.dtype, w.n_centres) == (1, 8, 1048576, 512, 32, "bf16", 4096)
    assert inputs.get("tiny").dtype == "f32"
    assert len([k for k in inputs.WORKLOADS if k.startswith("sweep_")]) == 24
    assert math.isclose(inputs.get("pde2d").scale, 1 / math.sqrt(32))


def test_deterministic_and_shaped():
    w = inputs.get("pde2d").with_(B=2, N=2048)
    a = inputs.make_inputs(w, seed=5)
    b = inputs.make_inputs(w, seed=5)
    c = inputs.make_inputs(w, seed=6)
    for k in a:
        assert torch.equal(a[k], b[k])
        assert a[k].dtype == torch.bfloat16
    assert not torch.equal(a["K"], c["K"])
    assert a["seeds"].shape == (8, 128, 32)
    assert a["K"].shape == (2, 8, 2048, 32)


def test_distributions():
    w = inputs.get("pde2d").with_(B=1, N=65536)
    x = inputs.make_inputs(w, seed=0)
    V = x["V"].float()
    assert abs(V.mean().item()) < 0.02 and abs(V.std().item() - 1) < 0.02
    # clustered keys: the spread is the centre spread 1.5 plus 0.5 noise per channel
    K = x["K"].float()
    assert 1.2 < K.std().item() < 2.2
    # within a head tokens concentrate on at most 64 centres: the pairwise nearest-centre
    # residual is the 0.5 noise
    k0 = K[0, 0, :4096]
    d = torch.cdist(k0[:256], k0)
    d.fill_diagonal_(float("inf"))
    assert d.min(dim=1).values.median().item() < 0.5 * math.sqrt(2 * 32) * 1.2


def test_f64_view_is_exact():
    w = inputs.get("tiny").with_(N=64)
    x = inputs.make_inputs(w, seed=1)
    y = inputs.to_f64_numpy(x)
    for k in x:
        assert torch.equal(torch.from_numpy(y[k]).to(x[k].dtype), x[k])
