"""Seeded synthetic workloads for the FLARE++ routing chain.

This module only draws random tensors; it holds none of the routing chain's arithmetic.
Both the CUDA path and the float64 oracle receive the tensors it returns.

The shapes stand in for the paper's workloads, none of whose data is available here:
  * ``tiny``      B1 H4 N1024 M32 D16, float32, all i.i.d. N(0,1)
  * ``pde2d``     B4 H8 N16384 M128 D32, bf16; K and Kt clustered around 64 centres
                  (a 2D PDE mesh of ~16K points, H=8 heads as in App. B.1)
  * ``longseq``   B32 H8 N4096 M256 D32, bf16; all i.i.d. N(0,1) (a long-sequence
                  classification shape)
  * ``mesh3d``    B1 H8 N1,048,576 M512 D32, bf16; K and Kt clustered around 4096 centres
                  (the 10^6-point single-GPU and context-parallel sweeps of App. A.7, C.3)
  * ``sweep_M{m}_D{d}``  B1 H8 N262144, M in 16..2048, D in {16, 32, 64}, bf16 i.i.d.

Recipe (one ``torch.Generator`` seeded with ``seed``; draw order seeds, Kt, Vt, K, V):
  * i.i.d. tensors: ``randn`` in float32, then rounded to the workload dtype.
  * clustered tensors (K and Kt when ``n_centres`` > 0): per head an independent set of
    ``n_centres`` centres drawn from N(0, 1.5^2) per channel; every (b, h, n) token picks a
    centre uniformly; the token is ``0.5 * N(0, 1) + centre``. This gives the peaked
    encoder softmaxes of smooth physical fields.
  * softmax scale 1/sqrt(D) (Sec. 2, eq. sdpa_definition).
"""
from dataclasses import dataclass, replace
import math

import torch


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    H: int
    N: int
    M: int
    D: int
    dtype: str  # "f32" or "bf16"
    n_centres: int = 0  # 0 = i.i.d. keys, else clustered K and Kt

    @property
    def torch_dtype(self):
        return torch.float32 if self.dtype == "f32" else torch.bfloat16

    @property
    def scale(self) -> float:
        return 1.0 / math.sqrt(self.D)

    @property
    def elt_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)

    def describe(self) -> str:
        kind = f"clustered K/Kt ({self.n_centres} centres)" if self.n_centres else "iid N(0,1)"
        return (f"{self.name}: B={self.B} H={self.H} N={self.N} M={self.M} D={self.D} "
                f"{self.dtype}, {kind}")


WORKLOADS = {
    "tiny": Workload("tiny", 1, 4, 1024, 32, 16, "f32"),
    "pde2d": Workload("pde2d", 4, 8, 16384, 128, 32, "bf16", 64),
    "longseq": Workload("longseq", 32, 8, 4096, 256, 32, "bf16"),
    "mesh3d": Workload("mesh3d", 1, 8, 1048576, 512, 32, "bf16", 4096),
}
SWEEP_M = (16, 32, 64, 128, 256, 512, 1024, 2048)
SWEEP_D = (16, 32, 64)
for _m in SWEEP_M:
    for _d in SWEEP_D:
        WORKLOADS[f"sweep_M{_m}_D{_d}"] = Workload(f"sweep_M{_m}_D{_d}", 1, 8, 262144, _m, _d,
                                                   "bf16")


def get(name: str) -> Workload:
    return WORKLOADS[name]


def _clustered(gen, B, H, N, D, n_centres, device):
    centres = torch.randn(H, n_centres, D, generator=gen, device=device) * 1.5
    idx = torch.randint(0, n_centres, (B, H, N), generator=gen, device=device)
    noise = torch.randn(B, H, N, D, generator=gen, device=device) * 0.5
    hidx = torch.arange(H, device=device).view(1, H, 1).expand(B, H, N)
    return noise + centres[hidx, idx]


def make_inputs(w: Workload, seed: int = 0, device="cpu"):
    """Draw (seeds [H,M,D], Kt, Vt, K, V [B,H,N,D]) for workload ``w`` in its dtype.

    The same ``seed`` and ``device`` give the same tensors on every call.
    """
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    B, H, N, M, D = w.B, w.H, w.N, w.M, w.D
    dt = w.torch_dtype

    def iid(*shape):
        return torch.randn(*shape, generator=gen, device=device).to(dt)

    def keys():
        if w.n_centres:
            return _clustered(gen, B, H, N, D, w.n_centres, device).to(dt)
        return iid(B, H, N, D)

    seeds = iid(H, M, D)
    Kt = keys()
    Vt = iid(B, H, N, D)
    K = keys()
    V = iid(B, H, N, D)
    return {"seeds": seeds, "Kt": Kt, "Vt": Vt, "K": K, "V": V}


def make_output_grad(w: Workload, seed: int = 0, device="cpu"):
    """Draw an output gradient dY [B,H,N,D] for workload ``w``: i.i.d. N(0,1) in its dtype,
    from a stream separate from :func:`make_inputs` (seed offset by 7919)."""
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed) + 7919)
    return torch.randn(w.B, w.H, w.N, w.D, generator=gen, device=device).to(w.torch_dtype)


def make_mixer_inputs(w: Workload, seed: int = 0, device="cpu", n_proj: int = 4):
    """Draw the mixer layer's inputs for workload ``w`` (C = H * D) in its dtype: X [B, N, C]
    i.i.d. N(0, 1); W_in [n_proj * C, C] and Wo [C, C] i.i.d. N(0, 1 / C) (unit-variance
    outputs); seeds [H, M, D] i.i.d. N(0, 1). Seed offset by 104729 from :func:`make_inputs`."""
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed) + 104729)
    B, H, N, M, D = w.B, w.H, w.N, w.M, w.D
    C = H * D
    dt = w.torch_dtype
    X = torch.randn(B, N, C, generator=gen, device=device).to(dt)
    W_in = (torch.randn(n_proj * C, C, generator=gen, device=device) / math.sqrt(C)).to(dt)
    Wo = (torch.randn(C, C, generator=gen, device=device) / math.sqrt(C)).to(dt)
    seeds = torch.randn(H, M, D, generator=gen, device=device).to(dt)
    return {"X": X, "W_in": W_in, "Wo": Wo, "seeds": seeds}


def to_f64_numpy(inputs):
    """The exact values of each input as float64 numpy arrays (bf16 and f32 upcast exactly)."""
    return {k: v.detach().to("cpu", torch.float64).numpy() for k, v in inputs.items()}
