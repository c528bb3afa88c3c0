"""Write tests/golden/route_small.json (a small routing-chain case and the oracle's answer)
and tests/golden/route_bwd_small.json (the oracle's gradients of that case for a stored dY).

The inputs are drawn here with numpy (seed 2608) and stored in full; the expected Q, Z
and Y come only from the float64 oracle (Sec. 3.2, eqs. flarepp_dynamic_query and
flarepp_mixer), whose pins live in tests/test_oracle_pins.py. The file is a regression
fixture for the oracle and a fixed parity case for the CUDA path.

Run from the repository root:  python tests/golden/make_golden.py
"""
import json
import math
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)
import oracle  # noqa: E402


def main():
    rng = np.random.default_rng(2608)
    B, H, N, M, D = 1, 2, 40, 6, 16
    s = 1.0 / math.sqrt(D)
    # values rounded to multiples of 2^-8 so that they are exact in float32 (not in bf16,
    # whose 8 significant bits do not hold 2^-8 steps above 1): the GPU cases run in float32
    r = lambda *sh: np.round(rng.standard_normal(sh) * 256.0) / 256.0
    seeds, Kt, Vt, K, V = r(H, M, D), r(B, H, N, D) * 2.0, r(B, H, N, D), r(B, H, N, D) * 2.0, r(B, H, N, D)
    Q, Z, Y = oracle.route(seeds, Kt, Vt, K, V, s)
    doc = {
        "what": "FLARE++ routing chain Q=SDPA(seeds,Kt,Vt), Z=SDPA(Q,K,V), Y=SDPA(K,Q,Z) "
                "(Sec. 3.2, eqs. flarepp_dynamic_query, flarepp_mixer); expected values from the "
                "float64 oracle",
        "shape": {"B": B, "H": H, "N": N, "M": M, "D": D}, "scale": s,
        "inputs": {k: v.tolist() for k, v in
                   dict(seeds=seeds, Kt=Kt, Vt=Vt, K=K, V=V).items()},
        "expected": {"Q": Q.tolist(), "Z": Z.tolist(), "Y": Y.tolist()},
    }
    here = os.path.dirname(os.path.abspath(__file__))
    out = os.path.join(here, "route_small.json")
    with open(out, "w") as f:
        json.dump(doc, f, indent=None, separators=(",", ":"))
        f.write("\n")
    print(out)

    # the backward of the same case for an output gradient dY (drawn after the inputs, so
    # the forward case above does not change)
    dY = r(B, H, N, D)
    grads = oracle.route_bwd(seeds, Kt, Vt, K, V, s, dY)
    doc = {
        "what": "gradients of the routing chain of route_small.json (same inputs and scale) for "
                "the output gradient dY (App. A.5); expected values from the float64 oracle",
        "dY": dY.tolist(),
        "expected": {k: g.tolist() for k, g in
                     zip(("dseeds", "dKt", "dVt", "dK", "dV"), grads)},
    }
    out = os.path.join(here, "route_bwd_small.json")
    with open(out, "w") as f:
        json.dump(doc, f, indent=None, separators=(",", ":"))
        f.write("\n")
    print(out)


if __name__ == "__main__":
    main()
