"""Write oracle_regression.json: the fp64 oracle's output on one tiny seeded
case.  Calls only oracle/; run from the repository root:

    python tests/golden/make_golden.py
"""
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)
from oracle import ecokv_oracle as O  # noqa: E402


def case():
    r = np.random.RandomState(20260)
    n, d, w, hkv, g = 24, 8, 3, 2, 2
    u = r.standard_normal((hkv, d))
    u /= np.linalg.norm(u, axis=1, keepdims=True)
    s = np.exp(0.5 * r.standard_normal((hkv, n)))
    K = s[..., None] * (4 * u[:, None, :] + r.standard_normal((hkv, n, d)))
    V = r.standard_normal((hkv, n, d))
    Q = 4 * np.repeat(u, g, axis=0)[:, None, :] + r.standard_normal((hkv * g, w, d))
    p = O.Params(n_layers=1, h_kv=hkv, h_q=hkv * g, n=n, d=d, window=w, budget=9, pool_kernel=3)
    return K[None], V[None], Q[None], p


def main():
    K, V, Q, p = case()
    res = O.evict(K, V, Q, p)
    out = {"params": p.__dict__, "units": {}}
    for (l, h), r in res.items():
        out["units"][f"{l},{h}"] = {k: (np.asarray(r[k]).tolist()) for k in
                                    ("S", "idx", "lam", "r_E", "r_C", "D_E", "s_imp", "d_e", "c")}
    with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "oracle_regression.json"), "w") as f:
        json.dump(out, f, indent=1)


if __name__ == "__main__":
    main()
