"""Writes tests/golden/oracle_small.json: a small seeded problem (inputs stored
in full) and the fp64 oracle's outputs for it.

The paper prints no worked numeric example for the output stage, so this
fixture pins the oracle against accidental change only; its independence from
the oracle's own code comes from the pins in tests/test_oracle.py.  It calls
nothing but the oracle.  Regenerate with:  python tests/golden/make_golden.py
"""
import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))
from oracle import oracle as orc  # noqa: E402


def main():
    rng = np.random.default_rng(2608)
    T, d, V = 8, (8, 16, 24), 40
    H = [rng.standard_normal((T, dm)).astype(np.float32) for dm in d]
    W = [(0.4 * rng.standard_normal((V, dm))).astype(np.float32) for dm in d]
    y = rng.integers(0, V, T).astype(np.int32)
    y[5] = -1
    kw = dict(teacher=2, tau=0.8, alpha=0.3, w=[1.0, 0.5, 2.0])
    f = orc.forward(H, W, y, **kw)
    dH, dW = orc.backward(H, W, y, grad_scale=1.0, **kw)
    fix = {
        "what": "fp64 oracle outputs for a small seeded 3-sub-model problem (Eq. 2, Eq. 3)",
        "T": T, "d": list(d), "V": V, **kw,
        "H": [h.tolist() for h in H], "W": [x.tolist() for x in W], "y": y.tolist(),
        "loss": f["loss"], "tok_loss": f["tok_loss"].tolist(), "ce": f["ce"].tolist(),
        "ld": f["ld"].tolist(), "kl": f["kl"].tolist(), "argmax": f["argmax"].tolist(),
        "lse": f["lse"].tolist(), "lse_tau": f["lse_tau"].tolist(),
        "dH": [x.tolist() for x in dH], "dW": [x.tolist() for x in dW],
    }
    with open(os.path.join(HERE, "oracle_small.json"), "w") as fh:
        json.dump(fix, fh)


if __name__ == "__main__":
    main()
