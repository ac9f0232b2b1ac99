"""Writes closed_forms.json: tiny Gauss sums whose values follow in closed
form from the definition of Phi_tau and Eq. 1 (Sec. 1 of arXiv 2609.04910).
Each expected value is the closed form evaluated with ``math.exp``; no
library code is involved.  Run from the repository root:
    python tests/golden/make_closed_forms.py
"""
import json
import math
import os

cases = [
    {
        "cite": "Sec. 1, Phi_tau(q,k) = exp(-tau/2 ||q-k||^2): D=1, q=0, k=1, tau=2 gives exp(-1)",
        "q": [[0.0]], "k": [[1.0]], "v": [[1.0]], "tau": 2.0,
        "formula": "exp(-1)",
        "s": [[math.exp(-1.0)]],
    },
    {
        "cite": "Eq. 1 with three keys: squared distances 1, 4, 25 from q=(0,0), tau=1",
        "q": [[0.0, 0.0]], "k": [[1.0, 0.0], [0.0, 2.0], [3.0, 4.0]],
        "v": [[1.0], [-2.0], [0.5]], "tau": 1.0,
        "formula": "exp(-1/2) - 2 exp(-2) + 0.5 exp(-25/2)",
        "s": [[math.exp(-0.5) - 2.0 * math.exp(-2.0) + 0.5 * math.exp(-12.5)]],
    },
    {
        "cite": "Eq. 1, C=2 channels: a coincident point gives Phi=1, a point at squared distance 2 gives exp(-1) at tau=1",
        "q": [[1.0, 1.0], [0.0, 0.0]], "k": [[1.0, 1.0]], "v": [[2.0, -3.0]], "tau": 1.0,
        "formula": "[[2, -3], [2 exp(-1), -3 exp(-1)]]",
        "s": [[2.0, -3.0], [2.0 * math.exp(-1.0), -3.0 * math.exp(-1.0)]],
    },
    {
        "cite": "Eq. 1, signed weights cancelling exactly: two keys symmetric about q",
        "q": [[0.5, 0.0, 0.0]], "k": [[0.0, 0.0, 0.0], [1.0, 0.0, 0.0]], "v": [[1.0], [-1.0]],
        "tau": 3.0, "formula": "exp(-3/8) - exp(-3/8) = 0",
        "s": [[0.0]],
    },
]

with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "closed_forms.json"), "w") as f:
    json.dump(cases, f, indent=1)
    f.write("\n")
