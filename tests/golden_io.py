"""Reader for the small text fixtures under tests/golden/ ("key: v v ; v v")."""
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def load(name):
    out = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, val = line.split(":", 1)
            rows = [r.split() for r in val.split(";")]
            arr = np.array([[float(v) for v in r] for r in rows])
            out[key.strip()] = arr[0] if arr.shape[0] == 1 else arr
    return out
