"""Reader for the small text fixtures in this folder (paper worked examples)."""
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))


def load(name: str) -> dict:
    out = {}
    with open(os.path.join(HERE, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if not line:
                continue
            key, *vals = line.split()
            out[key] = vals
    unit = int(out.pop("unit_ns")[0])
    R, S = int(out.pop("R")[0]), int(out.pop("S")[0])
    res = {"unit_ns": unit, "R": R, "S": S}
    res["d"] = np.array([int(v) for v in out.pop("d")], dtype=np.int64).reshape(1, R, S) * unit
    for k, v in out.items():
        if k == "labels":
            res[k] = v
        else:
            res[k] = np.array([int(x) for x in v], dtype=np.int64)
    return res
