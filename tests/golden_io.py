"""Reader for tests/golden/*.txt hand-worked fixtures."""
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _ranges(tokens):
    out = []
    for t in tokens:
        if "-" in t:
            a, b = t.split("-")
            out.extend(range(int(a), int(b) + 1))
        else:
            out.append(int(t))
    return out


def map_cases(name="map_small.txt"):
    cases, cur = [], None
    with open(os.path.join(GOLDEN, name)) as f:
        for raw in f:
            line = raw.split("#", 1)[0].strip()
            if not line:
                continue
            key, _, rest = line.partition(" ")
            if key == "case":
                cur = {"name": rest.strip(), "kept": []}
            elif key == "geometry":
                cur["geometry"] = {k: int(v) for k, v in (kv.split("=") for kv in rest.split())}
            elif key == "ctx":
                cur["ctx"] = [int(x) for x in rest.split()]
            elif key == "M":
                cur["M"] = [int(x) for x in rest.replace("|", " ").split()]
            elif key == "kept":
                cur["kept"].append(_ranges(rest.split()))
            elif key == "end":
                g = cur["geometry"]
                cur["M"] = np.array(cur["M"], np.uint8).reshape(g["L"], g["H"], g["D"])
                cases.append(cur)
                cur = None
    return cases
