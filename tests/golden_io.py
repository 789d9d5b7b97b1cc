"""Reader for the hand-derived fixtures in tests/golden/."""
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def read_worked_example(name="worked_repair.txt"):
    head, cases, cur = {"keys": []}, [], None
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if not line:
                continue
            tok = line.split()
            key, vals = tok[0], tok[1:]
            if key == "case":
                cur = {"name": vals[0]}
                cases.append(cur)
                continue
            target = cur if cur is not None else head
            if key == "key":
                head["keys"].append([float(v) for v in vals])
            elif key in ("N", "d", "window", "n_sink", "n_recent"):
                target[key] = int(vals[0])
            elif key in ("tau",):
                target[key] = float(vals[0])
            elif key in ("b_all", "b_ret"):
                target[key] = np.array([float(v) for v in vals])
            else:
                target[key] = np.array([int(v) for v in vals], dtype=np.int64)
    head["keys"] = np.array(head["keys"], dtype=np.float32)
    return head, cases
