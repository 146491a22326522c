"""Loader for the hand-worked 4x4-grid case in tests/golden/grid4x4_hand.json."""
import json
import os

import numpy as np

PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "grid4x4_hand.json")


def load():
    with open(PATH) as f:
        case = json.load(f)
    c = case["config"]
    C, N, D = c["n_cond"], c["n_image"], c["head_dim"]
    heads = []
    for hd in case["heads"]:
        q = np.zeros((N, D), dtype=np.float32)
        k = np.zeros((C + N, D), dtype=np.float32)
        for t, ent in hd["q"].items():
            for d, val in ent.items():
                q[int(t), int(d)] = val
        for j, ent in hd["k"].items():
            for d, val in ent.items():
                k[int(j), int(d)] = val
        v = np.zeros((C + N, D), dtype=np.float32)
        v[np.arange(C + N), np.arange(C + N) % D] = 1.0
        heads.append(dict(name=hd["name"], q=q, k=k, v=v, expected=hd["expected"]))
    return case, heads
