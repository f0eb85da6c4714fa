"""Reader for tests/golden/hand_cases.txt (hand-worked products)."""
import os

import numpy as np
import torch

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "hand_cases.txt")


def _bf16_bits(rows):
    t = torch.tensor(rows, dtype=torch.float64).to(torch.float32)
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def load():
    cases, cur, section = [], None, None
    for raw in open(GOLDEN):
        line = raw.split("#", 1)[0].strip()
        if not line:
            continue
        tok = line.split()
        if tok[0] == "case":
            cur = dict(name=tok[1], dtype=tok[2], M=int(tok[3]), N=int(tok[4]), K=int(tok[5]),
                       layout=int(tok[6]), A=[], B=[], C=[], MAG=[], RNE=[])
            cases.append(cur)
            continue
        if tok[0] in ("A", "B", "C", "MAG", "RNE"):
            section = tok[0]
            continue
        if section == "RNE":
            cur[section].append([int(x, 16) for x in tok])
        else:
            cur[section].append([float(x) for x in tok])
    out = []
    for c in cases:
        M, N, K, lay = c["M"], c["N"], c["K"], c["layout"]
        bshape = (K, N) if lay == 0 else (N, K)
        if c["dtype"] == "int8":
            A = np.array(c["A"], dtype=np.int8).reshape(M, K)
            B = np.array(c["B"], dtype=np.int8).reshape(bshape)
        else:
            A = _bf16_bits(c["A"]).reshape(M, K)
            B = _bf16_bits(c["B"]).reshape(bshape)
        c["A"], c["B"] = A, B
        c["C"] = np.array(c["C"], dtype=np.float64).reshape(M, N)
        if c["MAG"]:
            c["MAG"] = np.array(c["MAG"], dtype=np.float64).reshape(M, N)
            c["RNE"] = np.array(c["RNE"], dtype=np.uint16).reshape(M, N)
        out.append(c)
    return out
