"""Reader for the hand-worked block fixtures under tests/golden/."""
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _num(tok: str) -> float:
    tok = tok.strip()
    if "0x" in tok.lower() and "p" in tok.lower():
        return float.fromhex(tok)
    return float(tok)


def read_blocks(fname: str, default_code: int):
    blocks = []
    cur = None
    with open(os.path.join(GOLDEN, fname)) as fh:
        for line in fh:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, _, val = line.partition(":")
            key = key.strip()
            if key == "name":
                cur = {"name": val.strip()}
                blocks.append(cur)
            elif key == "w":
                w = np.zeros(32, dtype=np.float32)
                vals = [_num(t) for t in val.split()]
                w[:len(vals)] = np.array(vals, dtype=np.float32)
                # keep the sign of literal negative zeros
                cur["w"] = w
            elif key == "scale":
                cur["scale"] = int(val.strip(), 16)
            elif key == "codes":
                c = np.full(32, default_code, dtype=np.int64)
                vals = [int(t) for t in val.split()]
                c[:len(vals)] = vals
                cur["codes"] = c
            elif key in ("bytes", "low", "high"):
                cur[key] = np.array([int(t, 16) for t in val.split()], dtype=np.uint8)
            else:
                raise ValueError(f"unknown key {key!r} in {fname}")
    return blocks
