"""Writes tests/golden/oracle_vectors.json using only the oracle package.

The paper prints no worked example for this path (no digest, no GEMV output),
so these stored values are the oracle's own, frozen: they catch a drift in the
oracle between machines (x86 here, Arm beside the GPU) or across edits.  Every
input is a closed-form byte pattern, reproducible without any generator.
Run:  python tests/golden/make_golden.py
"""
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)
import oracle  # noqa: E402


def patterns():
    """name -> bytes, all closed forms."""
    return {
        "empty": b"",
        "zero_1": b"\0",
        "ramp_256": bytes(range(256)),
        "ramp_4096": bytes(i % 251 for i in range(4096)),
        "ramp_4097": bytes(i % 251 for i in range(4097)),
        "ramp_3leaves_17": bytes((7 * i + 3) % 256 for i in range(3 * 4096 + 17)),
    }


def gemv_case():
    """Integer bf16 W [5, 8] and x [8], exact in every precision."""
    W = [[(3 * i + 5 * j) % 7 - 3 for j in range(8)] for i in range(5)]
    x = [(j % 3) - 1 for j in range(8)]
    return W, x


def bf16_bytes(vals):
    out = bytearray()
    for v in vals:
        f = np.float32(v).view(np.uint32)
        out += int(f >> 16).to_bytes(2, "little")
    return bytes(out)


def main():
    d = {"digests": {}, "gemv": {}}
    for k, b in patterns().items():
        d["digests"][k] = {"n": len(b), "plain": "%016x" % oracle.fnv1a64(b),
                           "tree": "%016x" % oracle.fnv_tree(b)}
    W, x = gemv_case()
    yhat, a = oracle.gemv(np.frombuffer(bf16_bytes(sum(W, [])), np.uint8), 1, 5, 8,
                          np.frombuffer(bf16_bytes(x), np.uint8))
    d["gemv"] = {"W": W, "x": x, "yhat": list(map(float, yhat)), "a": list(map(float, a))}
    with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "oracle_vectors.json"), "w") as f:
        json.dump(d, f, indent=1)
        f.write("\n")


if __name__ == "__main__":
    main()
