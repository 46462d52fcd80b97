"""Parsers for the hand-written fixtures under tests/golden/."""
import os

import numpy as np

from workloads.manifests import Manifest

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _lines(name):
    with open(os.path.join(GOLDEN, name)) as f:
        for raw in f:
            line = raw.split("#", 1)[0].strip()
            if line:
                yield line.split()


def rne_cases():
    """[(fp32 bits, expected bf16 bits)] from rne_cases.txt."""
    return [(int(t[0], 16), int(t[1], 16)) for t in _lines("rne_cases.txt")]


def f16_cases():
    """[(direction, input bits, expected bits)] from f16_cases.txt."""
    return [(t[0], int(t[1], 16), int(t[2], 16)) for t in _lines("f16_cases.txt")]


def manifest_case(name):
    """(Manifest, blob uint8 array, {dst: expected bytes}, expected checksums)."""
    blob, dsts, entries, exp_dst, exp_ck, blob_bytes = None, [], [], {}, None, None
    for t in _lines(name):
        key = t[0]
        if key == "blob_bytes":
            blob_bytes = int(t[1])
        elif key == "blob":
            blob = np.array([int(x, 16) for x in t[1:]], dtype=np.uint8)
        elif key == "dst":
            dsts.append({"name": t[1], "dtype": t[2],
                         "shape": tuple(int(x) for x in t[3].split(","))})
        elif key == "entry":
            entries.append({"name": t[1], "dtype": t[2],
                            "shape": tuple(int(x) for x in t[3].split(",")),
                            "offset": int(t[4]), "dst": int(t[5]), "row": int(t[6]),
                            "cast": bool(int(t[7])), "cksum": True, "layer": 0,
                            "stride": int(t[8]) if len(t) > 8 else 0})
        elif key == "expect_dst":
            exp_dst[int(t[1])] = np.array([int(x, 16) for x in t[2:]], dtype=np.uint8)
        elif key == "expect_cksum":
            exp_ck = np.array([int(x) for x in t[1:]], dtype=np.uint64)
        else:
            raise ValueError(f"{name}: unknown key {key}")
    assert blob is not None and blob.size == blob_bytes
    m = Manifest(name, entries, dsts, blob_bytes, "bits", 0)
    return m, blob, exp_dst, exp_ck
