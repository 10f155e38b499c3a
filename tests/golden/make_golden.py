"""Writes tests/golden/tiny_ragged_case.json from the CPU oracle alone.

The paper prints no worked example for the graft, the page digest or the
decode step, so this fixture holds the oracle's own results for one small,
ragged case.  Its inputs come from an integer-only generator (SplitMix64), so
the file does not depend on a library's random numbers.  Re-running this
script must reproduce the file byte for byte.  A change to it goes in a
commit that names the passage of the paper (or the reading of it) that
changed the oracle's arithmetic.

Case (the Tiny geometry: 2 layers, 4 query / 2 KV heads, head_dim 64, page 16):
a 40-token block at positions 0..39 (two full pages and a half page),
deposited, grafted at its own positions into an empty sequence, followed by
13 fresh rows at positions 40..52 that fill the tail page and start another,
then one decode query per layer over the 53 rows (scale 1/8).
"""
from __future__ import annotations

import json
import math
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import kvg_synth as syn  # noqa: E402
import oracle  # noqa: E402

OUT = os.path.join(HERE, "tiny_ragged_case.json")
L, HQ, HKV, D, P, THETA = 2, 4, 2, 64, 16, 10000.0
N_BLOCK, N_FRESH = 40, 13
SEED_K, SEED_V, SEED_Q = 0x6B31, 0x7631, 0x7131


def inputs():
    """k, v [L][53][Hkv][D] and q [L][Hq][D], bf16 bit patterns."""
    n = N_BLOCK + N_FRESH
    k = syn.portable_bf16((L, n, HKV, D), SEED_K)
    v = syn.portable_bf16((L, n, HKV, D), SEED_V)
    q = syn.portable_bf16((L, HQ, D), SEED_Q)
    return k, v, q


def compute() -> dict:
    k, v, q = inputs()
    dims = oracle.Dims(L, HKV, D, P, THETA, 0)
    pos = np.arange(N_BLOCK + N_FRESH, dtype=np.int32)
    src = oracle.OracleCache(dims, 8, 1, 64)
    src.append(0, k[:, :N_BLOCK], v[:, :N_BLOCK], pos[:N_BLOCK])
    blk = src.deposit(0, 0, N_BLOCK)
    dst = oracle.OracleCache(dims, 8, 1, 64)
    dst.graft(0, blk)
    dst.append(0, np.ascontiguousarray(k[:, N_BLOCK:]), np.ascontiguousarray(v[:, N_BLOCK:]), pos[N_BLOCK:])
    scale = 1.0 / math.sqrt(D)
    o = np.stack([dst.decode(0, l, q[l], scale) for l in range(L)])
    return {
        "block_sha256": oracle.sha256(blk.serialize()).hex(),
        "block_digest": blk.block_digest.hex(),
        "page_digests": [blk.digests[l, kv, j].tobytes().hex()
                         for l in range(L) for kv in range(2) for j in range(blk.n_pages)],
        "page_table": [int(x) for x in dst.page_table[0, :4]],
        "page_fill": [int(x) for x in dst.page_fill[0, :4]],
        "decode_f64": [[[float("%.12e" % x) for x in o[l, h]] for h in range(HQ)] for l in range(L)],
        "decode_bf16_rne": [[oracle.bf16_rne(o[l, h]).astype("<u2").tobytes().hex() for h in range(HQ)]
                            for l in range(L)],
    }


def main():
    case = {"what": "oracle results for the tiny ragged graft case (see make_golden.py)",
            "geometry": {"n_layers": L, "n_q_heads": HQ, "n_kv_heads": HKV, "head_dim": D, "page_size": P,
                         "rope_theta": THETA, "block_tokens": N_BLOCK, "fresh_tokens": N_FRESH,
                         "seeds": [SEED_K, SEED_V, SEED_Q]},
            **compute()}
    with open(OUT, "w") as f:
        json.dump(case, f, indent=1)
        f.write("\n")
    print(f"wrote {OUT}")


if __name__ == "__main__":
    main()
