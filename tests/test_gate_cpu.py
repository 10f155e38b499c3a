"""The decode gate (kvg_testlib.compare_decode) can fail: mistakes planted on
the CPU, in fp64 attention computed by the oracle over altered rows (1% of
rows dropped, the last 16-row tile dropped, a tile read twice, the GQA
head mapping swapped, the scale applied twice), must be refused, while a
numpy model of the kernel's own roundings (softmax weights rounded to bf16
before the weighted sum of values, output rounded to bf16) must pass.  This
is where the gate's bounds come from (2^-7 relative, RNE-match floor 0.35),
checked at a 4,096-row and a 32,768-row context.  The partial-context
mistakes stay within the stated 1e-2 max-abs tolerance, which alone would
pass them.  (A single wrong row out of thousands moves the output by less
than the rounding does; the byte-exact pool comparisons catch those.)"""
import numpy as np
import pytest

from kvg_testlib import RNE_FLOOR, REL_TOL, compare_decode


def _rows(oracle, rng, n, hkv, d):
    bf = lambda x: oracle.bf16_rne(x)  # noqa: E731
    return bf(rng.standard_normal((n, hkv, d))), bf(rng.standard_normal((n, hkv, d)))


def _kernel_model(oracle, q, k, v, scale):
    """fp64 scores, weights exp(s - max) rounded to bf16, l summed over the
    rounded weights, o = sum(w v) / l rounded to bf16 (RNE) -> bits."""
    hq, d = q.shape
    g = hq // k.shape[1]
    qf, kf, vf = oracle.bf16_to_f64(q), oracle.bf16_to_f64(k), oracle.bf16_to_f64(v)
    out = np.zeros((hq, d))
    for h in range(hq):
        s = kf[:, h // g] @ qf[h] * scale
        p = oracle.bf16_to_f64(oracle.bf16_rne(np.exp(s - s.max())))
        out[h] = p @ vf[:, h // g] / p.sum()
    return oracle.bf16_rne(out)


@pytest.mark.parametrize("n", [4096, 32768])
def test_gate_passes_the_kernels_rounding_and_refuses_planted_mistakes(oracle, n):
    rng = np.random.default_rng(n)
    hkv, g, d = 2, 2, 128
    k, v = _rows(oracle, rng, n, hkv, d)
    q = oracle.bf16_rne(rng.standard_normal((hkv * g, d)))
    scale = 1.0 / np.sqrt(d)
    ref = oracle.gqa_decode(q, k, v, scale)
    # the kernel's roundings: within every bound
    err, rel, match = compare_decode(oracle, _kernel_model(oracle, q, k, v, scale), ref)
    assert rel <= REL_TOL / 1.5 and match >= RNE_FLOOR + 0.1
    bits = lambda o: oracle.bf16_rne(o)  # noqa: E731
    keep = np.ones(n, bool)
    keep[rng.choice(n, n // 100, replace=False)] = False
    planted = {
        # 1% of the rows never read
        "1% of rows dropped": oracle.gqa_decode(q, k[keep], v[keep], scale),
        # the last 16-row tile never read
        "last tile dropped": oracle.gqa_decode(q, k[:-16], v[:-16], scale),
        # one 16-row tile read twice (a page-table entry pointing at its neighbour)
        "a tile read twice": oracle.gqa_decode(q, np.concatenate([k, k[:16]]), np.concatenate([v, v[:16]]), scale),
        # query heads paired with the wrong KV head
        "GQA mapping swapped": oracle.gqa_decode(q[::-1].copy(), k, v, scale)[::-1],
        # the softmax scale applied twice
        "scale squared": oracle.gqa_decode(q, k, v, scale * scale),
    }
    blind = 0
    for name, o in planted.items():
        # max-abs <= 1e-2 alone lets the partial-context mistakes through
        blind += np.abs(oracle.bf16_to_f64(bits(o)) - ref).max() <= 1e-2
        with pytest.raises(AssertionError):
            compare_decode(oracle, bits(o), ref, what=name)
    assert blind >= 2
