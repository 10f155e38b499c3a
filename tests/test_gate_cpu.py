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
than the rounding does; the byte-exact pool comparisons catch those.)

The re-basing check (kvg_testlib.check_rotation_rounding) likewise accepts a
numpy model of the kernel's fp32 rotation and refuses planted mistakes:
rotation by -delta, frequencies off by one index, the other pairing, and
cos/sin rounded to bf16 (which the 2e-2 max-abs gate alone would pass)."""
import numpy as np
import pytest

from kvg_testlib import RNE_FLOOR, REL_TOL, check_rotation_rounding, compare_decode


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


def _fp32(x):
    return np.asarray(x, np.float64).astype(np.float32).astype(np.float64)


def _rotation_model(oracle, k_bits, delta, theta, style, sin_sign=1.0, freq_shift=0, trig_bf16=False):
    """numpy model of the kernel's re-basing of bf16 key rows: cos/sin of the
    fp64 angle delta * theta^(-2i/D) rounded to fp32, a' = fma(a, c, -(b s)),
    b' = fma(a, s, b c) in fp32, then bf16 RNE; pairs (i, i + D/2) for style
    0, (2i, 2i + 1) for style 1.  The keyword arguments plant mistakes."""
    x = oracle.bf16_to_f64(k_bits)
    d = x.shape[-1]
    half = d // 2
    ang = delta * theta ** (-2.0 * np.arange(half) / d)
    rnd = (lambda t: oracle.bf16_to_f64(oracle.bf16_rne(t))) if trig_bf16 else _fp32
    c, s = rnd(np.cos(ang)), rnd(np.sin(ang)) * sin_sign
    if freq_shift:
        c, s = np.roll(c, freq_shift), np.roll(s, freq_shift)
    a, b = (x[..., :half], x[..., half:]) if style == 0 else (x[..., 0::2], x[..., 1::2])
    ra = _fp32(a * c - _fp32(b * s))
    rb = _fp32(a * s + _fp32(b * c))
    out = np.empty_like(x)
    if style == 0:
        out[..., :half], out[..., half:] = ra, rb
    else:
        out[..., 0::2], out[..., 1::2] = ra, rb
    return oracle.bf16_rne(out)


@pytest.mark.parametrize("style", [0, 1])
@pytest.mark.parametrize("delta,theta", [(1, 1e6), (4096, 1e6), (100000, 1e4)])
def test_rotation_check_passes_fp32_rotation_and_refuses_planted_mistakes(oracle, style, delta, theta):
    """kvg_testlib.check_rotation_rounding (used on every re-based key the GPU
    writes) accepts a model of the kernel's fp32 arithmetic and refuses
    plausible mistakes, including ones the 2e-2 max-abs gate would pass
    (cos/sin rounded to bf16 instead of fp32)."""
    rng = np.random.default_rng(delta + style)
    k = oracle.bf16_rne(rng.standard_normal((512, 128)))
    ref = oracle.rope_rotate_rows(k, delta, theta, style)
    check_rotation_rounding(oracle, _rotation_model(oracle, k, delta, theta, style), ref)
    planted = {"rotation by -delta": dict(sin_sign=-1.0), "frequency index off by one": dict(freq_shift=1),
               "cos/sin rounded to bf16": dict(trig_bf16=True)}
    for what, kw in planted.items():
        bad = _rotation_model(oracle, k, delta, theta, style, **kw)
        with pytest.raises(AssertionError):
            check_rotation_rounding(oracle, bad, ref)
    bf = _rotation_model(oracle, k, delta, theta, style, trig_bf16=True)
    assert np.abs(oracle.bf16_to_f64(bf) - ref).max() <= 2e-2  # the coarse gate alone would pass it
    with pytest.raises(AssertionError):  # the other pairing
        check_rotation_rounding(oracle, _rotation_model(oracle, k, delta, theta, 1 - style), ref)


def test_max_abs_bound_allows_the_outputs_own_rounding_only(oracle):
    """The max-abs bound is 1e-2 beyond half a bf16 step of the reference:
    a correctly rounded output passes at any magnitude (|ref| ~ 5, where a
    bf16 step is 2^-5 and the rounding alone can exceed 1e-2), while an
    error of 0.015 on top of the rounding fails at |ref| ~ 0.5."""
    rng = np.random.default_rng(11)
    ref = 5.0 + rng.uniform(-0.9, 0.9, (4, 128))
    rounded = oracle.bf16_rne(ref)
    assert np.abs(oracle.bf16_to_f64(rounded) - ref).max() > 1e-2  # the rounding alone
    compare_decode(oracle, rounded, ref, what="correctly rounded, |ref| ~ 5")
    small = 0.5 + rng.uniform(-0.2, 0.2, (4, 128))
    off = small.copy()
    off[1, 7] += 0.015
    with pytest.raises(AssertionError, match="max-abs"):
        compare_decode(oracle, oracle.bf16_rne(off), small, rel=1.0, floor=0.0, what="0.015 off at |ref| ~ 0.5")
