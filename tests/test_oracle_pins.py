"""Pins for the CPU oracle: each check ties an oracle function to something
other than itself (hashlib, torch's fp32->bf16 cast, textbook closed forms,
numpy's softmax, exact invariants), chosen so that a dropped term, a wrong
sign, a wrong pairing index or a transposed operand fails at least one."""
import hashlib
import math
import struct

import numpy as np
import pytest
import torch

import kvg_synth as syn

# --------------------------------------------------------------------------
# SHA-256 (FIPS 180-4) and the two-level page digest
# --------------------------------------------------------------------------

NIST_MESSAGES = [
    b"",
    b"abc",
    b"abcdbcdecdefdefgefghfghighijhijkijkljklmklmnlmnomnopnopq",
    b"abcdefghbcdefghicdefghijdefghijkefghijklfghijklmghijklmnhijklmnoijklmnopjklmnopqklmnopqrlmnopqrs"
    b"mnopqrstnopqrstu",
    b"a" * 1_000_000,
]


@pytest.mark.parametrize("msg", NIST_MESSAGES, ids=["empty", "abc", "448bit", "896bit", "million_a"])
def test_sha256_standard_messages(oracle, msg):
    assert oracle.sha256(msg) == hashlib.sha256(msg).digest()


def test_sha256_every_padding_boundary(oracle):
    rng = np.random.default_rng(1)
    data = rng.integers(0, 256, 400, dtype=np.uint8).tobytes()
    for n in range(0, 300):
        assert oracle.sha256(data[:n]) == hashlib.sha256(data[:n]).digest(), n


def test_sha256_constants_first_primes(oracle):
    # K[0] and H0[0] follow from sqrt(2) and cbrt(2) alone (FIPS 180-4 4.2.2, 5.3.3):
    # floor(frac(2^(1/3)) * 2^32) and floor(frac(2^(1/2)) * 2^32), here from
    # python's exact integer roots.
    k, h = oracle.sha256_constants()
    assert int(h[0]) == math.isqrt(2 << 64) & 0xFFFFFFFF
    root = int(round((2 << 96) ** (1.0 / 3.0)))
    while root ** 3 > (2 << 96):
        root -= 1
    while (root + 1) ** 3 <= (2 << 96):
        root += 1
    assert int(k[0]) == root & 0xFFFFFFFF


def _two_level_hashlib(page: bytes, leaf: int = 4096) -> bytes:
    cat = b"".join(hashlib.sha256(page[i:i + leaf]).digest() for i in range(0, len(page), leaf))
    return hashlib.sha256(cat).digest()


@pytest.mark.parametrize("size", [4096, 262144, 10000, 4097, 64, 8192])
def test_page_digest_two_level(oracle, size):
    rng = np.random.default_rng(size)
    page = rng.integers(0, 256, size, dtype=np.uint8)
    assert oracle.page_digest(page) == _two_level_hashlib(page.tobytes())


def test_page_digest_detects_flip_and_leaf_swap(oracle):
    rng = np.random.default_rng(7)
    page = rng.integers(0, 256, 4 * 4096, dtype=np.uint8)
    d0 = oracle.page_digest(page)
    flipped = page.copy()
    flipped[12345] ^= 1
    assert oracle.page_digest(flipped) != d0
    swapped = page.reshape(4, 4096)[[1, 0, 2, 3]].reshape(-1)
    assert oracle.page_digest(swapped) != d0
    # one leaf: the page digest is the hash of the leaf's digest
    leaf = page[:4096]
    assert oracle.page_digest(leaf) == hashlib.sha256(hashlib.sha256(leaf.tobytes()).digest()).digest()


def test_page_digests_batch(oracle):
    rng = np.random.default_rng(3)
    pages = rng.integers(0, 256, (5, 8192), dtype=np.uint8)
    got = oracle.page_digests(pages, 8192)
    for i in range(5):
        assert got[i].tobytes() == _two_level_hashlib(pages[i].tobytes())


# --------------------------------------------------------------------------
# bf16 rounding
# --------------------------------------------------------------------------

def _finite_bf16_patterns():
    b = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    exp = (b >> 7) & 0xFF
    return b[exp != 0xFF]


def test_bf16_exact_values_roundtrip(oracle):
    b = _finite_bf16_patterns()
    assert np.array_equal(oracle.bf16_rne(oracle.bf16_to_f64(b)), b)


def test_bf16_ties_to_even_and_nearest(oracle):
    b = _finite_bf16_patterns()
    pos = np.sort(b[(b >> 15) == 0].astype(np.int64))
    pos = pos[pos < 0x7F7F]  # adjacent finite pairs (x, next)
    lo = oracle.bf16_to_f64(pos.astype(np.uint16))
    hi = oracle.bf16_to_f64((pos + 1).astype(np.uint16))
    mid = (lo + hi) / 2  # exact in fp64
    r = oracle.bf16_rne(mid).astype(np.int64)
    even = np.where(pos % 2 == 0, pos, pos + 1)
    assert np.array_equal(r, even)
    gap = hi - lo
    assert np.array_equal(oracle.bf16_rne(mid - gap / 8).astype(np.int64), pos)
    assert np.array_equal(oracle.bf16_rne(mid + gap / 8).astype(np.int64), pos + 1)
    # negative values mirror positive ones
    assert np.array_equal(oracle.bf16_rne(-mid).astype(np.int64), even | 0x8000)


def test_bf16_matches_torch_fp32_cast(oracle):
    g = torch.Generator().manual_seed(5)
    x = torch.randn(200000, generator=g) * torch.exp(torch.randn(200000, generator=g) * 8)
    ref = x.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = oracle.bf16_rne(x.double().numpy())
    assert np.array_equal(got, ref)


# --------------------------------------------------------------------------
# RoPE rotation by an offset
# --------------------------------------------------------------------------

def _bf16(a):
    return syn.as_u16(torch.tensor(np.asarray(a, np.float32)).to(torch.bfloat16))


def test_rope_zero_offset_is_identity(oracle):
    x = syn.as_u16(syn.normal_bf16((16, 128), 1))
    y = oracle.rope_rotate_rows(x, 0, 1e6, 0)
    assert np.array_equal(y, oracle.bf16_to_f64(x))
    assert np.array_equal(oracle.rope_rotate_rows_bf16(x, 0, 1e6, 0), x)


def test_rope_d2_is_plane_rotation(oracle):
    # D = 2: w_0 = theta^0 = 1, so the pair rotates by delta radians.
    x = _bf16([1.0, 0.5])
    for delta in [1.0, -3.0, 0.25 * math.pi * 4]:
        y = oracle.rope_rotate_rows(x, delta, 10000.0, 0)
        c, s = math.cos(delta), math.sin(delta)
        assert y[0] == pytest.approx(1.0 * c - 0.5 * s, abs=1e-15)
        assert y[1] == pytest.approx(1.0 * s + 0.5 * c, abs=1e-15)


def test_rope_pairing_and_frequency(oracle):
    D, theta, delta = 8, 10000.0, 7.0
    for style, partner in [(0, lambda i: i + D // 2), (1, lambda i: i ^ 1)]:
        for i in range(D // 2):
            a = i if style == 0 else 2 * i
            e = np.zeros(D, np.float32)
            e[a] = 1.0
            y = oracle.rope_rotate_rows(_bf16(e), delta, theta, style)
            ang = delta * theta ** (-2.0 * i / D)
            b = partner(a)
            expect = np.zeros(D)
            expect[a] = math.cos(ang)
            expect[b] = math.sin(ang)
            np.testing.assert_allclose(y, expect, atol=1e-15)


def test_rope_matches_complex_multiplication(oracle):
    D, theta = 128, 1e6
    x = syn.as_u16(syn.normal_bf16((4, D), 2))
    xf = oracle.bf16_to_f64(x)
    for delta in [1, 4096, 100000, -77]:
        y = oracle.rope_rotate_rows(x, delta, theta, 0)
        i = np.arange(D // 2)
        z = (xf[:, :D // 2] + 1j * xf[:, D // 2:]) * np.exp(1j * delta * np.power(theta, -2.0 * i / D))
        np.testing.assert_allclose(y[:, :D // 2], z.real, atol=1e-12)
        np.testing.assert_allclose(y[:, D // 2:], z.imag, atol=1e-12)


@pytest.mark.parametrize("style", [0, 1])
def test_rope_composition_and_inverse(oracle, style):
    D, theta = 256, 10000.0
    x = oracle.bf16_to_f64(syn.as_u16(syn.normal_bf16((8, D), 3)))
    for a, b in [(1, 4096), (4096, 100000), (-5, 5), (123, -7000)]:
        ab = oracle.rope_rotate_rows_f64(oracle.rope_rotate_rows_f64(x, b, theta, style), a, theta, style)
        direct = oracle.rope_rotate_rows_f64(x, a + b, theta, style)
        np.testing.assert_allclose(ab, direct, atol=1e-9, rtol=0)
    back = oracle.rope_rotate_rows_f64(oracle.rope_rotate_rows_f64(x, 4096, theta, style), -4096,
                                       theta, style)
    np.testing.assert_allclose(back, x, atol=1e-12)
    y = oracle.rope_rotate_rows_f64(x, 100000, theta, style)
    np.testing.assert_allclose(np.linalg.norm(y, axis=1), np.linalg.norm(x, axis=1), rtol=1e-13)


def test_rope_scores_depend_on_relative_position_only(oracle):
    # Sec. 4.2: in exact arithmetic attention depends only on relative position.
    D, theta = 128, 1e6
    q = syn.as_u16(syn.normal_bf16((1, D), 4))
    k = syn.as_u16(syn.normal_bf16((16, D), 5))
    s0 = oracle.bf16_to_f64(k) @ oracle.bf16_to_f64(q)[0]
    for delta in [1, 4096, 100000]:
        qr = oracle.rope_rotate_rows(q, delta, theta, 0)
        kr = oracle.rope_rotate_rows(k, delta, theta, 0)
        np.testing.assert_allclose(kr @ qr[0], s0, atol=1e-10)


# --------------------------------------------------------------------------
# Decode attention (fp64)
# --------------------------------------------------------------------------

def test_attention_single_token_returns_its_value(oracle):
    q = syn.as_u16(syn.normal_bf16((64,), 6))
    k = syn.as_u16(syn.normal_bf16((1, 64), 7))
    v = syn.as_u16(syn.normal_bf16((1, 64), 8))
    o = oracle.attention_head(q, k, v, 0.125)
    assert np.array_equal(o, oracle.bf16_to_f64(v[0]))


def test_attention_two_tokens_closed_form(oracle):
    D = 64
    q = np.zeros(D, np.float32); q[0] = 2.0
    k = np.zeros((2, D), np.float32); k[0, 0] = 1.0; k[1, 0] = -0.5
    v = np.zeros((2, D), np.float32); v[0, :] = 1.0; v[1, :] = -3.0; v[1, 5] = 8.0
    scale = 0.5
    o = oracle.attention_head(_bf16(q), _bf16(k), _bf16(v), scale)
    s0, s1 = 2.0 * 1.0 * scale, 2.0 * -0.5 * scale
    w0, w1 = math.exp(s0), math.exp(s1)
    expect = (w0 * v[0].astype(np.float64) + w1 * v[1].astype(np.float64)) / (w0 + w1)
    np.testing.assert_allclose(o, expect, rtol=1e-14)
    # equal scores -> plain mean
    k2 = np.zeros((2, D), np.float32)
    o2 = oracle.attention_head(_bf16(q), _bf16(k2), _bf16(v), scale)
    np.testing.assert_allclose(o2, (v[0] + v[1]) / 2.0, rtol=1e-15)


def test_attention_equal_values_and_one_hot(oracle):
    D, n = 64, 50
    q = syn.as_u16(syn.normal_bf16((D,), 9))
    k = syn.as_u16(syn.normal_bf16((n, D), 10))
    row = syn.as_u16(syn.normal_bf16((D,), 11))
    v = np.tile(row, (n, 1))
    o = oracle.attention_head(q, k, v, 0.125)
    np.testing.assert_allclose(o, oracle.bf16_to_f64(row), rtol=1e-14)
    # one dominant score -> that token's value
    qq = np.zeros(D, np.float32); qq[0] = 100.0
    kk = np.zeros((n, D), np.float32); kk[17, 0] = 1.0
    vv = syn.as_u16(syn.normal_bf16((n, D), 12))
    o = oracle.attention_head(_bf16(qq), _bf16(kk), vv, 1.0)
    np.testing.assert_allclose(o, oracle.bf16_to_f64(vv[17]), atol=1e-40)


def test_attention_matches_numpy_softmax(oracle):
    Hq, Hkv, D, n = 8, 2, 128, 300
    q = syn.as_u16(syn.normal_bf16((Hq, D), 13))
    k = syn.as_u16(syn.normal_bf16((n, Hkv, D), 14))
    v = syn.as_u16(syn.normal_bf16((n, Hkv, D), 15))
    scale = 1 / math.sqrt(D)
    o = oracle.gqa_decode(q, k, v, scale)
    qf, kf, vf = (oracle.bf16_to_f64(a) for a in (q, k, v))
    G = Hq // Hkv
    for h in range(Hq):
        s = kf[:, h // G, :] @ qf[h] * scale
        p = np.exp(s - s.max())
        p /= p.sum()
        np.testing.assert_allclose(o[h], p @ vf[:, h // G, :], rtol=1e-11, atol=1e-14)


def test_attention_gqa_head_mapping(oracle):
    Hq, Hkv, D, n = 8, 4, 64, 10
    q = syn.as_u16(syn.normal_bf16((Hq, D), 16))
    k = syn.as_u16(syn.normal_bf16((n, Hkv, D), 17))
    v = np.zeros((n, Hkv, D), np.float32)
    for g in range(Hkv):
        v[:, g, :] = g + 1
    o = oracle.gqa_decode(q, k, _bf16(v), 0.1)
    for h in range(Hq):
        np.testing.assert_allclose(o[h], np.full(D, h // 2 + 1.0), rtol=1e-15)


def test_attention_empty_context_is_zero(oracle):
    q = syn.as_u16(syn.normal_bf16((4, 64), 18))
    z = np.zeros((0, 2, 64), np.uint16)
    assert np.array_equal(oracle.gqa_decode(q, z, z, 0.1), np.zeros((4, 64)))


# --------------------------------------------------------------------------
# Block store and paged cache
# --------------------------------------------------------------------------

def _dims(w=syn.TINY):
    import oracle as o
    return o.Dims(w.n_layers, w.n_kv_heads, w.head_dim, w.page_size, w.rope_theta, 0)


def _kv(n, seed, w=syn.TINY):
    k, v = syn.kv_rows(w, n, seed)
    return syn.as_u16(k), syn.as_u16(v)


CANARY = 0x7FBF  # a bf16 NaN pattern: never produced by the method


def test_block_pages_digests_and_serialization(oracle):
    d = _dims()
    n = 250  # ragged: 15 full pages + 10 rows
    k, v = _kv(n, 1)
    blk = oracle.block_from_kv(d, k, v, syn.positions(0, n))
    assert blk.n_pages == 16
    # token t lives in page t // P, row t % P; padding rows are zero
    assert np.array_equal(blk.pages[1, 0, 3, 1, 5], k[1, 3 * 16 + 5, 1])
    assert np.array_equal(blk.pages[0, 1, 15, 0, 9], v[0, 249, 0])
    assert not blk.pages[:, :, 15, :, 10:, :].any()
    for l in range(d.L):
        for kv in range(2):
            for j in range(blk.n_pages):
                assert blk.digests[l, kv, j].tobytes() == _two_level_hashlib(blk.pages[l, kv, j].tobytes())
    ser = blk.serialize()
    f = struct.unpack_from("<8sIIiiiiqqdiiQQQQ", ser, 0)
    assert f[0] == b"KVGBLK01" and f[3:7] == (2, 2, 64, 16) and f[7] == n and f[8] == 16
    pos_off, dig_off, pages_off, total = f[12:16]
    assert total == len(ser) and pages_off % 4096 == 0 and dig_off % 256 == 0
    assert np.array_equal(np.frombuffer(ser, "<i4", n, pos_off), np.arange(n))
    assert ser[dig_off:dig_off + blk.digests.size] == blk.digests.tobytes()
    assert ser[pages_off:] == blk.pages.tobytes()
    assert ser[96:128] == hashlib.sha256(np.arange(n, dtype="<i4").tobytes() + blk.digests.tobytes()).digest()


def test_own_position_graft_is_identity_on_bytes(oracle):
    d = _dims()
    n = 256
    k, v = _kv(n, 2)
    blk = oracle.block_from_kv(d, k, v, syn.positions(0, n))
    c = oracle.OracleCache(d, n_pages=40, max_seqs=3, max_slots=512, fill=CANARY)
    before = c.pool.copy()
    c.graft(1, blk)
    kk, vv, pp = c.logical_kv(1, 0)
    assert np.array_equal(kk, k[0]) and np.array_equal(vv, v[0]) and np.array_equal(pp, np.arange(n))
    kk, vv, _ = c.logical_kv(1, 1)
    assert np.array_equal(kk, k[1]) and np.array_equal(vv, v[1])
    assert list(c.page_table[1, :16]) == list(range(16)) and (c.page_table[1, 16:] == -1).all()
    assert (c.page_fill[1, :16] == 16).all() and c.n_slots[1] == n
    # pages not handed out keep their canary bytes
    assert np.array_equal(c.pool[:, :, 16:], before[:, :, 16:])
    # restored pages equal the deposited pages byte for byte
    assert np.array_equal(c.pool[:, :, :16], blk.pages)


def test_graft_equals_fresh_write_under_permuted_pages(oracle):
    d = _dims()
    nb, nf = 100, 60  # ragged block, then fresh tokens on top
    k, v = _kv(nb + nf, 3)
    q = syn.as_u16(syn.queries(syn.TINY, 2, 1, 3))[:, 0]
    fresh = oracle.OracleCache(d, 32, 2, 256, fill=CANARY)
    fresh.set_free_order(syn.permutation(32, 9))
    fresh.append(0, k[:, :nb], v[:, :nb], syn.positions(0, nb))
    blk = fresh.deposit(0, 0, nb)
    fresh.append(0, k[:, nb:], v[:, nb:], syn.positions(nb, nf))
    grafted = oracle.OracleCache(d, 32, 2, 256, fill=CANARY)
    grafted.graft(1, blk)
    # the block's last page is partially filled; the fresh rows follow at the next page
    assert grafted.n_slots[1] == nb
    grafted.append(1, k[:, nb:], v[:, nb:], syn.positions(nb, nf))
    for l in range(2):
        a = fresh.logical_kv(0, l)
        b = grafted.logical_kv(1, l)
        for x, y in zip(a, b):
            assert np.array_equal(x, y)
        oa = fresh.decode(0, l, q[l], 0.125)
        ob = grafted.decode(1, l, q[l], 0.125)
        assert oa.tobytes() == ob.tobytes()
    # and equal to attention over the plain logical rows
    ref = oracle.gqa_decode(q[0], k[0], v[0], 0.125)
    assert ref.tobytes() == fresh.decode(0, 0, q[0], 0.125).tobytes()


def test_deposit_equals_block_from_rows(oracle):
    d = _dims()
    n = 77
    k, v = _kv(n, 4)
    c = oracle.OracleCache(d, 16, 1, 256, fill=CANARY)
    c.set_free_order(syn.permutation(16, 2))
    c.append(0, k, v, syn.positions(5, n))
    b1 = c.deposit(0, 0, n)
    b2 = oracle.block_from_kv(d, k, v, syn.positions(5, n))
    assert b1.serialize() == b2.serialize()


def test_relocated_graft(oracle):
    w = syn.TINY
    d = _dims()
    n = 40
    k, v = _kv(n, 5)
    blk = oracle.block_from_kv(d, k, v, syn.positions(0, n))
    own = oracle.OracleCache(d, 8, 1, 128)
    own.graft(0, blk)
    zero = oracle.OracleCache(d, 8, 1, 128)
    zero.graft(0, blk, delta=0)
    assert np.array_equal(own.pool, zero.pool)
    for delta in [1, 4096, 100000]:
        c = oracle.OracleCache(d, 8, 1, 128)
        c.graft(0, blk, delta=delta)
        for l in range(d.L):
            kk, vv, pp = c.logical_kv(0, l)
            assert np.array_equal(pp, np.arange(n) + delta)
            assert np.array_equal(vv, v[l])
            assert np.array_equal(kk, oracle.rope_rotate_rows_bf16(k[l], delta, w.rope_theta, 0))
        # padding rows of the last page stay zero (not rotated)
        assert not c.pool[:, 0, 2, :, 8:, :].any()


def test_relocated_attention_is_delta_invariant_in_fp64(oracle):
    # keys re-based by delta and the query rotated by the same delta keep the
    # relative geometry: the fp64 output moves only at the rounding level.
    w = syn.TINY
    n, D = 64, w.head_dim
    k, v = _kv(n, 6)
    q = syn.as_u16(syn.queries(w, 1, 1, 6))[0, 0]
    base = oracle.gqa_decode(q, k[0], v[0], 1 / math.sqrt(D))
    for delta in [1, 4096, 100000]:
        kr = oracle.rope_rotate_rows(k[0], delta, w.rope_theta, 0)
        qr = oracle.rope_rotate_rows(q, delta, w.rope_theta, 0)
        G = w.group
        for h in range(w.n_q_heads):
            s = kr[:, h // G, :] @ qr[h] / math.sqrt(D)
            p = np.exp(s - s.max()); p /= p.sum()
            np.testing.assert_allclose(p @ oracle.bf16_to_f64(v[0][:, h // G, :]), base[h], atol=1e-12)


def test_cache_errors_and_release(oracle):
    d = _dims()
    k, v = _kv(40, 7)
    blk = oracle.block_from_kv(d, k, v, syn.positions(0, 40))
    c = oracle.OracleCache(d, 4, 2, 64)
    with pytest.raises(oracle.KvgError):
        c.graft(0, blk, dst_slot=16)  # not the next page boundary
    c.graft(0, blk)
    with pytest.raises(oracle.KvgError):
        c.graft(1, blk)  # only one free page left
    with pytest.raises(oracle.KvgError):
        c.append(0, k[:, :30], v[:, :30], syn.positions(40, 30))  # past max_slots
    c.release(0)
    assert c.free == [3, 0, 1, 2]
    with pytest.raises(oracle.KvgError):
        c.graft(1, oracle.block_from_kv(d, k, v, syn.positions(2**31 - 10, 40)))


def test_pinned_block_graft_aliases_pages(oracle):
    d = _dims()
    n = 40  # 2 full pages + 8 rows
    k, v = _kv(n, 8)
    c = oracle.OracleCache(d, 12, 3, 64, fill=CANARY)
    c.append(0, k, v, syn.positions(0, n))
    pb = c.pin_block(0, 0, n)
    assert pb.pids == [3, 4, 5]  # taken after the sequence's own pages 0..2
    c.release(0)
    assert c.free == [6, 7, 8, 9, 10, 11, 0, 1, 2]  # pinned pages never return
    c.graft_pinned(1, pb)
    c.graft_pinned(2, pb)
    assert list(c.page_table[1, :2]) == list(c.page_table[2, :2]) == [3, 4]  # shared
    assert c.page_table[1, 2] == 6 and c.page_table[2, 2] == 7            # ragged page copied
    for sq in (1, 2):
        kk, vv, pp = c.logical_kv(sq, 1)
        assert np.array_equal(kk, k[1]) and np.array_equal(vv, v[1]) and np.array_equal(pp, np.arange(n))
    c.append(1, k[:, :3], v[:, :3], syn.positions(n, 3))
    assert np.array_equal(c.pool[:, :, 5], pb.block.pages[:, :, 2])  # the block's own page untouched
    c.release(1)
    assert 3 not in c.free and 6 in c.free


# --------------------------------------------------------------------------
# Sliding-window layers over a full-size cache (Sec. 4.3)
# --------------------------------------------------------------------------

def _stitched(oracle, seed):
    """Seq 0: a ragged 37-row block grafted, then 20 fresh rows appended on
    its partly filled last page, then a 21-row block grafted at the next page
    boundary (a hole of unfilled rows before it), then 5 fresh rows.
    Returns the cache and the rows written, in order, per layer."""
    d = _dims()
    c = oracle.OracleCache(d, 40, 2, 256, fill=CANARY)
    c.set_free_order(syn.permutation(40, seed))
    ka, va = _kv(37, seed)
    kb, vb = _kv(20, seed + 1)
    kc, vc = _kv(21, seed + 2)
    kd, vd = _kv(5, seed + 3)
    c.graft(0, oracle.block_from_kv(d, ka, va, syn.positions(0, 37)))
    c.append(0, kb, vb, syn.positions(37, 20))
    c.graft(0, oracle.block_from_kv(d, kc, vc, syn.positions(57, 21)))
    c.append(0, kd, vd, syn.positions(78, 5))
    k = np.concatenate([ka, kb, kc, kd], axis=1)
    v = np.concatenate([va, vb, vc, vd], axis=1)
    return c, k, v


@pytest.mark.parametrize("W", [1, 5, 16, 17, 40, 83, 500])
def test_window_attends_to_the_last_w_rows_written(oracle, W):
    c, k, v = _stitched(oracle, 21)
    q = syn.as_u16(syn.queries(syn.TINY, 2, 1, 22))[:, 0]
    c.set_layer_windows([W, 0])
    n = k.shape[1]  # 83 rows written; the hole is not among them
    assert n == 83
    got = c.decode(0, 0, q[0], 0.125)
    want = oracle.gqa_decode(q[0], k[0, -W:], v[0, -W:], 0.125)
    assert got.tobytes() == want.tobytes()
    # the other layer stays global
    assert c.decode(0, 1, q[1], 0.125).tobytes() == oracle.gqa_decode(q[1], k[1], v[1], 0.125).tobytes()
    if W >= n:
        c.set_layer_windows([])
        assert c.decode(0, 0, q[0], 0.125).tobytes() == got.tobytes()


def test_window_of_one_returns_the_last_value_row(oracle):
    c, k, v = _stitched(oracle, 23)
    c.set_layer_windows([1, 1])
    q = syn.as_u16(syn.queries(syn.TINY, 2, 1, 24))[:, 0]
    for l in range(2):
        o = c.decode(0, l, q[l], 0.125)
        G = q.shape[1] // v.shape[2]
        for h in range(q.shape[1]):
            assert np.array_equal(o[h], oracle.bf16_to_f64(v[l, -1, h // G]))


# Split decode over a slot range: the rows written, by construction of the
# stitched sequence, sit at slots 0..56 (rows 0..56) and 64..89 (rows 57..82).
def _rows_of_slots(lo, hi):
    slots = list(range(0, 57)) + list(range(64, 90))
    return [i for i, s in enumerate(slots) if lo <= s < hi]


@pytest.mark.parametrize("lo,hi,W", [(0, 1 << 20, 0), (0, 64, 0), (64, 1 << 20, 0), (48, 64, 0), (16, 16, 0),
                                     (64, 80, 0), (0, 64, 30), (64, 1 << 20, 30), (0, 32, 30)])
def test_decode_range_reads_the_rows_in_its_slots(oracle, lo, hi, W):
    c, k, v = _stitched(oracle, 27)
    q = syn.as_u16(syn.queries(syn.TINY, 2, 1, 28))[:, 0]
    c.set_layer_windows([W, 0])
    rows = _rows_of_slots(lo, hi)
    if W:
        rows = [r for r in rows if r >= 83 - W]
    for l in range(2):
        rr = rows if l == 0 else _rows_of_slots(lo, hi)
        got = c.decode_range(0, l, q[l], 0.125, lo, hi)
        want = oracle.gqa_decode(q[l], k[l, rr], v[l, rr], 0.125)
        assert got.tobytes() == want.tobytes()
        if not rr:
            assert not got.any()
    if (lo, hi) == (0, 1 << 20):
        assert c.decode_range(0, 0, q[0], 0.125, lo, hi).tobytes() == c.decode(0, 0, q[0], 0.125).tobytes()


def test_window_settings_are_checked(oracle):
    c, _, _ = _stitched(oracle, 25)
    with pytest.raises(oracle.KvgError):
        c.set_layer_windows([1])
    with pytest.raises(oracle.KvgError):
        c.set_layer_windows([-1, 0])


# --------------------------------------------------------------------------
# Quantized KV: fp8 E4M3 codes with per-tensor scales
# --------------------------------------------------------------------------

def test_e4m3_code_values_match_torch(oracle):
    codes = np.arange(256, dtype=np.uint8)
    ours = oracle.e4m3_to_f64(codes)
    ref = torch.from_numpy(codes.copy()).view(torch.float8_e4m3fn).to(torch.float64).numpy()
    nan = np.isnan(ref)
    assert (np.isnan(ours) == nan).all() and nan.sum() == 2  # 0x7F, 0xFF
    assert np.array_equal(ours[~nan], ref[~nan])
    assert ours[0x7E] == 448.0 and ours[0x01] == 2.0 ** -9 and ours[0x08] == 2.0 ** -6


def test_e4m3_rounding_matches_torch_on_every_bf16_in_range(oracle):
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    x = oracle.bf16_to_f64(bits)
    keep = np.isfinite(x) & (np.abs(x) <= 448.0)
    x = x[keep]
    ours = oracle.e4m3_rne(x)
    ref = torch.from_numpy(x.astype(np.float32)).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    assert np.array_equal(ours, ref)


def test_e4m3_saturates_and_keeps_nan(oracle):
    got = oracle.e4m3_rne(np.array([448.0, 449.0, 464.0, 1e6, -1e6, -500.0, np.nan, 0.0, -0.0]))
    assert list(got) == [0x7E, 0x7E, 0x7E, 0x7E, 0xFE, 0xFE, 0x7F, 0x00, 0x80]


@pytest.mark.parametrize("scale", [0.0625, 0.037, 3.3])
def test_e4m3_quantize_multiplies_by_the_fp32_reciprocal(oracle, scale):
    rng = np.random.default_rng(7)
    x = syn.as_u16(torch.from_numpy(rng.standard_normal(20000).astype(np.float32) * 4).to(torch.bfloat16))
    q = oracle.e4m3_quantize(x, scale)
    xf = torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).float()
    r = torch.tensor(1.0, dtype=torch.float32) / torch.tensor(scale, dtype=torch.float32)
    y = xf * r
    ok = (y.abs() <= 448).numpy()
    ref = y.to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    assert np.array_equal(q[ok], ref[ok])
    assert (q[~ok] & 0x7F == 0x7E).all()


def _fp8_dims(scale_k=0.125, scale_v=0.25):
    import oracle as o
    w = syn.TINY
    return o.Dims(w.n_layers, w.n_kv_heads, w.head_dim, w.page_size, w.rope_theta, 0, o.KV_E4M3, scale_k, scale_v)


def test_fp8_block_layout_and_header(oracle):
    d = _fp8_dims()
    n = 40
    k, v = _kv(n, 31)
    blk = oracle.block_from_kv(d, k, v, syn.positions(0, n))
    assert blk.pages.dtype == np.uint8 and d.page_bytes == d.page_elems
    assert np.array_equal(blk.pages[1, 0, 2, 1, 3], oracle.e4m3_quantize(k[1, 2 * 16 + 3, 1], 0.125))
    assert np.array_equal(blk.pages[0, 1, 0, 0, 5], oracle.e4m3_quantize(v[0, 5, 0], 0.25))
    ser = blk.serialize()
    f = struct.unpack_from("<8sIIiiiiqqdiiQQQQ", ser, 0)
    assert f[11] == 2 and struct.unpack_from("<ff", ser, 128) == (0.125, 0.25)
    assert len(ser) - f[14] == blk.pages.size  # one byte per element
    for l in range(d.L):
        for kv in range(2):
            for j in range(blk.n_pages):
                assert blk.digests[l, kv, j].tobytes() == _two_level_hashlib(blk.pages[l, kv, j].tobytes())


def test_fp8_decode_equals_bf16_decode_over_the_dequantized_rows(oracle):
    """With power-of-two scales every dequantized element is exactly a bf16
    value, so the fp8 cache's attention must equal the bf16 cache's attention
    over those values, in fp64, bit for bit."""
    import oracle as o
    d8 = _fp8_dims(0.125, 0.5)
    w = syn.TINY
    d16 = o.Dims(w.n_layers, w.n_kv_heads, w.head_dim, w.page_size, w.rope_theta, 0)
    n = 70
    k, v = _kv(n, 33)
    c8 = o.OracleCache(d8, 12, 1, 128)
    c8.append(0, k, v, syn.positions(0, n))
    kq = oracle.bf16_rne(oracle.e4m3_dequant(oracle.e4m3_quantize(k, 0.125), 0.125))
    vq = oracle.bf16_rne(oracle.e4m3_dequant(oracle.e4m3_quantize(v, 0.5), 0.5))
    assert np.array_equal(oracle.bf16_to_f64(kq), oracle.e4m3_dequant(oracle.e4m3_quantize(k, 0.125), 0.125))
    c16 = o.OracleCache(d16, 12, 1, 128)
    c16.append(0, kq, vq, syn.positions(0, n))
    q = syn.as_u16(syn.queries(w, 2, 1, 34))[:, 0]
    for l in range(2):
        assert c8.decode(0, l, q[l], 0.125).tobytes() == c16.decode(0, l, q[l], 0.125).tobytes()
    with pytest.raises(o.KvgError):
        c8.graft(0, c8.deposit(0, 0, 32), delta=5)
