"""Pins for the CPU oracle: checks against what the paper and the mathematics fix.

Each ``pin_*`` takes a loaded oracle library and raises ``AssertionError`` on a mismatch.
They avoid re-typing the oracle's own formulas: TopK is checked by rank counting and by
numpy's stable argsort, the error-feedback updates by their conservation identities,
quantisation by inputs whose codes are known in closed form, bit layouts by numpy's
``unpackbits``, and the generator by its published outputs.  ``test_oracle_pins.py``
runs them on the oracle; ``test_oracle_mutants.py`` runs them on deliberately broken
copies of the oracle to show that each plausible mistake is caught.
"""

from __future__ import annotations

import os

import numpy as np

import oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def bits_of(a: np.ndarray) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)


def brute_topk(row: np.ndarray, k: int):
    """Kept set by rank counting: j is kept iff fewer than k entries beat it, where i
    beats j when |x_i| > |x_j|, or |x_i| == |x_j| and i < j (§2.3, lower index first)."""
    a = np.abs(row.astype(np.float64))
    n = row.shape[0]
    i = np.arange(n)
    beats = (a[:, None] > a[None, :]) | ((a[:, None] == a[None, :]) & (i[:, None] < i[None, :]))
    rank = beats.sum(axis=0)
    kept = np.nonzero(rank < k)[0]
    return kept


# --------------------------------------------------------------------------------------
# generator
# --------------------------------------------------------------------------------------

def pin_splitmix64_published(lib):
    rows = []
    with open(os.path.join(GOLDEN, "splitmix64_seed0.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                c, v = line.split()
                rows.append((int(c), int(v, 16)))
    assert len(rows) == 3
    for c, v in rows:
        got = oracle.splitmix64(0, c, lib)
        assert got == v, (c, hex(got), hex(v))
    # u for even flat index uses the low half, odd index the high half of the same word
    z0 = rows[0][1]
    assert oracle.uniform(0, 0, lib) == float((z0 & 0xFFFFFFFF) >> 8) * 2.0 ** -24
    assert oracle.uniform(0, 1, lib) == float((z0 >> 32) >> 8) * 2.0 ** -24
    z1 = rows[1][1]
    assert oracle.uniform(0, 2, lib) == float((z1 & 0xFFFFFFFF) >> 8) * 2.0 ** -24
    assert oracle.uniform(0, 3, lib) == float((z1 >> 32) >> 8) * 2.0 ** -24


def pin_uniform_range(lib):
    us = np.array([oracle.uniform(12345, i, lib) for i in range(4096)])
    assert us.min() >= 0.0 and us.max() < 1.0
    assert np.all(us * 2 ** 24 == np.floor(us * 2 ** 24))
    assert abs(us.mean() - 0.5) < 0.03


# --------------------------------------------------------------------------------------
# TopK, §2.3
# --------------------------------------------------------------------------------------

def pin_topk_hand(lib):
    x = np.array([[3.0, -5.0, 1.0, 5.0, 0.0]], np.float32)
    expect = {1: ([1], [-5.0]), 2: ([1, 3], [-5.0, 5.0]), 3: ([0, 1, 3], [3.0, -5.0, 5.0]),
              4: ([0, 1, 2, 3], [3.0, -5.0, 1.0, 5.0]), 5: ([0, 1, 2, 3, 4], list(x[0]))}
    for k, (idx, vals) in expect.items():
        v, i = oracle.topk_compress(x, k, lib)
        assert i[0].tolist() == idx, (k, i)
        assert np.array_equal(bits_of(v[0]), bits_of(np.array(vals, np.float32))), (k, v)


def pin_topk_bruteforce(lib, n_rows: int = 10000, seed: int = 1):
    rng = np.random.default_rng(seed)
    for t in range(n_rows):
        L = int(rng.integers(1, 65))
        kind = t % 4
        if kind == 0:
            row = rng.standard_normal(L).astype(np.float32)
        elif kind == 1:  # many exact ties, both signs, signed zeros
            row = rng.integers(-3, 4, L).astype(np.float32)
            row[rng.random(L) < 0.2] = -0.0
        elif kind == 2:  # ReLU-like: about half exact zeros
            row = np.maximum(rng.standard_normal(L), 0).astype(np.float32)
        else:
            row = (rng.standard_normal(L) * 10.0 ** rng.integers(-30, 30)).astype(np.float32)
        k = int(rng.integers(1, L + 1))
        v, i = oracle.topk_compress(row[None, :], k, lib)
        kept = brute_topk(row, k)
        assert i[0].tolist() == kept.tolist(), (t, row, k, i, kept)
        assert np.array_equal(bits_of(v[0]), bits_of(row[kept]))


def pin_topk_argsort(lib, seed: int = 2):
    """Stable argsort of -|x| ranks equal magnitudes by lower index: a library routine
    that gives the same kept set."""
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((64, 1000)).astype(np.float32)
    x[:, ::7] = np.round(x[:, ::7])  # plant ties
    for k in (1, 10, 100, 999, 1000):
        v, i = oracle.topk_compress(x, k, lib)
        for r in range(x.shape[0]):
            order = np.argsort(-np.abs(x[r].astype(np.float64)), kind="stable")[:k]
            assert i[r].tolist() == np.sort(order).tolist()
            assert np.array_equal(bits_of(v[r]), bits_of(x[r, np.sort(order)]))


def pin_topk_invariants(lib, seed: int = 3):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((16, 4097)).astype(np.float32)
    for k in (1, 409, 4096, 4097):
        v, i = oracle.topk_compress(x, k, lib)
        for r in range(16):
            assert np.all(np.diff(i[r]) > 0)
            kept = np.zeros(4097, bool)
            kept[i[r]] = True
            assert kept.sum() == k
            if k < 4097:
                assert np.abs(x[r, kept]).min() >= np.abs(x[r, ~kept]).max()


def pin_topk_decompress(lib, seed: int = 4):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((8, 333)).astype(np.float32)
    x[0, :5] = -0.0
    # K = 100 %: the round trip is the identity, bit for bit
    v, i = oracle.topk_compress(x, 333, lib)
    y = oracle.topk_decompress(v, i, 333, lib)
    assert np.array_equal(bits_of(y), bits_of(x))
    v, i = oracle.topk_compress(x, 33, lib)
    y = oracle.topk_decompress(v, i, 333, lib)
    for r in range(8):
        kept = np.zeros(333, bool)
        kept[i[r]] = True
        assert np.array_equal(bits_of(y[r, kept]), bits_of(x[r, kept]))
        assert np.all(bits_of(y[r, ~kept]) == 0)  # +0 everywhere else


def pin_topk_gather(lib, seed: int = 14):
    """Index reuse (§3.2, Table 5): numpy's take_along_axis gives the values at the kept
    indices; at a tensor's own TopK indices the gather is its TopK payload; gathering,
    scattering back and gathering again changes nothing."""
    rng = np.random.default_rng(seed)
    a = rng.standard_normal((6, 257)).astype(np.float32)
    g = rng.standard_normal((6, 257)).astype(np.float32)
    g[1, 3] = -0.0
    for k in (1, 25, 128, 257):
        _, idx = oracle.topk_compress(a, k, lib)
        v = oracle.topk_gather(g, idx, lib)
        assert np.array_equal(bits_of(v), bits_of(np.take_along_axis(g, idx, axis=1)))
        own_v, own_i = oracle.topk_compress(g, k, lib)
        assert np.array_equal(bits_of(oracle.topk_gather(g, own_i, lib)), bits_of(own_v))
        y = oracle.topk_decompress(v, idx, 257, lib)
        assert np.array_equal(bits_of(oracle.topk_gather(y, idx, lib)), bits_of(v))


# --------------------------------------------------------------------------------------
# Error feedback, §2.4
# --------------------------------------------------------------------------------------

def pin_ef_identity(lib, seed: int = 5):
    rng = np.random.default_rng(seed)
    R, L, k = 12, 500, 37
    e = (rng.standard_normal((R, L)) * 0.3).astype(np.float32)
    x = rng.standard_normal((R, L)).astype(np.float32)
    s = x + e  # float32 add
    e1 = e.copy()
    v, i = oracle.ef_topk_compress(x, e1, k, lib)
    c = np.zeros((R, L), np.float32)
    for r in range(R):
        c[r, i[r]] = v[r]
        kept = brute_topk(s[r], k)
        assert i[r].tolist() == kept.tolist()  # the message is TopK of x + e
    assert np.array_equal(c + e1, s)  # s == C(s) + e' exactly
    for r in range(R):
        assert np.all(bits_of(e1[r, i[r]]) == 0)  # nothing left behind where sent
        mask = np.ones(L, bool)
        mask[i[r]] = False
        assert np.array_equal(bits_of(e1[r, mask]), bits_of(s[r, mask]))


def pin_ef_conservation(lib, seed: int = 6):
    """Over T steps, everything that went in either was sent or is still in the buffer:
    sum(sent) + e_T == sum(x_t) + e_0, up to fp32 addition error."""
    rng = np.random.default_rng(seed)
    R, L, k, T = 4, 256, 13, 30
    e = np.zeros((R, L), np.float32)
    e0 = e.astype(np.float64)
    sent = np.zeros((R, L))
    xin = np.zeros((R, L))
    for t in range(T):
        x = rng.standard_normal((R, L)).astype(np.float32)
        xin += x
        v, i = oracle.ef_topk_compress(x, e, k, lib)
        for r in range(R):
            sent[r, i[r]] += v[r]
    lhs = sent + e
    rhs = xin + e0
    assert np.linalg.norm(lhs - rhs) <= 1e-6 * np.linalg.norm(rhs)


def pin_efmix_bruteforce(lib, n_rows: int = 3000, seed: int = 15):
    """EF-mixed (§2.4) on tiny rows, every k: the input's ceil(k/2) by rank counting on
    |x|, the buffer's floor(k/2) by rank counting on |e| over the rest; x + e sent there
    in index order; the buffer keeps x + e elsewhere and +0 where sent; and the sent
    message plus the new buffer is x + e exactly."""
    rng = np.random.default_rng(seed)
    for t in range(n_rows):
        L = int(rng.integers(1, 24))
        x = rng.standard_normal(L).astype(np.float32)
        e = rng.standard_normal(L).astype(np.float32)
        if t % 5 == 0:
            x[rng.integers(0, L, L // 2)] = 0.5  # ties in |x|
        if t % 7 == 0:
            e[:] = 0.0  # the first step: an empty buffer
        k = int(rng.integers(1, L + 1))
        k1, k2 = k - k // 2, k // 2
        s = x + e
        first = set(brute_topk(x, k1).tolist())
        rest = np.array(sorted(set(range(L)) - first), dtype=np.int64)
        second = set(rest[brute_topk(e[rest], k2)].tolist()) if k2 else set()
        want = np.array(sorted(first | second), dtype=np.int64)
        e2 = e.copy()[None, :]
        v, i = oracle.efmix_topk_compress(x[None, :], e2, k, lib)
        assert np.array_equal(i[0], want), (t, i[0], want)
        assert np.array_equal(bits_of(v[0]), bits_of(s[want]))
        keep = np.ones(L, bool)
        keep[want] = False
        assert np.array_equal(bits_of(e2[0][keep]), bits_of(s[keep]))
        assert np.all(bits_of(e2[0][~keep]) == 0)
        y = oracle.topk_decompress(v, i, L, lib)
        assert np.array_equal(bits_of(y[0] + e2[0]), bits_of(s + np.float32(0)))


def pin_ef21_update(lib, seed: int = 7):
    rng = np.random.default_rng(seed)
    R, L, k = 10, 768, 76
    g = (rng.standard_normal((R, L))).astype(np.float32)
    x = (g + 0.05 * rng.standard_normal((R, L))).astype(np.float32)
    d = x - g
    g1 = g.copy()
    v, i = oracle.ef21_topk_compress(x, g1, k, lib)
    for r in range(R):
        kept = brute_topk(d[r], k)
        assert i[r].tolist() == kept.tolist()  # message is C(x - g)
        assert np.array_equal(bits_of(v[r]), bits_of(d[r, kept]))
    c = np.zeros((R, L), np.float32)
    for r in range(R):
        c[r, i[r]] = v[r]
    assert np.array_equal(bits_of(g1), bits_of(g + c))  # g' = g + C(x - g)


def pin_ef21_first_step(lib, seed: int = 8):
    """With g_0 = 0 the first EF21 message is plain TopK of x."""
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((6, 300)).astype(np.float32)
    g = np.zeros_like(x)
    v, i = oracle.ef21_topk_compress(x, g, 30, lib)
    v2, i2 = oracle.topk_compress(x, 30, lib)
    assert np.array_equal(i, i2) and np.array_equal(bits_of(v), bits_of(v2))


def pin_aqsgd(lib, seed: int = 9):
    rng = np.random.default_rng(seed)
    S, rps, L, k = 20, 3, 128, 38
    buf = rng.standard_normal((S, rps, L)).astype(np.float32)
    ids = rng.permutation(S)[:5].astype(np.int64)
    x = (buf[ids] + 0.05 * rng.standard_normal((5, rps, L))).astype(np.float32)
    before = buf.copy()
    b2 = buf.copy()
    v, i = oracle.aqsgd_compress(x, b2, ids, k, lib)
    # buffer after update == buffer before + decompressed delta, bitwise
    for n, sid in enumerate(ids):
        for r in range(rps):
            row = n * rps + r
            d = x[n, r] - before[sid, r]
            kept = brute_topk(d, k)
            assert i[row].tolist() == kept.tolist()
            c = np.zeros(L, np.float32)
            c[kept] = d[kept]
            assert np.array_equal(bits_of(b2[sid, r]), bits_of(before[sid, r] + c))
    untouched = np.setdiff1d(np.arange(S), ids)
    assert np.array_equal(bits_of(b2[untouched]), bits_of(before[untouched]))
    # the receiver's copy takes the same update
    recv = before.copy()
    oracle.aqsgd_decompress(v, i, recv, ids, lib)
    assert np.array_equal(bits_of(recv), bits_of(b2))
    # EF21 is AQ-SGD with the identity sample map
    g = before[ids].reshape(5 * rps, L).copy()
    v3, i3 = oracle.ef21_topk_compress(x.reshape(5 * rps, L), g, k, lib)
    assert np.array_equal(i3, i) and np.array_equal(bits_of(v3), bits_of(v))
    assert np.array_equal(bits_of(g), bits_of(b2[ids].reshape(5 * rps, L)))


# --------------------------------------------------------------------------------------
# Quantisation, §2.2
# --------------------------------------------------------------------------------------

def stream_codes(codes_row: np.ndarray, bits: int, n: int) -> np.ndarray:
    """Read n codes of width ``bits`` from an LSB-first bitstream with numpy."""
    b = np.unpackbits(codes_row.astype("<u4").view(np.uint8), bitorder="little")
    b = b[: n * bits].reshape(n, bits).astype(np.int64)
    return (b << np.arange(bits)).sum(axis=1)


def pin_quant_hand(lib):
    # integer grid: min 0, max 3, scale 1 -> codes are the values themselves
    c, s, m = oracle.quant_compress(np.array([[0.0, 1.0, 2.0, 3.0]], np.float32), 2, lib=lib)
    assert s[0] == 1.0 and m[0] == 0.0
    assert c[0, 0] == (0 | 1 << 2 | 2 << 4 | 3 << 6) and np.all(c[0, 1:] == 0)
    y = oracle.quant_decompress(c, s, m, 4, 2, lib)
    assert np.array_equal(y[0], [0.0, 1.0, 2.0, 3.0])
    # a half-way value rounds to the even code
    c, s, m = oracle.quant_compress(np.array([[0.0, 1.5, 3.0, 0.5, 2.5]], np.float32), 2, lib=lib)
    assert stream_codes(c[0], 2, 5).tolist() == [0, 2, 3, 0, 2]
    # shifted and scaled grid: min -2, step 0.5 at 3 bits (all exactly representable)
    x = np.array([[-2.0, 1.5, -0.5, 0.0, 1.0, -1.5]], np.float32)
    c, s, m = oracle.quant_compress(x, 3, lib=lib)
    assert s[0] == 0.5 and m[0] == -2.0
    assert stream_codes(c[0], 3, 6).tolist() == [0, 7, 3, 4, 6, 1]
    assert np.array_equal(oracle.quant_decompress(c, s, m, 6, 3, lib), x)


def pin_quant_degenerate(lib):
    x = np.full((1, 10), 2.5, np.float32)
    c, s, m = oracle.quant_compress(x, 4, lib=lib)
    assert np.all(c == 0) and s[0] == 0.0 and m[0] == 2.5
    assert np.array_equal(oracle.quant_decompress(c, s, m, 10, 4, lib), x)
    # +0 and -0 compare equal; the minimum is -0 (total order), the range is zero
    x = np.array([[0.0, -0.0, 0.0]], np.float32)
    c, s, m = oracle.quant_compress(x, 8, lib=lib)
    assert bits_of(m)[0] == 0x80000000 and s[0] == 0.0 and np.all(c == 0)


def pin_quant_grid_bitstream(lib, seed: int = 10):
    """Inputs on the integer grid 0..2^b-1 (with both ends present) give scale 1,
    min 0 and codes equal to the inputs, for every width, straddling words or not."""
    rng = np.random.default_rng(seed)
    for bits in (1, 2, 3, 4, 5, 6, 7, 8, 11, 12, 16):
        for L in (1, 2, 31, 32, 33, 100, 257):
            top = (1 << bits) - 1
            q = rng.integers(0, top + 1, L)
            q[0] = 0
            if L > 1:
                q[-1] = top
            x = q.astype(np.float32)[None, :]
            c, s, m = oracle.quant_compress(x, bits, lib=lib)
            W = oracle.quant_row_words(L, bits, lib)
            assert c.shape == (1, W) and W % 4 == 0 and W * 32 >= L * bits
            if L == 1:
                assert np.all(c == 0)
                continue
            assert s[0] == 1.0 and m[0] == 0.0, (bits, L, s, m)
            assert stream_codes(c[0], bits, L).tolist() == q.tolist(), (bits, L)
            rest = np.unpackbits(c[0].astype("<u4").view(np.uint8), bitorder="little")[L * bits:]
            assert not rest.any()  # padding bits are zero
            assert np.array_equal(oracle.quant_decompress(c, s, m, L, bits, lib), x)


def pin_quant_bounds(lib, seed: int = 11):
    rng = np.random.default_rng(seed)
    x = (rng.standard_normal((32, 1000)) * rng.uniform(0.001, 100, (32, 1))).astype(np.float32)
    for bits in (2, 4, 6, 8):
        c, s, m = oracle.quant_compress(x, bits, lib=lib)
        y = oracle.quant_decompress(c, s, m, 1000, bits, lib)
        q = np.stack([stream_codes(c[r], bits, 1000) for r in range(32)])
        levels = (1 << bits) - 1
        for r in range(32):
            mn, mx = x[r].min(), x[r].max()
            assert m[r] == mn
            assert np.isclose(s[r], (np.float64(mx) - mn) / levels, rtol=1e-6)
            t = (x[r].astype(np.float64) - mn) / (np.float64(mx) - mn) * levels
            assert np.all(np.abs(t - q[r]) <= 0.5 + 1e-4)  # nearest code
            assert q[r, np.argmin(x[r])] == 0 and q[r, np.argmax(x[r])] == levels
            assert y[r, np.argmin(x[r])] == mn  # the minimum comes back exactly
            ulp = np.spacing(np.float32(max(abs(mn), abs(mx))))
            assert np.all(np.abs(x[r].astype(np.float64) - y[r]) <= s[r] / 2 + 4 * ulp)


def pin_quant_identity32(lib, seed: int = 12):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((5, 77)).astype(np.float32)
    x[0, 0] = -0.0
    x[1, 1] = np.float32(1e-40)  # subnormal
    c, s, m = oracle.quant_compress(x, 32, lib=lib)
    y = oracle.quant_decompress(c, s, m, 77, 32, lib)
    assert np.array_equal(bits_of(y), bits_of(x))


def pin_quant_stochastic(lib, seed: int = 13, n_seeds: int = 10000):
    """Codes bracket t; over many seeds the dequantised mean is x (unbiased)."""
    rng = np.random.default_rng(seed)
    L, bits = 1000, 4
    # min 0 and max 15 are present, so scale = inv = 1 and t = x exactly
    x = np.sort(rng.uniform(0, 15, L)).astype(np.float32)
    x = np.round(x * 256) / 256  # exact fractions
    x[0], x[-1] = 0.0, 15.0
    x = x.astype(np.float32)[None, :]
    acc = np.zeros(L)
    fl = np.floor(x[0].astype(np.float64))
    for sd in range(n_seeds):
        c, s, m = oracle.quant_compress(x, bits, stochastic=True, seed=sd, lib=lib)
        q = stream_codes(c[0], bits, L)
        assert np.all((q == fl) | (q == fl + 1))
        acc += q
    mean = acc / n_seeds
    f = x[0] - fl
    sigma = np.sqrt(f * (1 - f) / n_seeds)
    assert np.all(np.abs(mean - x[0]) <= 5.5 * sigma + 2e-4)
    # the same seed gives the same codes, another seed other codes
    a = oracle.quant_compress(x, bits, True, 77, lib)[0]
    b = oracle.quant_compress(x, bits, True, 77, lib)[0]
    d = oracle.quant_compress(x, bits, True, 78, lib)[0]
    assert np.array_equal(a, b) and not np.array_equal(a, d)


def pin_aqsgd_quant(lib, seed: int = 16):
    """AQ-SGD with quantisation (§2.5): the stored rows take exactly the dequantised
    message (the same fp32 add), untouched samples stay bit-identical, the receiver's
    copy follows bit for bit; with an empty buffer the message is the plain quantisation
    of x; and the codes are those of the quantiser applied to x - buf, read back with
    numpy from the bitstream."""
    rng = np.random.default_rng(seed)
    S, rps, L = 9, 2, 100
    buf = rng.standard_normal((S, rps, L)).astype(np.float32)
    before = buf.copy()
    recv = buf.copy()
    ids = np.array([4, 0, 7], np.int64)
    x = rng.standard_normal((3, rps, L)).astype(np.float32)
    for bits, sr in ((4, False), (6, True), (2, True)):
        b0 = buf.copy()
        c, s, m = oracle.aqsgd_quant_compress(x, buf, ids, bits, sr, 11, lib)
        d = (x - b0[ids]).reshape(3 * rps, L)
        c2, s2, m2 = oracle.quant_compress(d, bits, sr, 11, lib)
        assert np.array_equal(c, c2) and np.array_equal(bits_of(s), bits_of(s2))
        dh = oracle.quant_decompress(c, s, m, L, bits, lib).reshape(3, rps, L)
        assert np.array_equal(bits_of(buf[ids]), bits_of(b0[ids] + dh))
        untouched = np.setdiff1d(np.arange(S), ids)
        assert np.array_equal(bits_of(buf[untouched]), bits_of(before[untouched]))
        oracle.aqsgd_quant_decompress(c, s, m, recv, ids, bits, lib)
        assert np.array_equal(bits_of(recv), bits_of(buf))
    zero = np.zeros((S, rps, L), np.float32)
    c, s, m = oracle.aqsgd_quant_compress(x, zero, ids, 8, False, 0, lib)
    c2, s2, m2 = oracle.quant_compress(x.reshape(3 * rps, L), 8, False, 0, lib)
    assert np.array_equal(c, c2) and np.array_equal(bits_of(m), bits_of(m2))
    q = stream_codes(c[0], 8, L)
    assert q.min() >= 0 and q.max() == 255


ALL_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_")]
