"""Shared helpers for the GPU parity tests: seeded rows of the value distributions the
selection and quantisation must handle, and bitwise comparison."""

from __future__ import annotations

import numpy as np

KINDS = ("normal", "relu", "zeros", "equal", "ties", "signed_zero", "heavy", "outlier")


def rows_of(kind: str, R: int, L: int, seed: int) -> np.ndarray:
    rng = np.random.default_rng(seed)
    if kind == "normal":
        x = rng.standard_normal((R, L))
    elif kind == "relu":
        x = np.maximum(rng.standard_normal((R, L)), 0.0)
    elif kind == "zeros":
        x = np.zeros((R, L))
    elif kind == "equal":
        x = np.full((R, L), -1.25)
    elif kind == "ties":  # few distinct magnitudes, both signs
        x = rng.integers(-3, 4, (R, L)).astype(np.float64)
    elif kind == "signed_zero":
        x = rng.standard_normal((R, L))
        x[rng.random((R, L)) < 0.6] = 0.0
        x = np.where(rng.random((R, L)) < 0.5, -np.abs(x) * (x == 0) + x * (x != 0), x)
        x = x.astype(np.float32)
        x[(x == 0) & (rng.random((R, L)) < 0.5)] = -0.0
        return np.ascontiguousarray(x, dtype=np.float32)
    elif kind == "heavy":  # magnitudes over many decades
        x = rng.standard_normal((R, L)) * 10.0 ** rng.integers(-20, 20, (R, L))
    elif kind == "outlier":  # one huge entry per row: the first histogram collapses
        x = rng.standard_normal((R, L))
        x[:, rng.integers(0, L)] = 1e30
    else:
        raise ValueError(kind)
    return np.ascontiguousarray(x, dtype=np.float32)


def u32(a) -> np.ndarray:
    return np.ascontiguousarray(a).view(np.uint32)


def assert_bits_equal(got: np.ndarray, want: np.ndarray, what: str) -> None:
    got = np.ascontiguousarray(got)
    want = np.ascontiguousarray(want)
    assert got.shape == want.shape, "%s: shape %s != %s" % (what, got.shape, want.shape)
    g = got.view(np.uint32) if got.dtype.itemsize == 4 else got
    w = want.view(np.uint32) if want.dtype.itemsize == 4 else want
    if not np.array_equal(g, w):
        bad = np.argwhere(g != w)
        i = tuple(bad[0])
        raise AssertionError("%s: %d mismatches, first at %s: got %r want %r"
                             % (what, len(bad), i, got[i], want[i]))


def row_blocks(fn, n_rows: int, *arrays, threads: int = 16):
    """Run ``fn(*blocks)`` on row blocks of ``arrays`` in threads and stack the results.

    For oracle calls that treat rows independently and whose results do not depend on a
    row's position in the call (TopK, error feedback, EF21, nearest quantisation; not
    stochastic rounding, whose counter runs over the flat index of the call).  The oracle
    is a C library called through ctypes, which releases the GIL, so blocks run on
    separate cores.  Arrays updated in place are passed as views of their row blocks."""
    from concurrent.futures import ThreadPoolExecutor

    step = max(1, -(-n_rows // threads))
    spans = [(r, min(n_rows, r + step)) for r in range(0, n_rows, step)]
    with ThreadPoolExecutor(len(spans)) as ex:
        outs = list(ex.map(lambda s: fn(*(a[s[0]:s[1]] for a in arrays)), spans))
    if outs and isinstance(outs[0], tuple):
        return tuple(np.concatenate(parts, axis=0) for parts in zip(*outs))
    return outs
