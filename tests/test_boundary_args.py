"""Argument checks of the compression block (no GPU needed)."""

import pytest


def test_block_arguments():
    import paper_2401_07788_gb300 as m

    with pytest.raises(ValueError):
        m.CompressionBoundary(m.Reuse(), None)
    with pytest.raises(ValueError):
        m.CompressionBoundary(m.Quant(4), m.Reuse())
    with pytest.raises(ValueError):
        m.CompressionBoundary(m.TopK(10), m.TopK(10, feedback="ef"))
    with pytest.raises(ValueError):
        m.CompressionBoundary(m.TopK(10, feedback="aqsgd"), None)
    with pytest.raises(ValueError):
        m.CompressionBoundary(m.Quant(4, feedback="aqsgd"), None)
    with pytest.raises(ValueError):
        m.CompressionBoundary(m.TopK(10), m.Quant(4, feedback="aqsgd"), aqsgd_samples=4)
    with pytest.raises(ValueError):
        m.Quant(4, feedback="ef")
    with pytest.raises(ValueError):
        m.TopK(10, feedback="other")
    with pytest.raises(ValueError):
        m.CompressionBoundary(m.TopK(10), None, rows="column")
    b = m.CompressionBoundary(m.TopK(10), m.Reuse())
    assert b.training and b.state is None
    seq = m.with_boundaries([object.__new__(type("S", (), {}))] * 0, lambda i: None)
    assert len(seq) == 0
