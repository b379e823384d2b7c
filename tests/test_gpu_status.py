"""Device-side waits give up cleanly: with the spin limit at 0 every first wait on a bulk
copy gives up, the kernel records a timeout in the status word, drains its copy and
returns; the context stays usable.  No fault, trap or hang is involved."""

import numpy as np
import pytest
import torch

import oracle
from gpu_cases import assert_bits_equal, rows_of

pytestmark = pytest.mark.gpu

DEFAULT_SPIN = 1 << 20


@pytest.fixture(scope="module")
def mpc():
    import __graft_entry__ as g

    g.build()
    import paper_2401_07788_gb300 as m

    torch.cuda.set_device(0)
    yield m
    m.mpc_set_knob(m.MPC_KNOB_SPIN_LIMIT, DEFAULT_SPIN)


# (op, row length, TopK path knob): the band kernel, the cluster kernels (knob 3: the
# two-pass row kernel, which waits on no copy, stays out), the warp kernel, quantisation
@pytest.mark.parametrize("op,L,path", [("ef", 4096, 0), ("ef", 32768, 3), ("plain", 768, 0),
                                       ("quant", 32768, 0)])
def test_timeout_is_reported_and_context_survives(mpc, op, L, path):
    x = torch.from_numpy(rows_of("normal", 6, L, seed=1)).cuda()
    err = torch.zeros_like(x)
    mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, path)
    mpc.mpc_set_knob(mpc.MPC_KNOB_SPIN_LIMIT, 0)
    try:
        if op == "ef":
            mpc.mpc_ef_topk_compress(x, err, L // 10)
        elif op == "plain":
            mpc.mpc_topk_compress(x, L // 10)
        else:
            mpc.mpc_quant_compress(x, 4)
        assert mpc.mpc_get_status() == 5  # MPC_ERR_TIMEOUT
        assert "wait" in mpc.mpc_last_error()
    finally:
        mpc.mpc_set_knob(mpc.MPC_KNOB_SPIN_LIMIT, DEFAULT_SPIN)
        mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, 0)
    assert mpc.mpc_get_status() == 0
    # the same call now succeeds and matches the oracle
    xn = x.cpu().numpy()
    v, i = mpc.mpc_topk_compress(x, L // 10)
    ov, oi = oracle.topk_compress(xn, L // 10)
    assert mpc.mpc_get_status() == 0
    assert_bits_equal(i.cpu().numpy(), oi, "idx after timeout")
    assert_bits_equal(v.cpu().numpy(), ov, "vals after timeout")


def test_results_do_not_depend_on_dependent_launch(mpc):
    """The same sequence of dependent calls (error feedback carried across steps, then
    decompression and quantisation of the result) gives the same bits with programmatic
    dependent launch on and off."""
    import numpy as np

    def run():
        torch.manual_seed(0)
        x = torch.randn(64, 32768, device="cuda")
        e = torch.zeros_like(x)
        outs = []
        for _ in range(3):
            v, i = mpc.mpc_ef_topk_compress(x, e, 3276)
            y = mpc.mpc_topk_decompress(v, i, 32768)
            c, s, m = mpc.mpc_quant_compress(y, 4, stochastic=True, seed=5)
            outs += [v, i, e.clone(), mpc.mpc_quant_decompress(c, s, m, 32768, 4)]
            x = x + 0.1
        torch.cuda.synchronize()
        return [o.cpu().numpy() for o in outs]

    try:
        mpc.mpc_set_knob(mpc.MPC_KNOB_PDL, 1)
        a = run()
        mpc.mpc_set_knob(mpc.MPC_KNOB_PDL, 0)
        b = run()
    finally:
        mpc.mpc_set_knob(mpc.MPC_KNOB_PDL, 1)
    for p, q in zip(a, b):
        assert np.array_equal(p.view(np.uint32) if p.dtype.itemsize == 4 else p,
                              q.view(np.uint32) if q.dtype.itemsize == 4 else q)
    assert mpc.mpc_get_status() == 0

