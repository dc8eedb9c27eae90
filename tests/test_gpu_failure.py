"""Failure detection on the GPU without a fault: a bounded wait runs out.

A kernel waits on an mbarrier that nothing completes; after a 50 ms limit it
records GF_ETIMEOUT and returns.  The host reads the status, and the same
CUDA context then runs ordinary work correctly.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def test_bounded_wait_runs_out_and_the_context_stays_usable():
    import paper_2605_31464_gb300 as gf
    from paper_2605_31464_gb300 import _build
    _build.build()
    s = torch.cuda.current_stream().cuda_stream
    assert gf.gf_selftest_timeout(50, s) == gf.GF_ETIMEOUT
    assert "timed out" in gf.gf_last_error()
    # the status word was cleared and the context still works
    gf.gf_gemm_status(s)
    lg = torch.zeros(2, 16, device="cuda")
    lg[1, 11] = float(np.log(4.0))
    p, conf, arg, defer = gf.verdict(lg, (10, 11), 0.5)
    np.testing.assert_allclose(p.cpu().numpy()[1], [0.2, 0.8], atol=1e-6)
    assert list(defer.cpu().numpy()) == [0, 0]


def test_selftest_rejects_bad_limits():
    import paper_2605_31464_gb300 as gf
    assert gf.gf_selftest_timeout(0, None) == gf.GF_EINVAL
    assert gf.gf_selftest_timeout(5000, None) == gf.GF_EINVAL
