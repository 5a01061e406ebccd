"""Failure detection without a GPU fault: a bounded device wait that runs out (on a barrier that
nothing arrives at) is reported to the host as BLA_ERR_TIMEOUT, and the context stays usable."""
import pytest

from gpu_util import TOL_BF16, rel, require_cuda, to_dev

pytestmark = pytest.mark.gpu


def test_wait_timeout_is_reported_and_context_survives(orc):
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_qkv
    dev = require_cuda()
    bla.bla_device_error()                      # no stale error
    bla.bla_selftest_wait_timeout(20)
    with pytest.raises(bla.BlaError) as ei:
        bla.bla_device_error()
    assert ei.value.status == bla.BLA_ERR_TIMEOUT
    assert b"kernel 15" in bla.load().bla_last_error_string()
    bla.bla_device_error()                      # the error word was cleared by the report
    # the context still runs the forward correctly
    q, k, v = make_qkv(1, 2, 300, 64, dtype="bf16", seed=5)
    o, _, _ = bla.bla_forward_chunked(to_dev(q, dev, torch.bfloat16), to_dev(k, dev, torch.bfloat16),
                                      to_dev(v, dev, torch.bfloat16), 32, 32, 256.0)
    bla.bla_device_error()
    ref = orc.forward(q, k, v, 32, 32, 256.0, form="modes")
    assert rel(o.float().cpu().numpy(), ref["o"]) <= TOL_BF16


def test_selftest_rejects_bad_limit():
    from paper_2606_09862_gb300 import bla
    require_cuda()
    with pytest.raises(bla.BlaError):
        bla.bla_selftest_wait_timeout(0)
