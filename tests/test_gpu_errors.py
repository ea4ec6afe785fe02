"""Device-side timeout path: a bounded wait on an mbarrier nothing arrives at
gives up, sets the error word and leaves the context usable."""
import pytest
import torch

pytestmark = pytest.mark.gpu


def test_wait_timeout_is_reported_and_context_survives(cuda_ok):
    from paper_2609_32415_gb300 import api
    from paper_2609_32415_gb300._lib import RA_ETIMEOUT, RefAdaptError
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    api.refadapt_selftest_wait_timeout(err, 2_000_000)   # 2 ms budget
    with pytest.raises(RefAdaptError) as e:
        api.refadapt_check_error(err)
    assert e.value.status == RA_ETIMEOUT
    assert err.item() == 0                                # check_error clears it
    x = torch.ones(1024, device="cuda")
    assert float(x.sum()) == 1024.0                        # context still usable
    api.refadapt_check_error(err)                          # and the word reads clean
