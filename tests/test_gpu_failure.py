"""Failure detection without a GPU fault: a bounded device wait runs out and
reports PPAS_DEVERR_TIMEOUT through the error flag; the context stays usable."""
import pytest
import torch

from _cases import assert_close, device_case, host64, oracle_full, run_step
from paper_2608_15171_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ppas():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_15171_gb300 import ppas as p
    return p


def test_wait_that_nothing_completes_times_out(ppas):
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    ppas.ppas_debug_wait_timeout(err, 2000)        # 2 ms limit, nothing ever arrives
    torch.cuda.synchronize()
    assert err.item() == ppas.PPAS_DEVERR_TIMEOUT
    # the context is still healthy: a normal step runs and is correct
    c = device_case(wl.QWEN25_3B, wl.StepShape([1, 70], [300, 200]), seed=31)
    out = run_step(ppas, c, True)
    torch.cuda.synchronize()
    assert_close(host64(out), oracle_full(c), "after timeout")


def test_timeout_entry_rejects_bad_arguments(ppas):
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    for lim in (0, 2_000_001):
        with pytest.raises(ppas.PpasError) as e:
            ppas.ppas_debug_wait_timeout(err, lim)
        assert e.value.status == ppas.PPAS_ERR_INVALID_ARG
    with pytest.raises(ppas.PpasError):
        ppas.ppas_debug_wait_timeout(None, 100)
