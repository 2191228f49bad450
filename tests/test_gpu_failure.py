"""Failure paths, exercised without a GPU fault.

An in-kernel wait that runs out: with a short wait bound (DARD_TEST_WAIT_CYCLES) each
tensor-core attention kernel is told not to issue one K copy (DARD_TEST_DROP_KV; nothing
invalid is issued, the copy simply never lands). Every wait that depends on it gives up,
the launch ends with DARD_STATUS_TIMEOUT in the status word, and a normal call on the same
device afterwards matches the oracle. An injected launch failure (DARD_TEST_FAIL_LAUNCH:
the launcher reports cudaErrorLaunchFailure without launching) returns DARD_ERR_CUDA with
the CUDA message from dard_last_error(), and the next call works.
"""
import pytest
import torch

from paper_2608_26574_gb300 import binding as B
from paper_2608_26574_gb300 import workloads as W
from paper_2608_26574_gb300.device import DeviceStep

from . import parity as P

pytestmark = pytest.mark.gpu

STATUS_TIMEOUT = 0x8


def _small(vocab=None):
    specs = [dict(n_orig=300, block_start=200, block_len=32, fractions=(0.4, 0.3, 0.3))]
    kw = {} if vocab is None else dict(vocab=vocab)
    return W.custom(specs, 2, 2, 128, seed=5, **kw)


@pytest.mark.parametrize("tc", ["1", "2", "4"])
def test_wait_runs_out_and_the_device_stays_usable(monkeypatch, tc):
    """Every tensor-core kernel: the one-tile and two-tile kernels drop the K copy of key
    tile 1 in every CTA, the CTA-pair kernel the second K stage use of every pair."""
    wl = _small()
    ds = DeviceStep(wl, layers=[0], scoring=False)
    monkeypatch.setenv("DARD_ATTN_TC", tc)
    monkeypatch.setenv("DARD_TEST_WAIT_CYCLES", str(1 << 20))  # about half a millisecond
    monkeypatch.setenv("DARD_TEST_DROP_KV", "1")
    ds.attention(0)
    torch.cuda.synchronize()
    assert int(ds.status.item()) & STATUS_TIMEOUT
    monkeypatch.delenv("DARD_TEST_WAIT_CYCLES")
    monkeypatch.delenv("DARD_TEST_DROP_KV")
    ds.status.zero_()
    o = ds.attention(0)
    torch.cuda.synchronize()
    assert int(ds.status.item()) == 0
    mx, mean, _ = P.compare_attention(wl, 0, o.float().cpu().numpy())
    assert mx <= P.ATT_MAX_ABS and mean <= P.ATT_MEAN_ABS


@pytest.mark.parametrize("which", ["attention", "scoring"])
def test_injected_launch_failure(monkeypatch, which):
    wl = _small(vocab=4096)
    ds = DeviceStep(wl, layers=[0])
    run = (lambda: ds.attention(0)) if which == "attention" else (lambda: ds.score())
    monkeypatch.setenv("DARD_TEST_FAIL_LAUNCH", "1")
    with pytest.raises(B.DardError) as err:
        run()
    assert err.value.code == 5  # DARD_ERR_CUDA
    assert "launch failed" in str(err.value) and "DARD_TEST_FAIL_LAUNCH" in str(err.value)
    monkeypatch.delenv("DARD_TEST_FAIL_LAUNCH")
    run()
    torch.cuda.synchronize()
    assert int(ds.status.item()) == 0
