"""Failure detection on the GPU, without faulting it.

* Bounded waits: every wait inside the library's kernels gives up after a
  limit, records CER_ERR_TIMEOUT in the device status word and unwinds.
  cer_selftest_bounded_wait runs that same wait (flag polling, or an mbarrier
  phase) with a 1 ms limit on a flag nothing publishes / a phase nothing
  completes; the status must come back as CER_ERR_TIMEOUT, and the next
  ordinary call on the same context must be green.  Nothing else is in flight
  in that kernel: no copies, no MMAs, no tensor memory.
* Index lists: the checked scatter-add gets a keep list with a duplicate and
  one with an out-of-range entry, both planted on the host; the bad sequence
  is reported and left untouched, the good ones are updated bit-exactly.
"""
import time

import numpy as np
import pytest
import torch

from oracle import cer_oracle as ora
from paper_2608_29291_gb300 import cer
from tests.gpu_helpers import bf16_dev, bits_host, i32_dev

pytestmark = pytest.mark.gpu

TIMEOUT = 7
INDEX = 10


@pytest.fixture(scope="module", autouse=True)
def _device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    cer.load()
    cer.cer_sync_status()
    yield
    cer.cer_sync_status()


def _ordinary_call_is_green():
    lg = torch.tensor([[0.3, -1.0, 2.0, 0.5]], dtype=torch.float32, device="cuda")
    idx = torch.empty((1, 2), dtype=torch.int32, device="cuda")
    cer.cer_select_topk(lg, 0, 4, 2, idx)
    cer.cer_sync_status()
    assert idx.cpu().tolist() == [[2, 3]]


def _timed(fn):
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    fn()
    b.record()
    b.synchronize()
    return a.elapsed_time(b)


def test_flag_wait_that_nothing_publishes_times_out():
    flag = torch.zeros(1, dtype=torch.int64, device="cuda")
    ms = _timed(lambda: cer.cer_selftest_bounded_wait(0, flag, token=0x5EED, limit_us=1000))
    with pytest.raises(cer.CerError) as e:
        cer.cer_sync_status()
    assert e.value.status == TIMEOUT
    assert 0.9 <= ms < 1000.0, ms          # it waited about its limit, then gave up
    cer.cer_sync_status()                  # the status word was cleared
    _ordinary_call_is_green()


def test_flag_wait_that_is_published_returns():
    flag = torch.full((1,), 0x5EED, dtype=torch.int64, device="cuda")
    cer.cer_selftest_bounded_wait(0, flag, token=0x5EED, limit_us=1000)
    cer.cer_sync_status()


def test_mbarrier_wait_that_nothing_completes_times_out():
    ms = _timed(lambda: cer.cer_selftest_bounded_wait(1, arrive=False, limit_us=2000))
    with pytest.raises(cer.CerError) as e:
        cer.cer_sync_status()
    assert e.value.status == TIMEOUT
    assert 1.9 <= ms < 1000.0, ms
    _ordinary_call_is_green()


def test_mbarrier_wait_that_completes_returns():
    t0 = time.perf_counter()
    cer.cer_selftest_bounded_wait(1, arrive=True, limit_us=100000)
    cer.cer_sync_status()
    assert time.perf_counter() - t0 < 0.1   # returned at once, not after its 100 ms limit


def test_selftest_argument_checks():
    lib = cer.load()
    assert lib.cer_selftest_bounded_wait(2, None, 0, 0, 1000, None) == 4        # kind
    assert lib.cer_selftest_bounded_wait(0, None, 0, 0, 1000, None) == 1        # kind 0 needs a flag
    assert lib.cer_selftest_bounded_wait(1, None, 0, 0, 0, None) == 4           # limit below 1 us
    assert lib.cer_selftest_bounded_wait(1, None, 0, 0, 100001, None) == 4      # limit above 100 ms


def _rows(B, N, d, K, seed):
    rng = np.random.default_rng(seed)
    h = rng.normal(0, 1, (B, N, d)).astype(np.float32)
    from paper_2608_29291_gb300 import inputs as gen
    h = gen.f32_to_bf16_bits(h)
    idx, _ = ora.select_topk(rng.normal(0, 1, (B, N)).astype(np.float32), 0, N, K)
    Y = gen.f32_to_bf16_bits(rng.normal(0, 1, (B * K, d)).astype(np.float32))
    return h, idx, Y


@pytest.mark.parametrize("B,N,d,K", [(1, 1, 8, 1), (3, 100, 264, 37), (2, 4096, 3584, 1229)])
def test_checked_scatter_matches_oracle(B, N, d, K):
    h, idx, Y = _rows(B, N, d, K, 5)
    hd = bf16_dev(h)
    cer.cer_scatter_add_checked(hd, i32_dev(idx), bf16_dev(Y))
    cer.cer_sync_status()
    assert np.array_equal(bits_host(hd), ora.scatter_add(h, idx, ora.bf16_to_f64(Y)))


@pytest.mark.parametrize("fault", ["duplicate", "out_of_range", "negative"])
def test_checked_scatter_rejects_a_bad_sequence(fault):
    B, N, d, K = 3, 200, 64, 50
    h, idx, Y = _rows(B, N, d, K, 6)
    bad = idx.copy()
    if fault == "duplicate":
        bad[1, 7] = bad[1, 30]          # planted on the host: one row listed twice
    elif fault == "out_of_range":
        bad[1, 7] = N
    else:
        bad[1, 7] = -1
    hd = bf16_dev(h)
    cer.cer_scatter_add_checked(hd, i32_dev(bad), bf16_dev(Y))
    with pytest.raises(cer.CerError) as e:
        cer.cer_sync_status()
    assert e.value.status == INDEX
    got = bits_host(hd)
    want = ora.scatter_add(h, idx, ora.bf16_to_f64(Y))
    assert np.array_equal(got[1], h[1])                      # the bad sequence is untouched
    assert np.array_equal(got[[0, 2]], want[[0, 2]])         # the others are updated
    _ordinary_call_is_green()
