"""ro_batch_ready (Section 4.3, Eq. 2) takes one of two paths: candidate
lists of up to a few thousand tiles go through one cooperative kernel
(claims, grid barrier, tile counts, grid barrier, writes); longer lists, and
every admission when RO_ADMIT_TWO_PASS=1 is set at context creation, go
through the count and scatter passes.  The admission tests elsewhere run on
the first path (their lists are short) and the full-size ones on the second
(the 1M-document list is 16.4M children long); here the same scenarios run
again on the two-pass path, each against the oracle: explicit lists with
repeats and ids past the expansion, Calls and a refused reservation, the
streaming configuration's waves, Call streams with a GroupFailure (sealed
queue entries leave undispatched) and a retry (recovery groups go first),
and random GroupFailures and retried attempts across many calls."""
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _two_pass(monkeypatch):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    monkeypatch.setenv("RO_ADMIT_TWO_PASS", "1")


@pytest.mark.parametrize("seed", range(2))
def test_two_pass_waves_with_duplicates(seed):
    from tests import test_gpu_parity
    test_gpu_parity.test_batch_ready_waves_with_duplicates(seed)


def test_two_pass_calls_and_capacity():
    from tests import test_gpu_parity
    test_gpu_parity.test_batch_ready_calls_and_capacity()


@pytest.mark.parametrize("B", [32, 2048])
def test_two_pass_streaming_calls(B):
    from tests import test_gpu_parity
    test_gpu_parity.test_pipeline_streaming_calls(B)


def test_two_pass_call_streams_with_failures_retries_and_capacity():
    from tests import test_gpu_streams
    test_gpu_streams.test_call_streams_with_failures_retries_and_capacity()


def test_two_pass_random_group_failures():
    from tests import test_gpu_group_failure
    test_gpu_group_failure.test_random_group_failures_many_calls(0)


def test_two_pass_retried_attempts():
    from tests import test_gpu_retry
    test_gpu_retry.test_random_failed_attempts_with_late_stale_reports(0)
