"""The averaging entry point that allocates nothing, against the context-based one.

adpsgd_average_and_variance_static serves callers that cannot allocate device memory
themselves: code inside a host framework whose pool allocator owns the GPU's memory, and
latency-critical code where cudaMalloc / cudaFree would synchronise the device.  It keeps its
partial sums in a fixed array inside the library instead of a context's allocation.  Two
calls in a row, with different shapes so that the second reuses the array left by the first,
must give what adpsgd_average_and_variance gives on the same input: the same averaged
parameters bit for bit, and the variance and loss within the relative 1e-4 the parity tests
use.  This file is collected last, so a run that stops at the first failure has already run
every other test.
"""
import numpy as np
import pytest

from paper_2007_06134_gb300 import abi, inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
DEV = "cuda:0"
REL = 1e-4


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def _rel(a, b):
    return abs(a - b) / max(abs(b), 1e-300)


def _with_context(x, h, c):
    xd = _dev(x)
    n, P = x.shape
    with abi.adpsgd_init(abi.make_config(n, P), xd, torch.zeros_like(xd), _dev(h), _dev(c)) as ctx:
        D, L = abi.adpsgd_average_and_variance(ctx)
    torch.cuda.synchronize()
    return xd.cpu().numpy(), D, L


def test_static_scratch_entry_matches_context_entry_on_two_calls():
    w = inputs.WORKLOADS["resnet18-n8"]
    cases = [(8, (1 << 22) + 3 * 4), (3, 4099)]  # a large grid first, then a smaller one
    for call, (n, P) in enumerate(cases):
        h, c = inputs.problem(w, P)
        x, _ = inputs.random_state(n, P, 100 + call)
        ref_x, ref_D, ref_L = _with_context(x, h, c)
        xd = _dev(x)
        D, L = abi.adpsgd_average_and_variance_static(xd, _dev(h), _dev(c), n, P)
        torch.cuda.synchronize()
        got_x = xd.cpu().numpy()
        assert np.array_equal(got_x.view(np.uint32), ref_x.view(np.uint32)), f"call {call}: averaged x"
        assert _rel(D, ref_D) <= REL, (call, D, ref_D)
        assert _rel(L, ref_L) <= REL, (call, L, ref_L)


def test_static_scratch_entry_without_loss_and_argument_checks():
    n, P = 4, 1 << 16
    x, _ = inputs.random_state(n, P, 7)
    h = np.ones(P, np.float32)
    ref_x, ref_D, _ = _with_context(x, h, h)
    xd = _dev(x)
    D, L = abi.adpsgd_average_and_variance_static(xd, None, None, n, P, want_loss=False)
    torch.cuda.synchronize()
    assert L is None and _rel(D, ref_D) <= REL
    assert np.array_equal(xd.cpu().numpy(), ref_x)
    with pytest.raises(abi.AdpsgdError) as e:
        abi.adpsgd_average_and_variance_static(xd, None, None, n, P, want_loss=True)
    assert e.value.status == abi.E_INVAL
    with pytest.raises(abi.AdpsgdError) as e:
        abi.adpsgd_average_and_variance_static(xd, None, None, 0, P, want_loss=False)
    assert e.value.status == abi.E_INVAL


def test_static_scratch_entry_refuses_misaligned_x():
    n, P = 2, 4096
    xd = torch.zeros(n * P + 4, device=DEV)
    with pytest.raises(abi.AdpsgdError) as e:
        abi.adpsgd_average_and_variance_static(xd[1:], None, None, n, P, want_loss=False)
    assert e.value.status == abi.E_ALIGN


def test_static_scratch_entry_bounded_wait_behind_queued_work():
    # A short wait limit behind work already queued on the stream returns E_TIMEOUT without
    # blocking; once the stream has drained, the next call returns the right sums.
    w = inputs.WORKLOADS["resnet18-n8"]
    n, P = 8, 1 << 22
    h, c = inputs.problem(w, P)
    busy_x = torch.zeros((n, P), device=DEV)
    busy_v = torch.zeros_like(busy_x)
    x, _ = inputs.random_state(4, 4096, 21)
    ref_x, ref_D, _ = _with_context(x, np.ones(4096, np.float32), np.zeros(4096, np.float32))
    xd = _dev(x)
    with abi.adpsgd_init(abi.make_config(n, P), busy_x, busy_v, _dev(h), _dev(c)) as ctx:
        abi.adpsgd_local_steps(ctx, 0, [0.01] * 400)  # tens of milliseconds of queued work
        with pytest.raises(abi.AdpsgdError) as e:
            abi.adpsgd_average_and_variance_static(xd, None, None, 4, 4096, want_loss=False, wait_timeout_ms=1)
        assert e.value.status == abi.E_TIMEOUT
        torch.cuda.synchronize()
    assert np.array_equal(xd.cpu().numpy(), ref_x)  # the timed-out averaging still ran to the end
    D, _ = abi.adpsgd_average_and_variance_static(xd, None, None, 4, 4096, want_loss=False)
    assert D == 0.0  # averaged replicas have no spread
    xd.copy_(_dev(x))
    D, _ = abi.adpsgd_average_and_variance_static(xd, None, None, 4, 4096, want_loss=False)
    torch.cuda.synchronize()
    assert _rel(D, ref_D) <= REL
