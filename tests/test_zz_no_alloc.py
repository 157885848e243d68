"""poseidon_argmin_noalloc, the argmin for callers that cannot allocate device
memory during a call (their device memory belongs to another allocator, or
allocation is forbidden after start-up).  It must give exactly the index
poseidon_argmin gives, on two calls in a row that share its fixed scratch.
This file is collected last on purpose."""
import ctypes as C

import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def test_noalloc_argmin_matches_allocating_argmin_twice():
    import torch

    import paper_2609_06086_gb300 as P
    L = P.lib()
    stream = torch.cuda.current_stream().cuda_stream
    rng = np.random.default_rng(31)
    # the second call has fewer blocks than the first, so it must not read
    # partial results the first call left behind
    for n in (3_000_000, 5_000):
        T = rng.integers(0, 1000, n).astype(np.int32)
        F = (rng.random(n) < 0.3).astype(np.uint8)
        dT, dF = torch.from_numpy(T).cuda(), torch.from_numpy(F).cuda()
        want = torch.full((1,), -9, dtype=torch.int64, device="cuda")
        got = torch.full((1,), -9, dtype=torch.int64, device="cuda")
        assert L.poseidon_argmin(dT.data_ptr(), dF.data_ptr(), n, want.data_ptr(), stream) == 0
        assert L.poseidon_argmin_noalloc(dT.data_ptr(), dF.data_ptr(), n, got.data_ptr(),
                                         stream) == 0, L.poseidon_last_error()
        torch.cuda.synchronize()
        idx = np.flatnonzero(F == 1)
        assert got.item() == want.item() == int(idx[np.argmin(T[idx])])


def test_noalloc_argmin_edge_cases_and_no_device_allocation():
    """No entry (n = 0) and no feasible entry both give -1, as the
    allocating argmin does; 3,000,000 entries need more than 256 x 4 x
    (SM count) threads, so the partial results reach their 4-per-SM cap.
    After a first call (which may load the module holding the fixed array),
    a call changes neither the device's free memory nor torch's."""
    import torch

    import paper_2609_06086_gb300 as P
    L = P.lib()
    stream = torch.cuda.current_stream().cuda_stream
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    n_big = 3_000_000
    assert n_big > 256 * 4 * sms
    rng = np.random.default_rng(37)
    cases = [(np.zeros(0, np.int32), np.zeros(0, np.uint8)),
             (rng.integers(0, 50, 70_000).astype(np.int32), np.zeros(70_000, np.uint8)),
             (rng.integers(0, 50, n_big).astype(np.int32),
              (rng.random(n_big) < 0.01).astype(np.uint8))]
    for T, F in cases:
        n = len(T)
        dT = torch.from_numpy(T).cuda() if n else torch.zeros(1, dtype=torch.int32, device="cuda")
        dF = torch.from_numpy(F).cuda() if n else torch.zeros(1, dtype=torch.uint8, device="cuda")
        want = torch.full((1,), -9, dtype=torch.int64, device="cuda")
        got = torch.full((1,), -9, dtype=torch.int64, device="cuda")
        assert L.poseidon_argmin(dT.data_ptr(), dF.data_ptr(), n, want.data_ptr(), stream) == 0
        assert L.poseidon_argmin_noalloc(dT.data_ptr(), dF.data_ptr(), n, got.data_ptr(),
                                         stream) == 0, L.poseidon_last_error()
        torch.cuda.synchronize()
        idx = np.flatnonzero(F == 1)
        expect = int(idx[np.argmin(T[idx])]) if len(idx) else -1
        assert got.item() == want.item() == expect
        free0, _ = torch.cuda.mem_get_info()
        used0 = torch.cuda.memory_allocated()
        got.fill_(-9)
        torch.cuda.synchronize()
        assert L.poseidon_argmin_noalloc(dT.data_ptr(), dF.data_ptr(), n, got.data_ptr(),
                                         stream) == 0
        torch.cuda.synchronize()
        assert torch.cuda.mem_get_info()[0] == free0
        assert torch.cuda.memory_allocated() == used0
        assert got.item() == expect


def test_noalloc_argmin_rejects_bad_arguments():
    import paper_2609_06086_gb300 as P
    L = P.lib()
    assert L.poseidon_argmin_noalloc(None, None, -1, None, None) == 1
    assert L.poseidon_argmin_noalloc(None, None, 10, C.c_void_p(16), None) == 1
