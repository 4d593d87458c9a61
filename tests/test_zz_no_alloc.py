"""Allocation-free compact attention (arckv_attend_static).

Some callers cannot allocate device memory when they run -- an inference
engine plugin whose execute step must not allocate, a serving loop with a
memory budget fixed up front.  arckv_attend_static serves them from a fixed
scratch array compiled into the library.  This file is collected last so that
a failure here leaves every other test already run; it passes alone in a
fresh process and after the rest of the suite.
"""
import ctypes

import numpy as np
import pytest
import torch

import synth
from oracle import parity
import paper_2609_36835_gb300 as pk
from paper_2609_36835_gb300 import workload

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def static_fn(lib):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    f = lib.arckv_attend_static
    P = ctypes.c_void_p
    f.argtypes = [ctypes.c_int32] * 4 + [ctypes.c_float, P, P, P, P, P, P]
    f.restype = ctypes.c_int
    lib.arckv_attend_static_floats.argtypes = [ctypes.c_int32] * 4
    lib.arckv_attend_static_floats.restype = ctypes.c_size_t
    return f


def _inputs(H, n, t, seed):
    rng = np.random.default_rng(seed)
    Q = workload.bf16_tensor(synth.bf16_round((rng.normal(size=(H, n, 128)) * 3).astype(np.float32)), "cuda")
    f = lambda *s: torch.from_numpy(rng.normal(size=s).astype(np.float32)).cuda()
    return Q, f(H, t, 128), f(H, t), f(H, t, 128)


def test_static_scratch_attend_matches_workspace_attend(static_fn, lib):
    """Two calls in a row against arckv_attend (the same kernels, so the same
    bits); from the second call on, a call changes neither the device's free
    memory nor torch's allocations: the first call on a device did the set-up."""
    H, n, t = 3, 200, 77
    stream = torch.cuda.current_stream().cuda_stream
    for call in range(2):                       # two calls in a row share the scratch array
        Q, Ck, beta, Cv = _inputs(H, n, t, seed=call)
        ref = pk.attend(Q, Ck, beta, Cv)        # the workspace entry point
        O = torch.full((H, n, 128), float("nan"), device="cuda")
        torch.cuda.synchronize()
        free0, alloc0 = torch.cuda.mem_get_info()[0], torch.cuda.memory_allocated()
        st = static_fn(H, n, t, 128, 0.0, Q.data_ptr(), Ck.data_ptr(), beta.data_ptr(), Cv.data_ptr(),
                       O.data_ptr(), stream)
        assert st == 0, pk.status_string(st)
        torch.cuda.synchronize()
        free1, alloc1 = torch.cuda.mem_get_info()[0], torch.cuda.memory_allocated()
        if call > 0:
            assert free1 == free0 and alloc1 == alloc0, (free0, free1, alloc0, alloc1)
        assert torch.equal(O, ref)
        assert parity.rel_fro(O.cpu().numpy(), ref.cpu().numpy()) <= 2e-3


def test_static_scratch_rejects_oversized_problem(static_fn, lib):
    H, n, t = 8, 4096, 4096                     # needs far more than the fixed scratch
    assert lib.arckv_attend_static_floats(H, n, t, 128) > (8 << 20)
    st = static_fn(H, n, t, 128, 0.0, 1, 1, 1, 1, 1, torch.cuda.current_stream().cuda_stream)
    assert st == 3
