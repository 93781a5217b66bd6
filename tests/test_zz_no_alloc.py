"""gar_allreduce_noalloc: the step-faithful Allreduce for callers that cannot allocate
device memory while they run it (their memory is owned by a caching allocator or by
another runtime).  It keeps its workspace in a fixed device array inside the library,
so it must give exactly what the regular step-faithful entry point and the CPU oracle
give -- bit for bit, the tolerance every parity test here uses -- on consecutive calls
that reuse that array (also when plans of different sizes take turns), it must not
change the device's free memory, and it must refuse plans whose workspace does not fit.

Collected last on purpose (file name), so a failure here stops a -x run only after
every other test has run.  Independent of test order and process state.
"""

import ctypes

import numpy as np
import pytest
import torch

import gar_inputs
from oracle import gar_oracle as O

pytestmark = pytest.mark.gpu

gar = pytest.importorskip("paper_2004_09362_gb300.gar")


def _rows(t):
    """[P, n] tensor on the GPU whose rows are 16-byte aligned (row stride padded)."""
    P, n = t.shape
    per16 = 16 // t.element_size()
    n_pad = max(per16, (n + per16 - 1) // per16 * per16)
    store = torch.zeros((P, n_pad), dtype=t.dtype, device="cuda")
    store[:, :n] = t.to("cuda")
    return store


def _noalloc(plan, store):
    P = store.shape[0]
    ptrs = (ctypes.c_void_p * P)(*[store[x].data_ptr() for x in range(P)])
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return gar._lib.gar_allreduce_noalloc(plan.handle, ptrs, stream)


def _bits(t):
    a = t.contiguous().cpu()
    return a.view(torch.int16 if a.element_size() == 2 else torch.int32).numpy()


def _host(x, dtype):
    t = x.float() if dtype == "bf16" else x
    return [t[r].numpy().copy() for r in range(t.shape[0])]


def _assert_oracle(got, x, dtype, op, S):
    want = O.allreduce(_host(x, dtype), S, op, dtype)
    g = got.float().cpu().numpy() if dtype == "bf16" else got.cpu().numpy()
    for r in range(len(want)):
        np.testing.assert_array_equal(g[r].view(np.int32), np.asarray(want[r], g.dtype).view(np.int32))


CASES = [
    (7, 1001, "f32", "sum", 3),            # latency-optimal: ping-pong + q* slices
    (8, 262144, "f32", "sum", 4),          # 1 MiB per rank, intermediate step count
    (6, 999, "bf16", "sum", 6),            # bandwidth-optimal bf16: fp32 partial slice
    (5, 1024, "i32", "max", 4),
    (24, 24 * 1000 + 7, "f32", "sum", 7),  # ragged blocks, K = 6
    (2, 33, "f32", "sum", 1),              # P = 2 latency-optimal (finalize launch)
    (64, 4096 + 5, "f32", "sum", 6),       # GAR_NOALLOC_MAX_P, latency-optimal: 2P ops a launch
    (64, 4096 + 5, "bf16", "sum", 12),     # GAR_NOALLOC_MAX_P, bandwidth-optimal
]


@pytest.mark.parametrize("P,n,dtype,op,S", CASES)
def test_noalloc_matches_step_faithful_on_consecutive_calls(P, n, dtype, op, S):
    plan = gar.gar_plan_create(P, n, dtype, op, S)
    ws, _, _ = gar.gar_plan_bytes(plan)
    assert ws <= gar_scratch_bytes()
    dist = ("int", -1000, 1000) if dtype == "i32" else ("normal", 0.0, 1.0)
    for call in range(2):
        x = gar_inputs.rank_inputs(P, n, dtype, dist, seed=100 * P + call)
        mine, ref = _rows(x), _rows(x)
        rc = _noalloc(plan, mine)
        assert rc == 0, gar.gar_last_error()
        gar.gar_allreduce(plan, ref, "step")
        torch.cuda.synchronize()
        np.testing.assert_array_equal(_bits(mine[:, :n]), _bits(ref[:, :n]))
        _assert_oracle(mine[:, :n], x, dtype, op, S)


def gar_scratch_bytes():
    return 64 << 20     # GAR_NOALLOC_SCRATCH_BYTES in include/gar.h


def test_noalloc_rejects_plans_that_do_not_fit():
    big = gar.gar_plan_create(24, 16 << 20, "f32", "sum", 7)      # 3 x 1.5 GiB workspace
    store = torch.empty((24, 16), device="cuda")
    assert _noalloc(big, store) == -1
    assert "bytes of workspace" in gar.gar_last_error()
    many = gar.gar_plan_create(65, 1000, "f32", "sum", gar.GAR_STEPS_BO)
    store = torch.empty((65, 16), device="cuda")
    assert _noalloc(many, store) == -1
    assert "P <=" in gar.gar_last_error()


def test_noalloc_alternating_plans_and_free_memory():
    """Two plans of different sizes take turns on one stream: each call starts from what
    the other left in the shared array and still gives the oracle's bits; once the
    library is loaded, a call leaves the device's free memory unchanged."""
    a = (gar.gar_plan_create(64, 3000, "f32", "sum", 6), 64, 3000, 6)
    b = (gar.gar_plan_create(5, 70001, "f32", "sum", 4), 5, 70001, 4)
    first = True
    for i, (plan, P, n, S) in enumerate([a, b, a, b, a]):
        x = gar_inputs.rank_inputs(P, n, "f32", ("normal", 0.0, 1.0), seed=7 + i)
        mine = _rows(x)
        torch.cuda.synchronize()
        free0, _ = torch.cuda.mem_get_info()
        assert _noalloc(plan, mine) == 0, gar.gar_last_error()
        torch.cuda.synchronize()
        free1, _ = torch.cuda.mem_get_info()
        if not first:
            assert free1 == free0
        first = False
        _assert_oracle(mine[:, :n], x, "f32", "sum", S)
