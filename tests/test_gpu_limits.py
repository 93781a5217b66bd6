"""GPU parity at the size limits: the largest number of virtual ranks (GAR_MAX_P = 1024,
whose fused parameter block holds 2 x 1024 pointers) and more than 2^31 elements per
rank (element indices and byte offsets beyond 32 bits), against the CPU oracle."""

import numpy as np
import pytest
import torch

import gar_inputs
from oracle import gar_oracle as G

pytestmark = pytest.mark.gpu

gar = pytest.importorskip("paper_2004_09362_gb300.gar")


def _bits(a):
    a = np.ascontiguousarray(a)
    return a.view(np.uint32)


def _padded(t):
    P, n = t.shape
    n_pad = (n + 3) // 4 * 4
    store = torch.zeros((P, n_pad), dtype=t.dtype, device="cuda")
    store[:, :n] = t.to("cuda")
    return store


@pytest.mark.parametrize("S,mode", [(10, "step"), (15, "step"), (20, "step"), (20, "fused"),
                                    (19, "fused"), (20, "persistent")])
def test_maximum_p(S, mode):
    """P = 1024 ranks, 3 or 4 elements per block: step-faithful at the latency-optimal,
    an intermediate and the bandwidth-optimal step count; fused at the bandwidth-optimal
    one and at S = 19 (K = 2: a rotated program whose pointer tables are too large to
    store twice); persistent at the bandwidth-optimal one.  The latency-optimal fused
    program exceeds GAR_FUSED_MAX_OPS."""
    P = gar.GAR_MAX_P
    n = 3 * P + 5
    t = gar_inputs.rank_inputs(P, n, "f32", ("normal", 0.0, 1.0), 1024 + S)
    host = [t[x].numpy().copy() for x in range(P)]
    plan = gar.gar_plan_create(P, n, "f32", "sum", S)
    store = _padded(t)
    gar.gar_allreduce(plan, store, mode)
    torch.cuda.synchronize()
    got = store[:, :n].cpu().numpy()
    want = G.allreduce(host, S, "sum", "f32")
    for x in range(P):
        np.testing.assert_array_equal(_bits(got[x]), _bits(want[x]), err_msg=f"rank {x}")
    if mode != "fused":
        assert gar.gar_last_step_bytes(plan) == gar.gar_plan_bytes(plan)[1]


def _sample_positions(n, P, seed):
    rng = np.random.default_rng(seed)
    picks = [rng.integers(0, n, 2048), np.arange(2 ** 31 - 64, min(2 ** 31 + 64, n)), np.array([0, n - 1])]
    for (lo, hi) in G.block_bounds(n, P):
        picks.append(np.array([lo, lo + 1, hi - 2, hi - 1]))
    idx = np.unique(np.concatenate(picks))
    assert idx.min() >= 0 and idx.max() < n
    return idx


@pytest.mark.parametrize("S,mode", [(4, "fused"), (2, "fused"), (4, "step")])
def test_more_than_2_31_elements_per_rank(S, mode):
    """P = 3 ranks of n = 2^31 + 37 fp32 (8.6 GB each, ragged blocks): sampled positions
    (random, those from 2^31 - 64 to the end, both ends of every block) against the oracle on
    the same positions; bandwidth-optimal results are identical on every rank."""
    P, n = 3, 2 ** 31 + 37
    # rows padded to a 16-byte multiple (rank buffers must be 16-byte aligned); the
    # Allreduce covers the first n elements of each row
    inp = gar_inputs.rank_inputs(P, (n + 3) // 4 * 4, "f32", ("normal", 0.0, 1.0), 31, device="cuda")
    idx = _sample_positions(n, P, S)
    sel = torch.from_numpy(idx).to("cuda")
    sub = inp[:, sel].cpu().numpy()
    buf = inp            # in place: the inputs at the sampled positions are kept in `sub`
    plan = gar.gar_plan_create(P, n, "f32", "sum", S)
    gar.ensure_workspace(plan)
    gar.gar_allreduce(plan, buf, mode)
    torch.cuda.synchronize()
    got = buf[:, sel].cpu().numpy()
    if S == 4:
        assert bool((buf[1, :n] == buf[0, :n]).all()) and bool((buf[2, :n] == buf[0, :n]).all())
    full = [np.zeros(n, np.float32) for _ in range(P)]
    for x in range(P):
        full[x][idx] = sub[x]
    want = G.allreduce(full, S, "sum", "f32", elements=idx)
    for x in range(P):
        np.testing.assert_array_equal(_bits(got[x]), _bits(want[x]), err_msg=f"rank {x}")
    del buf, inp
    torch.cuda.empty_cache()
