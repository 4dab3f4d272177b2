"""GPU test of grid_masks_static, the mask entry point that allocates nothing.

Callers that cannot allocate device memory when they need a mask (a serving
engine whose pool has reserved the device up front, or one that cannot afford
the synchronization of freeing memory mid-step) keep their parser
configurations in device memory they own and pass them in as plain arrays; the
step's scratch is the library's fixed static device area.  This file checks,
through the C ABI, that two calls in a row give exactly the masks and status
codes of grid_masks on the same configurations (the second call sees the
first call's leftovers in the shared area), and that a batch too large for the
area is refused before anything runs.  It is collected last so that a run
stopping at the first failure has run every other test.
"""
import numpy as np
import pytest

from tests.harness import GpuRun, unpack
from workloads import configs

pytestmark = pytest.mark.gpu

MAX_DEPTH = 4096  # grid_compile's default stack capacity, which GpuRun uses
GRID_E_TOO_LARGE = -8


def _torch():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    return torch


def _state_arrays(run, torch):
    """Copy every row of run.cfg into caller-owned device arrays."""
    B = run.B
    stack = np.zeros((B, MAX_DEPTH), np.uint16)
    depth = np.zeros(B, np.int32)
    q = np.zeros(B, np.int32)
    lx = np.zeros(B, np.int32)
    fl = np.zeros(B, np.int32)
    for b in range(B):
        e = run.cfg.export(b)
        assert e["depth"] <= MAX_DEPTH
        stack[b, :e["depth"]] = e["stack"]
        depth[b], q[b], lx[b], fl[b] = e["depth"], e["dfa_state"], e["lex_node"], e["flags"]
    to = lambda a: torch.from_numpy(a).to(run.dev)
    return [to(stack.view(np.int16)), to(depth), to(q), to(lx), to(fl)]


def _masks_static(run, torch, arrays):
    from paper_2607_11951_gb300 import grid as G
    mask = torch.full_like(run.mask, -1)  # every word must be written by the call
    status = torch.full_like(run.status, -99)
    G.grid_masks_static(run.spec.h, *arrays, mask, status)
    torch.cuda.synchronize()
    return mask.cpu().numpy().view(np.uint32), status.cpu().numpy()


def test_masks_static_matches_grid_masks_twice():
    torch = _torch()
    from paper_2607_11951_gb300 import grid as G
    run = GpuRun(configs.sql_admin())
    st = run.build_configs()
    assert (st == 0).all(), st

    # call 1: the prefixes' configurations
    ref_w, ref_s = run.masks()
    w1, s1 = _masks_static(run, torch, _state_arrays(run, torch))
    np.testing.assert_array_equal(s1, ref_s)
    np.testing.assert_array_equal(w1, ref_w)

    # call 2, right after: every row advanced by one admitted token
    bits = unpack(ref_w, run.V)
    rng = np.random.default_rng(77)
    tok = np.full(run.B, -1, np.int32)
    for b in range(run.B):
        ids = np.flatnonzero(bits[b])
        if len(ids):
            tok[b] = int(rng.choice(ids))
    G.grid_advance(run.spec.h, run.cfg.h, run.cfg.h, torch.from_numpy(tok).to(run.dev), run.status)
    torch.cuda.synchronize()
    st2 = run.status.cpu().numpy()
    assert set(st2.tolist()) <= {G.GRID_ST_OK, G.GRID_ST_COMPLETE}, st2
    ref_w2, ref_s2 = run.masks()
    assert not np.array_equal(ref_w2, ref_w)
    w2, s2 = _masks_static(run, torch, _state_arrays(run, torch))
    np.testing.assert_array_equal(s2, ref_s2)
    np.testing.assert_array_equal(w2, ref_w2)


def test_masks_static_refuses_batch_beyond_area():
    torch = _torch()
    from paper_2607_11951_gb300 import grid as G
    run = GpuRun(configs.sql_admin(B=2))
    # 2048 rows need two verdict bitmaps of ceil(NS/32)+1 words each per row:
    # about 16 MB for this vocabulary, twice the 8 MiB area
    B = 2048
    dev = run.dev
    stack = torch.zeros((B, MAX_DEPTH), dtype=torch.int16, device=dev)
    depth = torch.ones(B, dtype=torch.int32, device=dev)
    q = torch.ones(B, dtype=torch.int32, device=dev)  # the lexer's start state
    lx = torch.zeros(B, dtype=torch.int32, device=dev)
    fl = torch.zeros(B, dtype=torch.int32, device=dev)
    mask = torch.full((B, run.W), 7, dtype=torch.int32, device=dev)
    status = torch.full((B,), -99, dtype=torch.int32, device=dev)
    with pytest.raises(G.GridError) as ei:
        G.grid_masks_static(run.spec.h, stack, depth, q, lx, fl, mask, status)
    assert ei.value.code == GRID_E_TOO_LARGE
    assert "static area" in str(ei.value)
    torch.cuda.synchronize()
    assert bool((mask == 7).all()) and bool((status == -99).all())
    # and the area still serves a batch that fits
    st = run.build_configs()
    assert (st == 0).all()
    ref_w, ref_s = run.masks()
    w, s = _masks_static(run, torch, _state_arrays(run, torch))
    np.testing.assert_array_equal(s, ref_s)
    np.testing.assert_array_equal(w, ref_w)


def test_masks_static_headline_and_capacity_boundary():
    """At the headline vocabulary (V = 151,936) the static call matches
    grid_masks on the 32 headline rows; the largest batch the area holds
    (found by the refusals themselves) runs and matches grid_masks, and one
    row more is refused."""
    torch = _torch()
    from paper_2607_11951_gb300 import grid as G
    run = GpuRun(configs.sql_select_only())
    assert (run.build_configs() == 0).all()
    ref_w, ref_s = run.masks()
    w, s = _masks_static(run, torch, _state_arrays(run, torch))
    np.testing.assert_array_equal(s, ref_s)
    np.testing.assert_array_equal(w, ref_w)

    dev = run.dev

    def start_rows(B):
        return [torch.zeros((B, MAX_DEPTH), dtype=torch.int16, device=dev),
                torch.ones(B, dtype=torch.int32, device=dev), torch.ones(B, dtype=torch.int32, device=dev),
                torch.zeros(B, dtype=torch.int32, device=dev), torch.zeros(B, dtype=torch.int32, device=dev)]

    def fits(B):
        mask = torch.zeros((B, run.W), dtype=torch.int32, device=dev)
        status = torch.zeros(B, dtype=torch.int32, device=dev)
        try:
            G.grid_masks_static(run.spec.h, *start_rows(B), mask, status)
        except G.GridError as e:
            assert e.code == GRID_E_TOO_LARGE
            return None
        torch.cuda.synchronize()
        return mask.cpu().numpy().view(np.uint32), status.cpu().numpy()

    lo, hi = 1, 4096
    assert fits(lo) is not None and fits(hi) is None
    while hi - lo > 1:
        mid = (lo + hi) // 2
        if fits(mid) is None:
            hi = mid
        else:
            lo = mid
    assert 8 <= lo < 4096
    w, s = fits(lo)
    assert fits(lo + 1) is None
    ref = G.Configs(run.spec, lo)  # every row at the start configuration
    m = torch.zeros((lo, run.W), dtype=torch.int32, device=dev)
    st = torch.zeros(lo, dtype=torch.int32, device=dev)
    G.grid_masks(run.spec.h, ref.h, m, st)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(w, m.cpu().numpy().view(np.uint32))
    np.testing.assert_array_equal(s, st.cpu().numpy())
