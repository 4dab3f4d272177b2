"""Randomized full-vocabulary parity: random grammars of the statement family
(``workloads/randgram.py``: keyword-led statements, comma lists, optional
clauses, a precedence ladder with unary operators, calls, nested blocks, role
tags, identifier categories sharing one regex), each with its own vocabulary
of single bytes, random strings and sentence pieces that cross lexeme
boundaries, and prefixes cut at random byte offsets of random sentences.

Per grammar: the masks of every row equal the oracle's bit for bit (Def. 4,
EOS gate of Sec. 3.2), and one decoding step (``grid_advance_masks``, a random
admitted token per row) gives the oracle's masks of prefix + token, with
COMPLETE and an empty mask for rows fed EOS."""
import numpy as np
import pytest

from tests.harness import GpuRun, oracle_masks, unpack
from workloads.randgram import rand_grammar_workload

pytestmark = pytest.mark.gpu

# (seed, role): plain grammars, both identifier categories (a shared word read
# as TA), the column category alone, role-tagged statements kept or dropped
CASES = [(0, None), (1, None), (2, None), (5, []), (6, None), (6, []), (8, None), (11, []), (14, None),
         (17, None), (19, None), (22, None)]


def _compare(wl, bits, rows, want):
    for k, r in enumerate(rows):
        assert want[k] is not None, ("oracle rejects prefix", r)
        w = np.asarray(want[k], dtype=np.uint8)
        diff = np.nonzero(bits[r] != w)[0]
        assert diff.size == 0, ("row", r, "ids", diff[:10].tolist(), [wl["tokens"][i] for i in diff[:5]],
                                "gpu", bits[r][diff[:5]].tolist())


@pytest.mark.parametrize("seed,role", CASES)
def test_random_grammar_full_parity_and_step(seed, role):
    import torch
    from paper_2607_11951_gb300 import grid as G
    wl = rand_grammar_workload(seed, B=32, V=3000, role=role)
    run = GpuRun(wl)
    st = run.build_configs()
    assert (st == 0).all(), ("grid_advance status", st)
    words, status = run.masks()
    assert (status == 0).all(), ("grid_masks status", status)
    bits = unpack(words, run.V)
    _compare(wl, bits, range(run.B), oracle_masks(wl))
    assert bits[:, wl["eos"]].sum() >= 2  # whole sentences admit EOS

    # one decoding step with a random admitted token per row
    rng = np.random.default_rng(seed + 1)
    tok = np.array([rng.choice(np.flatnonzero(bits[b])) for b in range(run.B)], np.int32)
    tok[np.flatnonzero(bits[:, wl["eos"]])[0]] = wl["eos"]  # one row completes
    out = G.Configs(run.spec, run.B)
    mask = torch.zeros((run.B, run.W), dtype=torch.int32, device="cuda")
    st2 = torch.full((run.B,), 99, dtype=torch.int32, device="cuda")
    G.grid_advance_masks(run.spec.h, run.cfg.h, out.h, torch.from_numpy(tok).cuda(), mask, st2)
    torch.cuda.synchronize()
    st2 = st2.cpu().numpy()
    b2 = unpack(mask.cpu().numpy().view(np.uint32), run.V)
    is_eos = tok == wl["eos"]
    assert (st2[is_eos] == G.GRID_ST_COMPLETE).all() and not b2[is_eos].any()
    assert (st2[~is_eos] == 0).all(), st2
    rows = [b for b in range(run.B) if not is_eos[b]]
    w2 = dict(wl)
    w2["prefixes"] = [list(wl["prefixes"][b]) + [int(tok[b])] for b in range(run.B)]
    _compare(w2, b2, rows, oracle_masks(w2, rows))


@pytest.mark.parametrize("seed", range(24, 72))
def test_random_grammar_sweep_full_parity(seed):
    """Forty-eight more random grammars, smaller (16 rows, V = 1,500), masks
    only; odd seeds with the role-tagged statements dropped."""
    wl = rand_grammar_workload(seed, B=16, V=1500, role=[] if seed % 2 else None)
    run = GpuRun(wl)
    st = run.build_configs()
    assert (st == 0).all(), ("grid_advance status", st)
    words, status = run.masks()
    assert (status == 0).all(), ("grid_masks status", status)
    _compare(wl, unpack(words, run.V), range(run.B), oracle_masks(wl, procs=1))


@pytest.mark.parametrize("seed", [1, 6, 14])
def test_random_grammar_fused_fill_and_static_path(seed):
    """On random grammars: the masks with the fused -inf fill (fp32 and bf16)
    equal the masks followed by grid_apply_mask, bit for bit, and the
    allocation-free entry point gives grid_masks' masks and statuses."""
    import torch
    from paper_2607_11951_gb300 import grid as G
    from workloads import configs
    from tests.test_zz_no_alloc import _masks_static, _state_arrays
    wl = rand_grammar_workload(seed, B=32, V=3000)
    run = GpuRun(wl)
    assert (run.build_configs() == 0).all()
    words, status = run.masks()
    for dt in (torch.float32, torch.bfloat16):
        base = torch.from_numpy(configs.logits(seed, run.B, run.V)).to(dt).cuda()
        la, lb = base.clone(), base.clone()
        mask = torch.zeros_like(run.mask)
        st = torch.zeros_like(run.status)
        G.grid_masks_apply(run.spec.h, run.cfg.h, mask, st, la)
        G.grid_apply_mask(run.mask, lb)
        torch.cuda.synchronize()
        assert (mask.cpu().numpy().view(np.uint32) == words).all() and (st.cpu().numpy() == status).all()
        iv = torch.int32 if dt == torch.float32 else torch.int16
        assert torch.equal(la.view(iv), lb.view(iv)), dt
    w2, s2 = _masks_static(run, torch, _state_arrays(run, torch))
    np.testing.assert_array_equal(w2, words)
    np.testing.assert_array_equal(s2, status)
