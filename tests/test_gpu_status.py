"""Per-row status codes of the CUDA path on inputs that reach them (device
status array, no trap): a stack that would exceed max_depth, a token whose
walk needs more overlay entries than a lane holds, a viable row whose mask is
empty because the vocabulary is not byte-complete.  Each affected row keeps
its configuration as of its last accepted token; the other rows are
unaffected and still match the oracle bit for bit."""
import numpy as np
import pytest

from tests.harness import GpuRun, unpack
from workloads import grammar_text

pytestmark = pytest.mark.gpu

ALPHA = b"abcdefghijklmnopqrstuvwxyz0123456789+*() "


def _expr_wl(tokens, prefixes, max_depth=4096):
    toks = list(tokens) + [b"<eos>"]
    return dict(name="status", grammar=grammar_text("expr"), role=None, lexicons={}, tokens=toks,
                eos=len(toks) - 1, specials=[], prefixes=prefixes, max_depth=max_depth)


def _oracle():
    from oracle import compile_grammar
    return compile_grammar(grammar_text("expr"))


def test_stack_overflow_keeps_last_configuration():
    """max_depth = 8: row 0 feeds twelve '(' tokens; the push past depth 8 is
    GRID_ST_STACK_OVERFLOW and the row keeps the configuration after the
    last token that fit, which the oracle reaches with the same tokens; row
    1 stays within the bound."""
    import torch
    from paper_2607_11951_gb300 import grid as G
    toks = [bytes([c]) for c in ALPHA]
    lp = toks.index(b"(")
    wl = _expr_wl(toks, [[lp] * 12, [toks.index(b"a"), toks.index(b"+"), toks.index(b"1")]], max_depth=8)
    run = GpuRun(wl)
    st = run.build_configs()
    assert st.tolist() == [G.GRID_ST_STACK_OVERFLOW, G.GRID_ST_OK]
    og = _oracle()
    # the longest prefix of '(' tokens whose stack fits in 8 states
    k, cfg = 0, og.start_config()
    while True:
        nxt = og.advance(cfg, lp, wl["tokens"], wl["eos"])
        assert nxt is not None
        if len(og.stack_list(nxt)) > 8:
            break
        k, cfg = k + 1, nxt
    assert 0 < k < 12
    row = run.cfg.export(0)
    assert row["depth"] == len(og.stack_list(cfg))
    # its mask is the oracle's at that configuration; row 1 as usual
    words, status = run.masks()
    assert status.tolist() == [0, 0]
    bits = unpack(words, run.V)
    want0 = og.mask(cfg, wl["tokens"], wl["eos"])
    want1 = og.mask(og.config_from_ids(wl["prefixes"][1], wl["tokens"], wl["eos"]), wl["tokens"], wl["eos"])
    assert (bits[0] == np.asarray(want0, np.uint8)).all()
    assert (bits[1] == np.asarray(want1, np.uint8)).all()


def test_overlay_bound_in_walk_and_advance():
    """A 40-byte token of '(' needs 40 pushes in one walk, more than the 32
    overlay entries a walk lane holds: the mask step sets GRID_ST_BOUND on
    that row (and leaves the token's bit 0; the oracle, which has no bound,
    admits it) while every other bit matches the oracle.  A 60-byte token
    exceeds the advance's 48 entries: GRID_ST_BOUND, configuration kept."""
    import torch
    from paper_2607_11951_gb300 import grid as G
    toks = [bytes([c]) for c in ALPHA] + [b"(" * 40, b"(" * 60]
    t40, t60 = len(toks) - 2, len(toks) - 1
    a = toks.index(b"a")
    wl = _expr_wl(toks, [[], [a]])
    run = GpuRun(wl)
    assert (run.build_configs() == 0).all()
    words, status = run.masks()
    assert status.tolist() == [G.GRID_ST_BOUND, G.GRID_ST_OK]
    bits = unpack(words, run.V)
    og = _oracle()
    for r in range(2):
        cfg = og.config_from_ids(wl["prefixes"][r], wl["tokens"], wl["eos"])
        want = np.asarray(og.mask(cfg, wl["tokens"], wl["eos"]), np.uint8)
        if r == 0:
            assert want[t40] == 1 and want[t60] == 1 and bits[0][t40] == 0
            keep = np.ones(run.V, bool)
            keep[[t40, t60]] = False
            assert (bits[0][keep] == want[keep]).all()
        else:
            assert (bits[1] == want).all()
    before = run.cfg.export(0)
    toks_d = torch.tensor([t60, -1], dtype=torch.int32, device="cuda")
    st = torch.zeros(2, dtype=torch.int32, device="cuda")
    G.grid_advance(run.spec.h, run.cfg.h, run.cfg.h, toks_d, st)
    torch.cuda.synchronize()
    assert st.cpu().tolist() == [G.GRID_ST_BOUND, G.GRID_ST_OK]
    assert run.cfg.export(0) == before


def test_empty_mask_without_byte_complete_vocabulary():
    """Prop. 8 needs a byte-complete vocabulary.  With only '+' and EOS, the
    start configuration is viable but no token continues it: the mask step
    reports GRID_ST_EMPTY_MASK and writes an all-zero mask; a row where '+'
    fits is unaffected."""
    from paper_2607_11951_gb300 import grid as G
    wl = _expr_wl([b"+", b"a"], [[], [1]])
    run = GpuRun(wl)
    assert run.vocab.info()["byte_complete"] == 0
    assert (run.build_configs() == 0).all()
    words, status = run.masks()
    bits = unpack(words, run.V)
    # row 0: "" -> "+" rejected, "a" admitted: not empty; use a prefix "a+"
    # instead for the empty case below
    assert status.tolist() == [0, 0]
    wl2 = _expr_wl([b"+"], [[]])
    run2 = GpuRun(wl2)
    assert (run2.build_configs() == 0).all()
    words2, status2 = run2.masks()
    assert status2.tolist() == [G.GRID_ST_EMPTY_MASK]
    assert (words2 == 0).all()
    og = _oracle()
    want = og.mask(og.start_config(), wl2["tokens"], wl2["eos"])
    assert sum(want) == 0
    for r in range(2):
        cfg = og.config_from_ids(wl["prefixes"][r], wl["tokens"], wl["eos"])
        assert (bits[r] == np.asarray(og.mask(cfg, wl["tokens"], wl["eos"]), np.uint8)).all()
