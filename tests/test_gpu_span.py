"""grid_forced_span (Sec. 6.1 step 6, jump-forward) against the oracle: the
forced ids of every row, the span lengths, and the mask and status of each
row's final configuration, bit for bit."""
import numpy as np
import pytest

from tests.harness import GpuRun, unpack
from workloads import configs

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name", ["forced_pick", "forced_sql"])
@pytest.mark.parametrize("max_span", [0, 1, 16])
def test_forced_span_parity(name, max_span):
    import torch
    from oracle import compile_grammar
    from paper_2607_11951_gb300 import grid as G
    wl = getattr(configs, name)()
    run = GpuRun(wl)
    assert (run.build_configs() == 0).all()
    B, toks, eos = run.B, wl["tokens"], wl["eos"]
    span = torch.full((B, max(max_span, 1)), 7, dtype=torch.int32, device="cuda")[:, :max_span].contiguous()
    span_len = torch.full((B,), 7, dtype=torch.int32, device="cuda")
    G.grid_forced_span(run.spec.h, run.cfg.h, max_span, run.mask, span, span_len, run.status)
    torch.cuda.synchronize()
    got_span, got_len = span.cpu().numpy(), span_len.cpu().numpy()
    bits = unpack(run.mask.cpu().numpy().view(np.uint32), run.V)
    status = run.status.cpu().numpy()
    og = compile_grammar(wl["grammar"], wl["role"], wl["lexicons"])
    total = 0
    for b, pre in enumerate(wl["prefixes"]):
        cfg = og.config_from_ids(pre, toks, eos)
        want, end = og.forced_span(cfg, toks, eos, max_span=max_span)
        assert got_len[b] == len(want), (b, got_len[b], want)
        assert list(got_span[b][:len(want)]) == want
        assert (got_span[b][len(want):] == -1).all()
        total += len(want)
        if end.complete:
            assert status[b] == G.GRID_ST_COMPLETE and bits[b].sum() == 0
        else:
            assert status[b] == 0
            assert (bits[b] == np.asarray(og.mask(end, toks, eos), np.uint8)).all(), b
    if max_span >= 16:
        assert total >= 3
    # the configurations were advanced in place: a plain mask step agrees
    words, st = run.masks()
    assert (unpack(words, run.V) == bits).all() and (st == status).all()
