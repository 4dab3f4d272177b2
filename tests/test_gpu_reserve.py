"""grid_reserve (Sec. 5 Prop. 9, Sec. 6.1 step 3) against the oracle: the
reserve of every row equals the oracle's, and the completion the GPU writes
is legal -- the oracle admits each of its tokens in turn and then EOS -- with
exactly that many tokens; the trigger fires where the budget is within the
reserve plus the safety margin."""
import numpy as np
import pytest

from tests.harness import GpuRun
from workloads import configs
from workloads.randgram import rand_grammar_workload

pytestmark = pytest.mark.gpu


def _cases():
    return {
        "tiny_expr": lambda: configs.tiny_expr(B=32),
        "tiny_pick": lambda: configs.tiny_pick(B=32),
        "sql_admin": lambda: configs.sql_admin(B=8),
        "sql_shared": lambda: configs.sql_shared(B=8),
        "sweep_deep": lambda: configs.sql_sweep_cell(100, 32),
        "forced_sql": configs.forced_sql,
        # random statement grammars: keyword-led statements, lists, optional
        # clauses, calls, nested blocks, identifier categories
        **{"rand_%d" % k: (lambda k=k: rand_grammar_workload(k, B=16, V=1500)) for k in (0, 1, 6, 8, 14)},
    }


@pytest.mark.parametrize("name", list(_cases()))
def test_reserve_parity(name):
    import torch
    from oracle import compile_grammar
    from oracle.reserve import Reserve
    from paper_2607_11951_gb300 import grid as G
    wl = _cases()[name]()
    if name == "sweep_deep":
        wl = dict(wl)
        wl["prefixes"] = wl["prefixes"][:6]
    run = GpuRun(wl)
    assert (run.build_configs() == 0).all()
    B, cap = run.B, 512
    cost = torch.zeros(B, dtype=torch.int32, device="cuda")
    toks = torch.zeros((B, cap), dtype=torch.int32, device="cuda")
    st = torch.zeros(B, dtype=torch.int32, device="cuda")
    budget = torch.arange(B, dtype=torch.int32, device="cuda")
    fire = torch.zeros(B, dtype=torch.int32, device="cuda")
    G.grid_reserve(run.spec.h, run.cfg.h, cost, toks, st, budget, 2, fire)
    torch.cuda.synchronize()
    cost, toks, st, fire = cost.cpu().numpy(), toks.cpu().numpy(), st.cpu().numpy(), fire.cpu().numpy()
    og = compile_grammar(wl["grammar"], wl["role"], wl["lexicons"])
    R = Reserve(og, wl["tokens"], wl["eos"], wl["specials"])
    longest = 0
    for b, pre in enumerate(wl["prefixes"]):
        cfg = og.config_from_ids(pre, wl["tokens"], wl["eos"], wl["specials"])
        want = R.reserve(cfg)
        if want is None:  # no completion under the cost model (e.g. no token spells a blank)
            assert st[b] == G.GRID_ST_NONVIABLE and cost[b] == -1 and (toks[b] == -1).all() and fire[b] == 0
            continue
        assert st[b] == 0 and cost[b] == want, (b, cost[b], want, st[b])
        seq = [int(x) for x in toks[b] if x >= 0]
        assert len(seq) == want and (toks[b][len(seq):] == -1).all()
        assert seq[-1] == wl["eos"]
        c = cfg
        for t in seq:
            c = og.advance(c, t, wl["tokens"], wl["eos"], wl["specials"])
            assert c is not None, (b, t)
        assert c.complete
        assert fire[b] == (1 if b <= want + 2 else 0)
        longest = max(longest, want)
    if name == "sweep_deep":
        assert longest > 20
