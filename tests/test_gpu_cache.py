"""The configuration-keyed mask cache (Sec. 4.3, Prop. OBL-KEY1): cache-on
equals cache-off, bit for bit, over randomized replays -- the same
configurations masked through a cache that fills on first sight of a key and
is read on every later step, rows sharing keys within a batch and across
steps, identifier and generic positions -- for masks, statuses and the fused
logits fill; and the cache is really used (hits)."""
import numpy as np
import pytest

from tests.harness import GpuRun, unpack
from workloads import configs
from workloads.randgram import rand_grammar_workload

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name", ["tiny_expr", "sql_admin", "sql_select_only", "sql_shared", "rand_2", "rand_6"])
def test_cache_on_equals_cache_off_over_replays(name):
    import torch
    from paper_2607_11951_gb300 import grid as G
    if name.startswith("rand_"):  # random statement grammars with identifier categories
        wl = rand_grammar_workload(int(name[5:]), B=32, V=3000)
    else:
        wl = getattr(configs, name)()
    run = GpuRun(wl)
    assert (run.build_configs() == 0).all()
    cache = G.Cache(run.spec, 256)
    B, V = run.B, run.V
    rng = np.random.default_rng(17)
    m_on = torch.zeros_like(run.mask)
    st_on = torch.zeros_like(run.status)
    for step in range(5):
        for rep in range(2):  # the second pass meets every key of the batch again
            words, status = run.masks()
            G.grid_masks_cached(run.spec, run.cfg, cache, m_on, st_on)
            torch.cuda.synchronize()
            assert (m_on.cpu().numpy().view(np.uint32) == words).all(), (name, step, rep)
            assert (st_on.cpu().numpy() == status).all()
        bits = unpack(words, V)
        tok = np.full(B, -1, np.int32)
        for b in range(B):
            if status[b] == 0:
                adm = np.flatnonzero(bits[b])
                adm = adm[adm != wl["eos"]] if adm.size > 1 else adm
                tok[b] = int(rng.choice(adm))
        G.grid_advance(run.spec.h, run.cfg.h, run.cfg.h, torch.from_numpy(tok).cuda(), run.status)
        torch.cuda.synchronize()
    st = cache.stats()
    assert st["hits"] >= (B if not name.startswith("rand_") else 1) and st["ready"] > 0, st


def test_cache_fused_logits_and_clear():
    import torch
    from paper_2607_11951_gb300 import grid as G
    wl = configs.sql_select_only()
    run = GpuRun(wl)
    assert (run.build_configs() == 0).all()
    cache = G.Cache(run.spec, 1024)
    lg = torch.from_numpy(configs.logits(3, run.B, run.V)).cuda()
    for rep in range(3):
        a, b = lg.clone(), lg.clone()
        m1, s1 = torch.zeros_like(run.mask), torch.zeros_like(run.status)
        m2, s2 = torch.zeros_like(run.mask), torch.zeros_like(run.status)
        G.grid_masks_apply(run.spec.h, run.cfg.h, m1, s1, a)
        G.grid_masks_cached(run.spec, run.cfg, cache, m2, s2, b)
        torch.cuda.synchronize()
        assert torch.equal(m1, m2) and torch.equal(s1, s2) and torch.equal(a.view(torch.int32), b.view(torch.int32))
        if rep == 1:
            assert cache.stats()["hits"] > 0
            cache.clear()
            torch.cuda.synchronize()
            assert cache.stats() == {"lookups": 0, "hits": 0, "fills": 0, "ready": 0}


@pytest.mark.parametrize("name", ["sql_admin", "sql_select_only"])
def test_cache_on_equals_cache_off_in_the_fused_step(name):
    """The fused decoding step (grid_advance_masks) through a cache equals it
    without one, over replays of several steps in place: masks, statuses,
    configurations and the fp32 fill bit for bit, with hits from the second
    step on."""
    import torch
    from paper_2607_11951_gb300 import grid as G
    wl = getattr(configs, name)()
    run_a, run_b = GpuRun(wl), GpuRun(wl)
    assert (run_a.build_configs() == 0).all() and (run_b.build_configs() == 0).all()
    cache = G.Cache(run_b.spec, 1024)
    B, V = run_a.B, run_a.V
    rng = np.random.default_rng(23)
    words, _ = run_a.masks()
    for step in range(4):
        bits = unpack(words, V)
        tok = np.array([rng.choice(np.flatnonzero(bits[b])) if bits[b].any() else -1 for b in range(B)], np.int32)
        t = torch.from_numpy(tok).cuda()
        lg = torch.from_numpy(configs.logits(40 + step, B, V)).cuda()
        la, lb = lg.clone(), lg.clone()
        st_a = torch.zeros(B, dtype=torch.int32, device="cuda")
        st_b = torch.zeros(B, dtype=torch.int32, device="cuda")
        G.grid_advance_masks(run_a.spec.h, run_a.cfg.h, run_a.cfg.h, t, run_a.mask, st_a, la)
        G.grid_advance_masks(run_b.spec.h, run_b.cfg.h, run_b.cfg.h, t, run_b.mask, st_b, lb, cache=cache)
        torch.cuda.synchronize()
        assert torch.equal(run_a.mask, run_b.mask) and torch.equal(st_a, st_b), (name, step)
        assert torch.equal(la.view(torch.int32), lb.view(torch.int32)), (name, step)
        assert [G.grid_configs_export(run_a.cfg.h, b) for b in range(0, B, 5)] == \
               [G.grid_configs_export(run_b.cfg.h, b) for b in range(0, B, 5)]
        words = run_a.mask.cpu().numpy().view(np.uint32)
    assert cache.stats()["hits"] > 0
