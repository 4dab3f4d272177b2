"""grid_advance_masks (the advance fed inside the mask step's first kernel)
equals grid_advance followed by grid_masks / grid_masks_apply: the same
configurations, masks and masked logits bit for bit, the advance's error as
the status of a row whose token was refused and the mask step's otherwise,
in place and out of place, and with audit on the same node hashes."""
import numpy as np
import pytest

from tests.harness import GpuRun, unpack
from workloads import configs

pytestmark = pytest.mark.gpu


def _tokens(wl, run, seed):
    """Per row: mostly an admitted token; every fifth row a refused one, every
    seventh an out-of-range id, and EOS where the gate admits it."""
    words, _ = run.masks()
    bits = unpack(words, run.V)
    rng = np.random.default_rng(seed)
    tok = np.zeros(run.B, np.int32)
    for b in range(run.B):
        adm = np.flatnonzero(bits[b])
        rej = np.flatnonzero(bits[b] == 0)
        if b % 7 == 6:
            tok[b] = run.V + 3
        elif b % 5 == 4 and rej.size:
            tok[b] = rng.choice(rej)
        elif adm.size and bits[b][wl["eos"]] and b % 3 == 0:
            tok[b] = wl["eos"]
        elif adm.size:
            tok[b] = rng.choice(adm)
        else:
            tok[b] = -1
    return tok


def _state(G, cfg, B):
    return [G.grid_configs_export(cfg.h, b) for b in range(B)]


@pytest.mark.parametrize("name,dtype", [("headline", "f32"), ("admin", "bf16"), ("admin", None),
                                        ("tiny", "f32")])
def test_fused_step_equals_advance_then_masks(name, dtype):
    import torch
    from paper_2607_11951_gb300 import grid as G
    wl = {"headline": lambda: configs.sql_select_only(prefix_seed=5003),
          "admin": lambda: configs.sql_admin(),
          "tiny": lambda: configs.tiny_expr(B=21)}[name]()
    run = GpuRun(wl)
    run.build_configs()
    B, V, W = run.B, run.V, run.W
    tok = torch.from_numpy(_tokens(wl, run, 11)).cuda()
    before = _state(G, run.cfg, B)
    tdt = {"f32": torch.float32, "bf16": torch.bfloat16, None: None}[dtype]
    base = torch.randn((B, V + 7), generator=torch.Generator().manual_seed(5)).to(tdt or torch.float32).cuda()
    out_a, out_b = G.Configs(run.spec, B), G.Configs(run.spec, B)
    mask_a = torch.zeros((B, W), dtype=torch.int32, device="cuda")
    mask_b = torch.full((B, W), -1, dtype=torch.int32, device="cuda")
    st_adv = torch.zeros(B, dtype=torch.int32, device="cuda")
    st_a = torch.zeros(B, dtype=torch.int32, device="cuda")
    st_b = torch.full((B,), 99, dtype=torch.int32, device="cuda")
    lg_a, lg_b = base.clone(), base.clone()
    G.grid_advance(run.spec.h, run.cfg.h, out_a.h, tok, st_adv)
    if dtype is None:
        G.grid_masks(run.spec.h, out_a.h, mask_a, st_a)
        G.grid_advance_masks(run.spec.h, run.cfg.h, out_b.h, tok, mask_b, st_b)
    else:
        G.grid_masks_apply(run.spec.h, out_a.h, mask_a, st_a, lg_a[:, :V])
        G.grid_advance_masks(run.spec.h, run.cfg.h, out_b.h, tok, mask_b, st_b, lg_b[:, :V])
    torch.cuda.synchronize()
    sa, sm, sb = st_adv.cpu().numpy(), st_a.cpu().numpy(), st_b.cpu().numpy()
    assert (mask_a.cpu().numpy() == mask_b.cpu().numpy()).all()
    assert (sb == np.where(sa != 0, sa, sm)).all(), (sa, sm, sb)
    assert (sa != 0).any() and (sa == 0).any()  # both kinds of rows are covered
    if dtype is not None:
        assert torch.equal(lg_a.view(torch.int16 if dtype == "bf16" else torch.int32),
                           lg_b.view(torch.int16 if dtype == "bf16" else torch.int32))
    assert _state(G, out_a, B) == _state(G, out_b, B)
    assert _state(G, run.cfg, B) == before  # out of place: the input is unchanged


def test_fused_step_in_place_over_several_steps():
    import torch
    from paper_2607_11951_gb300 import grid as G
    wl = configs.sql_admin()
    run_a, run_b = GpuRun(wl), GpuRun(wl)
    run_a.build_configs()
    run_b.build_configs()
    B = run_a.B
    st_a = torch.zeros(B, dtype=torch.int32, device="cuda")
    st_b = torch.zeros(B, dtype=torch.int32, device="cuda")
    for k in range(4):
        tok = torch.from_numpy(_tokens(wl, run_a, 20 + k)).cuda()
        G.grid_advance(run_a.spec.h, run_a.cfg.h, run_a.cfg.h, tok, st_a)
        G.grid_masks(run_a.spec.h, run_a.cfg.h, run_a.mask, run_a.status)
        G.grid_advance_masks(run_b.spec.h, run_b.cfg.h, run_b.cfg.h, tok, run_b.mask, st_b)
        torch.cuda.synchronize()
        assert (run_a.mask.cpu().numpy() == run_b.mask.cpu().numpy()).all(), k
        sa, sm, sb = st_a.cpu().numpy(), run_a.status.cpu().numpy(), st_b.cpu().numpy()
        assert (sb == np.where(sa != 0, sa, sm)).all(), k
        assert _state(G, run_a.cfg, B) == _state(G, run_b.cfg, B), k


def test_fused_step_matches_oracle_masks():
    """The fused step's masks of the advanced rows are the oracle's masks of
    prefix + token (rows whose token was refused: of the prefix)."""
    import torch
    from oracle import compile_grammar
    from paper_2607_11951_gb300 import grid as G
    wl = configs.tiny_expr(B=21)
    run = GpuRun(wl)
    run.build_configs()
    tok = _tokens(wl, run, 7)
    t = torch.from_numpy(tok).cuda()
    out, tmp = G.Configs(run.spec, run.B), G.Configs(run.spec, run.B)
    st = torch.zeros(run.B, dtype=torch.int32, device="cuda")
    sa = torch.zeros(run.B, dtype=torch.int32, device="cuda")
    G.grid_advance(run.spec.h, run.cfg.h, tmp.h, t, sa)  # which tokens the advance accepts
    G.grid_advance_masks(run.spec.h, run.cfg.h, out.h, t, run.mask, st)
    torch.cuda.synchronize()
    bits = unpack(run.mask.cpu().numpy().view(np.uint32), run.V)
    sa = sa.cpu().numpy()
    og = compile_grammar(wl["grammar"], wl["role"], wl["lexicons"])
    for b in range(run.B):
        ids = list(wl["prefixes"][b]) + ([int(tok[b])] if sa[b] == 0 and tok[b] >= 0 else [])
        cfg = og.config_from_ids(ids, wl["tokens"], wl["eos"], wl["specials"])
        if cfg is None or getattr(cfg, "complete", False):
            assert not bits[b].any(), b
            continue
        want = np.asarray(og.mask(cfg, wl["tokens"], wl["eos"], wl["specials"]), dtype=np.uint8)
        assert (bits[b] == want).all(), b


def test_fused_step_with_audit_keeps_node_hashes():
    import torch
    from paper_2607_11951_gb300 import grid as G
    wl = configs.tiny_expr(B=8)
    run_a, run_b = GpuRun(wl), GpuRun(wl)
    for r in (run_a, run_b):
        r.build_configs()
        G.grid_configs_enable_audit(r.spec.h, r.cfg.h)
    out_a, out_b = G.Configs(run_a.spec, run_a.B), G.Configs(run_b.spec, run_b.B)
    G.grid_configs_enable_audit(run_a.spec.h, out_a.h)
    G.grid_configs_enable_audit(run_b.spec.h, out_b.h)
    tok = torch.from_numpy(_tokens(wl, run_a, 3)).cuda()
    st = torch.zeros(run_a.B, dtype=torch.int32, device="cuda")
    G.grid_advance(run_a.spec.h, run_a.cfg.h, out_a.h, tok, st)
    G.grid_masks(run_a.spec.h, out_a.h, run_a.mask, run_a.status)
    G.grid_advance_masks(run_b.spec.h, run_b.cfg.h, out_b.h, tok, run_b.mask, st)
    nxt = torch.zeros(run_a.B, dtype=torch.int32, device="cuda")  # token 0 as the next record's token
    rec_a = torch.zeros((run_a.B, 80), dtype=torch.uint8, device="cuda")
    rec_b = torch.zeros((run_a.B, 80), dtype=torch.uint8, device="cuda")
    G.grid_audit_append(run_a.spec.h, out_a.h, run_a.mask, nxt, 0, rec_a)
    G.grid_audit_append(run_b.spec.h, out_b.h, run_b.mask, nxt, 0, rec_b)
    torch.cuda.synchronize()
    # the records carry the rolling hash of each row's stack: equal records,
    # equal node hashes
    assert torch.equal(rec_a, rec_b)


def test_fused_step_refuses_bad_arguments():
    """Mismatched batch sizes, a row stride below V and an unknown logits
    type are refused with an error before anything is enqueued."""
    import torch
    from paper_2607_11951_gb300 import grid as G
    wl = configs.tiny_expr(B=4)
    run = GpuRun(wl)
    run.build_configs()
    other = G.Configs(run.spec, 5)
    tok = torch.zeros(4, dtype=torch.int32, device="cuda")
    st = torch.zeros(4, dtype=torch.int32, device="cuda")
    with pytest.raises(G.GridError):
        G.grid_advance_masks(run.spec.h, run.cfg.h, other.h, tok, run.mask, st)
    lib = G.lib()
    logits = torch.zeros((4, run.V), device="cuda")
    out = G.Configs(run.spec, 4)
    rc = lib.grid_advance_masks(run.spec.h, run.cfg.h, out.h, None, G._ptr(tok), 1, G._ptr(run.mask), G._ptr(st),
                                G._ptr(logits), G.GRID_DTYPE_F32, run.V - 1, None)
    assert rc == -1  # GRID_E_INVALID_ARG
    rc = lib.grid_advance_masks(run.spec.h, run.cfg.h, out.h, None, G._ptr(tok), 1, G._ptr(run.mask), G._ptr(st),
                                G._ptr(logits), 7, run.V, None)
    assert rc == -1  # GRID_E_INVALID_ARG
    other_spec = G.Spec(run.grammar, run.vocab)  # a cache of another spec
    cache = G.Cache(other_spec, 64)
    with pytest.raises(G.GridError):
        G.grid_advance_masks(run.spec.h, run.cfg.h, out.h, tok, run.mask, st, cache=cache)
