"""CUDA path vs oracle, bit-exact (Def. 4 masks, EOS gate, masked logits).

Every test calls the library through the C ABI binding on the same seeded
inputs as the oracle.  Masks are integer results: the bar is bit equality.
"""
import numpy as np
import pytest

from tests.harness import GpuRun, oracle_masks, oracle_masks_split, unpack
from workloads import configs

pytestmark = pytest.mark.gpu

_runs = {}


def _run(name, fn):
    if name not in _runs:
        wl = fn()
        run = GpuRun(wl)
        st = run.build_configs()
        assert (st == 0).all(), ("grid_advance status", st)
        _runs[name] = (wl, run)
    return _runs[name]


def _compare_full(wl, run, rows=None, split=False):
    words, status = run.masks()
    assert (status == 0).all(), ("grid_masks status", status)
    bits = unpack(words, run.V)
    rows = list(range(run.B)) if rows is None else rows
    want = oracle_masks_split(wl, rows) if split else oracle_masks(wl, rows)
    for k, r in enumerate(rows):
        assert want[k] is not None, ("oracle rejects prefix", r)
        w = np.asarray(want[k], dtype=np.uint8)
        diff = np.nonzero(bits[r] != w)[0]
        assert diff.size == 0, ("row", r, "ids", diff[:10].tolist(),
                                [wl["tokens"][i] for i in diff[:5]], "gpu", bits[r][diff[:5]].tolist())
    # padding bits beyond V are zero
    W = words.shape[1]
    if W * 32 > run.V:
        pad = words[:, -1] >> np.uint32(run.V - (W - 1) * 32)
        assert (pad == 0).all()
    return bits


def _doubled(wl):
    """The workload with a second id for every spelling: ids V..2V-1 repeat ids
    0..V-1 as ordinary tokens (the copies of EOS and the specials included),
    so that every spelling of the original vocabulary has an alias."""
    w = dict(wl)
    w["tokens"] = list(wl["tokens"]) + list(wl["tokens"])
    return w


@pytest.mark.parametrize("name", ["tiny", "admin"])
def test_alias_ids_share_verdicts(name):
    # alias ids (several ids, one spelling) share one verdict, whichever way
    # the spelling is decided: a CI class, a verdict class, or a byte walk,
    # whose verdict the walk sets for every id of the spelling
    wl0 = configs.tiny_expr(B=16) if name == "tiny" else configs.sql_admin(B=8)
    wl = _doubled(wl0)
    run = GpuRun(wl)
    st = run.build_configs()
    assert (st == 0).all(), ("grid_advance status", st)
    bits = _compare_full(wl, run, split=(name == "admin"))
    V0 = len(wl0["tokens"])
    own = np.ones(V0, dtype=bool)
    own[[wl0["eos"]] + list(wl0["specials"])] = False
    np.testing.assert_array_equal(bits[:, :V0][:, own], bits[:, V0:][:, own])


def test_tiny_expr_full_parity():
    wl, run = _run("tiny", configs.tiny_expr)
    _compare_full(wl, run)


def test_sql_admin_full_parity():
    wl, run = _run("admin", configs.sql_admin)
    _compare_full(wl, run, split=True)


def test_sql_select_only_full_parity():
    wl, run = _run("headline", configs.sql_select_only)
    bits = _compare_full(wl, run, split=True)
    # the headline batch is not degenerate: every row admits something, EOS never
    assert bits.sum(axis=1).min() > 0


def test_tiny_pick_full_parity():
    """Pick grammar: a word of both lexicons where both identifier categories
    are parser-viable is read as the earlier-declared TABLE_NAME."""
    wl, run = _run("pick", configs.tiny_pick)
    _compare_full(wl, run)


def test_sql_shared_words_full_parity():
    """SQL admin workload whose schema shares words between tables and
    columns; a quarter of the rows end with such a word where a column may
    stand, so the pending lexeme has two parser-viable candidates."""
    wl, run = _run("shared", configs.sql_shared)
    bits = _compare_full(wl, run, split=True)
    # the priority is observable on these rows: "," after the shared word
    # is rejected (it was read as a table name, which needs "."), "." admitted
    comma, dot = wl["tokens"].index(b","), wl["tokens"].index(b".")
    tail = range(run.B - run.B // 4, run.B)
    assert all(bits[r][comma] == 0 and bits[r][dot] == 1 for r in tail)


SWEEP_N, SWEEP_D = (100, 1000, 4000, 16000), (1, 8, 32, 64)


def test_sweep_cells_full_parity():
    """Flatness sweep at full size: all 16 cells (n x depth) x 32 rows, every
    row's full V = 128,256 mask against the oracle."""
    from tests.harness import oracle_masks
    cells = [(n, d) for d in SWEEP_D for n in SWEEP_N]
    first = configs.sql_sweep_cell(*cells[0])
    run = GpuRun(first)
    merged = dict(first)
    merged["prefixes"] = []
    gpu_bits = []
    for n, d in cells:
        wl = configs.sql_sweep_cell(n, d)
        assert wl["tokens"] is first["tokens"] and wl["lexicons"] == first["lexicons"]
        st = run.build_configs(prefixes=wl["prefixes"])
        assert (st == 0).all(), (n, d, st)
        words, status = run.masks()
        assert (status == 0).all(), (n, d, status)
        gpu_bits.append(unpack(words, run.V))
        merged["prefixes"] += list(wl["prefixes"])
    want = oracle_masks(merged)
    for c, (n, d) in enumerate(cells):
        for r in range(run.B):
            w = want[c * run.B + r]
            assert w is not None, (n, d, r)
            diff = np.nonzero(gpu_bits[c][r] != np.asarray(w, dtype=np.uint8))[0]
            assert diff.size == 0, (n, d, r, diff[:10].tolist())


def test_cold_schema_full_parity():
    """Cold-schema workload (B=256, 50k identifiers): every row's full mask."""
    wl, run = _run("cold", configs.sql_cold_schema)
    _compare_full(wl, run)


@pytest.mark.parametrize("n_cat,n_kw,ci_on,in_codes", [(10, 9, 0, 1), (9, 21, 1, 0)])
def test_manycat_code_space_edges_full_parity(n_cat, n_kw, ci_on, in_codes):
    """The two edges of the 16-bit class-code space.  Ten categories over 36
    lexer states: 2 x 36 x 2^10 class ids do not fit, CI classes are off and
    every spelling of every row is decided by a walk.  Nine categories over
    63 lexer states: the 64,512 class ids fit but the largest table's verdict
    classes do not fit beside them, so the packing reads each verdict-class
    id's index from the per-id table.  Both bit-exact against the oracle on
    every row, and the fused decoding step equal to the two calls."""
    import torch
    from paper_2607_11951_gb300 import grid as G
    wl, run = _run("manycat%d" % n_cat, lambda: configs.manycat(n_cat, n_kw))
    info = run.spec.info()
    assert info["ci_on"] == ci_on and info["vc_in_codes"] == in_codes, info
    bits = _compare_full(wl, run)
    rng = np.random.default_rng(n_cat)
    tok = np.array([rng.choice(np.flatnonzero(bits[b])) for b in range(run.B)], dtype=np.int32)
    t = torch.from_numpy(tok).cuda()
    a, c = G.Configs(run.spec, run.B), G.Configs(run.spec, run.B)
    st_a = torch.zeros(run.B, dtype=torch.int32, device="cuda")
    st_c = torch.zeros(run.B, dtype=torch.int32, device="cuda")
    m_a = torch.zeros_like(run.mask)
    m_c = torch.zeros_like(run.mask)
    G.grid_advance(run.spec.h, run.cfg.h, a.h, t, st_a)
    G.grid_masks(run.spec.h, a.h, m_a, st_a)
    G.grid_advance_masks(run.spec.h, run.cfg.h, c.h, t, m_c, st_c)
    torch.cuda.synchronize()
    assert torch.equal(m_a, m_c) and torch.equal(st_a, st_c)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_masked_logits_bit_exact(dtype):
    """grid_apply_mask: rejected -> -inf, accepted values bit-identical (incl.
    NaN payloads); strided rows."""
    import torch
    from paper_2607_11951_gb300 import grid as G
    wl, run = _run("headline", configs.sql_select_only)
    run.masks()
    bits = torch.from_numpy(unpack(run.mask.cpu().numpy().view(np.uint32), run.V).astype(bool))
    lg = torch.from_numpy(configs.logits(7, run.B, run.V))
    lg[0, :7] = float("nan")
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    for stride in (run.V, run.V + 4, run.V + 8):  # 32-byte aligned rows and not
        buf = torch.zeros(run.B, stride, dtype=tdt)
        buf[:, :run.V] = lg.to(tdt)
        ref = buf.clone()
        ref[:, :run.V] = torch.where(bits, buf[:, :run.V], torch.tensor(float("-inf"), dtype=tdt))
        d = buf.cuda()
        view = d[:, :run.V]
        G.grid_apply_mask(run.mask, view)
        torch.cuda.synchronize()
        got = d.cpu()
        iv = torch.int32 if dtype == "f32" else torch.int16
        assert torch.equal(got.view(iv), ref.view(iv))


@pytest.mark.parametrize("name", ["headline", "tiny_ragged"])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_masks_apply_fused_equals_masks_then_apply(name, dtype):
    """grid_masks_apply: the same mask words and statuses as grid_masks, and
    the same logits bit for bit as grid_apply_mask on that mask (NaN
    payloads kept), for 32-byte aligned rows and unaligned strides and a
    vocabulary whose last mask word is ragged."""
    import torch
    from paper_2607_11951_gb300 import grid as G
    if name == "headline":
        wl, run = _run("headline", configs.sql_select_only)
    else:
        wl = configs.tiny_expr(B=5, V=517)
        run = GpuRun(wl)
        assert (run.build_configs() == 0).all()
    words, status = run.masks()
    lg = torch.from_numpy(configs.logits(11, run.B, run.V))
    lg[0, :5] = float("nan")
    lg[1, 3] = float("nan")
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    iv = torch.int32 if dtype == "f32" else torch.int16
    for stride in (run.V, run.V + 1, run.V + 16):
        buf = torch.zeros(run.B, stride, dtype=tdt)
        buf[:, :run.V] = lg.to(tdt)
        ref = buf.cuda()
        G.grid_apply_mask(run.mask, ref[:, :run.V])
        got = buf.cuda()
        m2 = torch.zeros_like(run.mask)
        st2 = torch.full_like(run.status, -1)
        G.grid_masks_apply(run.spec.h, run.cfg.h, m2, st2, got[:, :run.V])
        torch.cuda.synchronize()
        assert (m2.cpu().numpy().view(np.uint32) == words).all()
        assert (st2.cpu().numpy() == status).all()
        assert torch.equal(got.cpu().view(iv), ref.cpu().view(iv)), stride


def test_advance_semantics_and_status():
    """Out-of-place advance leaves its input alone; a token outside the mask,
    an out-of-range id and a special id give TOKEN_NOT_ALLOWED and keep the
    row; EOS at a sentence completes the row (all-zero mask, COMPLETE)."""
    import torch
    from paper_2607_11951_gb300 import grid as G
    wl, run = _run("admin", configs.sql_admin)
    words0, _ = run.masks()
    bits0 = unpack(words0, run.V)
    out = G.Configs(run.spec, run.B)
    B = run.B
    rng = np.random.default_rng(3)
    tok = np.zeros(B, dtype=np.int32)
    kinds = []
    for b in range(B):
        adm = np.nonzero(bits0[b])[0]
        rej = np.nonzero(bits0[b] == 0)[0]
        k = b % 4
        kinds.append(k)
        if k == 0:
            tok[b] = rng.choice(adm)
        elif k == 1:
            tok[b] = rng.choice(rej[rej != wl["eos"]])
        elif k == 2:
            tok[b] = run.V + 5
        else:
            tok[b] = wl["specials"][0]
    st = torch.zeros(B, dtype=torch.int32, device="cuda")
    G.grid_advance(run.spec.h, run.cfg.h, out.h, torch.from_numpy(tok).cuda(), st)
    torch.cuda.synchronize()
    st = st.cpu().numpy()
    for b in range(B):
        assert st[b] == (0 if kinds[b] == 0 else 3), (b, kinds[b], st[b])
    # input unchanged
    words1, _ = run.masks()
    assert (words1 == words0).all()
    # rejected rows of `out` equal their input; accepted rows match the oracle
    words2, s2 = run.masks(out)
    bits2 = unpack(words2, run.V)
    from oracle import compile_grammar
    og = compile_grammar(wl["grammar"], wl["role"], wl["lexicons"])
    for b in range(0, B, 3):
        if kinds[b] != 0:
            assert (bits2[b] == bits0[b]).all()
        else:
            cfg = og.config_from_ids(list(wl["prefixes"][b]) + [int(tok[b])], wl["tokens"], wl["eos"], wl["specials"])
            want = np.asarray(og.mask(cfg, wl["tokens"], wl["eos"], wl["specials"]), dtype=np.uint8)
            assert (bits2[b] == want).all(), b


def test_eos_completes_row_and_empty_prefix():
    import torch
    from paper_2607_11951_gb300 import grid as G
    from workloads.gen import GreedyTokenizer
    wl = configs.tiny_expr(B=4)
    tk = GreedyTokenizer(wl["tokens"], [wl["eos"]])
    wl["prefixes"] = [tk.encode(b"a+1"), [], tk.encode(b"(a"), tk.encode(b"1 ")]
    run = GpuRun(wl)
    assert (run.build_configs() == 0).all()
    words, status = run.masks()
    bits = unpack(words, run.V)
    eos = wl["eos"]
    assert bits[0][eos] == 1 and bits[1][eos] == 0 and bits[2][eos] == 0 and bits[3][eos] == 1
    toks = torch.tensor([eos, eos, eos, -1], dtype=torch.int32, device="cuda")
    st = torch.zeros(4, dtype=torch.int32, device="cuda")
    G.grid_advance(run.spec.h, run.cfg.h, run.cfg.h, toks, st)
    torch.cuda.synchronize()
    assert st.cpu().tolist() == [0, 3, 3, 0]
    words, status = run.masks()
    assert status.tolist()[0] == G.GRID_ST_COMPLETE and (words[0] == 0).all()
    assert status.tolist()[1:] == [0, 0, 0]


def test_ragged_vocab_tail_and_single_row():
    """V not a multiple of 32, B = 1, alias spellings."""
    wl = configs.tiny_expr(B=1, V=517)
    run = GpuRun(wl)
    assert (run.build_configs() == 0).all()
    _compare_full(wl, run)


def test_walk_work_counters():
    """The measurement hook counts without changing the masks: with counters
    on, the masks equal those without; lexer steps, ACTION lookups and the
    records and spellings evaluated are all counted on the headline batch, and
    a step evaluates no more records per row and context than the tables
    hold."""
    import torch
    from paper_2607_11951_gb300 import grid as G
    wl, run = _run("headline", configs.sql_select_only)
    words0, st0 = run.masks()
    work = torch.zeros(6, dtype=torch.int64, device="cuda")
    G.grid_spec_set_work_counters(run.spec.h, work)
    words1, st1 = run.masks()
    G.grid_spec_set_work_counters(run.spec.h, None)
    torch.cuda.synchronize()
    assert (words1 == words0).all() and (st1 == st0).all()
    w = work.cpu().tolist()
    assert all(x > 0 for x in w), w
    assert w[4] <= 2 * run.B * run.spec.info()["verdict_classes"]
    words2, _ = run.masks()  # counting off again: the counters stay as they were
    torch.cuda.synchronize()
    assert work.cpu().tolist() == w and (words2 == words0).all()
