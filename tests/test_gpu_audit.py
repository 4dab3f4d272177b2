"""Audit chain on the GPU (Sec. 6.4) replayed by the oracle: every record of
a decoding run -- step, rolling configuration hash, mask entry id, token,
blocked count, kind, link and hash -- equal byte for byte to the records the
oracle makes from the same tokens; forced-span records and the seal too; and
the logs pass the verifier while a tampered log fails where it was altered."""
import numpy as np
import pytest

from tests.harness import GpuRun, unpack
from workloads import configs

pytestmark = pytest.mark.gpu




@pytest.mark.parametrize("name", ["tiny_expr", "sql_admin"])
def test_audit_records_replay_bit_identically(name):
    import torch
    from oracle import audit, compile_grammar
    from paper_2607_11951_gb300 import grid as G
    wl = configs.tiny_expr(B=6) if name == "tiny_expr" else configs.sql_admin(B=4)
    run = GpuRun(wl)
    assert (run.build_configs() == 0).all()
    G.grid_configs_enable_audit(run.spec.h, run.cfg.h)
    B, steps = run.B, (8 if name == "tiny_expr" else 4)
    rng = np.random.default_rng(5)
    rec = torch.zeros((steps, B, 80), dtype=torch.uint8, device="cuda")
    log = [[] for _ in range(B)]
    for k in range(steps):
        words, status = run.masks()
        bits = unpack(words, run.V)
        tok = np.full(B, -1, np.int32)
        for b in range(B):
            if status[b] == 0:
                adm = np.flatnonzero(bits[b])
                adm = adm[adm != wl["eos"]] if adm.size > 1 else adm
                tok[b] = int(rng.choice(adm))
                log[b].append((int(tok[b]), 0))
        t = torch.from_numpy(tok).cuda()
        G.grid_audit_append(run.spec.h, run.cfg.h, run.mask, t, 0, rec[k])
        G.grid_advance(run.spec.h, run.cfg.h, run.cfg.h, t, run.status)
    reason = torch.arange(B, dtype=torch.int32, device="cuda") + 100
    seal = torch.zeros((B, 80), dtype=torch.uint8, device="cuda")
    G.grid_audit_seal(run.spec.h, run.cfg.h, reason, 0x5, seal)
    torch.cuda.synchronize()
    recs, seals = rec.cpu().numpy(), seal.cpu().numpy()
    og = compile_grammar(wl["grammar"], wl["role"], wl["lexicons"])
    spec_fp = audit.spec_fingerprint(audit.grammar_fingerprint(wl["grammar"], wl["role"], wl["lexicons"]),
                                     audit.vocab_fingerprint(wl["tokens"], wl["eos"], wl["specials"]))
    assert G.grid_fingerprint(spec=run.spec) == spec_fp
    for b in range(B):
        want, end = audit.replay(og, wl["prefixes"][b], log[b], wl["tokens"], wl["eos"], wl["specials"])
        got = [recs[k, b].tobytes() for k in range(len(log[b]))]
        assert got == want, (b, [i for i in range(len(got)) if got[i] != want[i]])
        seal_want = audit.record(len(want), audit.config_hash(og, end), spec_fp, 100 + b, 0x5, 3,
                                 audit.record_hash(want[-1]) if want else audit.GENESIS)
        assert seals[b].tobytes() == seal_want
        full = b"".join(got) + seal_want
        assert G.grid_audit_verify(full) == -1
        head, n = G.grid_audit_head(run.cfg.h, b)
        assert head == audit.record_hash(seal_want) and n == len(want) + 1
        bad = bytearray(full)
        bad[min(len(got) - 1, 1) * 80 + 33] ^= 0x80  # a token byte
        assert G.grid_audit_verify(bytes(bad)) == min(len(got) - 1, 1)


def test_audit_forced_span_records():
    """Each interior token of a forced span is audited (kind 1) at the
    configuration its mask was computed at."""
    import torch
    from oracle import audit, compile_grammar
    from paper_2607_11951_gb300 import grid as G
    wl = configs.forced_sql()
    run = GpuRun(wl)
    assert (run.build_configs() == 0).all()
    G.grid_configs_enable_audit(run.spec.h, run.cfg.h)
    B, M = run.B, 8
    span = torch.full((B, M), -7, dtype=torch.int32, device="cuda")
    span_len = torch.zeros(B, dtype=torch.int32, device="cuda")
    rec = torch.zeros((B, M, 80), dtype=torch.uint8, device="cuda")
    G.grid_forced_span(run.spec.h, run.cfg.h, M, run.mask, span, span_len, run.status, rec)
    torch.cuda.synchronize()
    sp, sl, rc = span.cpu().numpy(), span_len.cpu().numpy(), rec.cpu().numpy()
    og = compile_grammar(wl["grammar"], wl["role"], wl["lexicons"])
    n_forced = 0
    for b in range(B):
        steps = [(int(t), 1) for t in sp[b][:sl[b]]]
        want, _ = audit.replay(og, wl["prefixes"][b], steps, wl["tokens"], wl["eos"], wl["specials"])
        got = [rc[b, k].tobytes() for k in range(sl[b])]
        assert got == want, b
        n_forced += len(got)
        head, n = G.grid_audit_head(run.cfg.h, b)
        assert n == len(want) and head == (audit.record_hash(want[-1]) if want else audit.GENESIS)
    assert n_forced >= 3
    # records are required while audit is on
    with pytest.raises(G.GridError):
        G.grid_forced_span(run.spec.h, run.cfg.h, M, run.mask, span, span_len, run.status)
