"""Audit chain pieces that need no GPU (Sec. 6.4): the library's BLAKE2b
against hashlib, the input fingerprints against the oracle's own
serialization, tamper detection by both verifiers on chains the oracle
builds, and the rolling configuration hash's invariants."""
import hashlib
import struct

import numpy as np
import pytest

from oracle import audit, compile_grammar
from workloads import configs, grammar_text


def _G():
    from paper_2607_11951_gb300 import grid as G
    G.lib()
    return G


def test_blake2b_matches_hashlib():
    G = _G()
    rng = np.random.default_rng(3)
    for n in list(range(0, 260)) + [511, 512, 513, 1024, 4097]:
        data = rng.integers(0, 256, size=n, dtype=np.uint8).tobytes()
        for ob in (1, 16, 32, 64) if n % 7 == 0 else (16,):
            assert G.grid_blake2b(data, ob) == hashlib.blake2b(data, digest_size=ob).digest(), (n, ob)
    assert G.grid_audit_genesis() == audit.GENESIS


@pytest.mark.parametrize("name", ["tiny_expr", "sql_admin", "tiny_pick"])
def test_fingerprints_match_oracle(name):
    G = _G()
    wl = getattr(configs, name)(**({"B": 2} if name != "tiny_pick" else {}))
    g = G.Grammar(wl["grammar"], wl["role"], wl["lexicons"])
    v = G.Vocab(wl["tokens"], wl["eos"], wl["specials"])
    assert G.grid_fingerprint(grammar=g) == audit.grammar_fingerprint(wl["grammar"], wl["role"], wl["lexicons"])
    assert G.grid_fingerprint(vocab=v) == audit.vocab_fingerprint(wl["tokens"], wl["eos"], wl["specials"])
    # any change of an input changes the fingerprint
    g2 = G.Grammar(wl["grammar"], wl["role"], wl["lexicons"], max_depth=4095)
    assert G.grid_fingerprint(grammar=g2) != G.grid_fingerprint(grammar=g)


def _oracle_chain():
    og = compile_grammar(grammar_text("expr"))
    toks = [b"a", b"+", b"(", b")", b"1", b"*", b" ", b"<eos>"]
    steps = [(2, 0), (0, 0), (1, 0), (4, 0), (3, 0), (5, 1), (0, 0), (7, 2)]
    recs, _ = audit.replay(og, [], steps, toks, 7)
    return recs


def test_tamper_detection_both_verifiers():
    """Every chain the oracle builds passes both verifiers; flipping any one
    byte of any record is caught at that record (or, for a hash byte, at
    that record too, its stored hash no longer matching)."""
    G = _G()
    recs = _oracle_chain()
    blob = b"".join(recs)
    assert audit.verify(recs) == -1 and G.grid_audit_verify(blob) == -1
    for k in range(len(recs)):
        for off in (0, 8, 16, 31, 32, 36, 40, 44, 59, 60, 64, 79):
            bad = bytearray(blob)
            bad[k * 80 + off] ^= 0x01
            assert G.grid_audit_verify(bytes(bad)) == k, (k, off)
            parts = [bytes(bad[i * 80:(i + 1) * 80]) for i in range(len(recs))]
            assert audit.verify(parts) == k
    # dropping or reordering records breaks the chain
    assert G.grid_audit_verify(b"".join(recs[1:])) == 0
    assert G.grid_audit_verify(b"".join([recs[0], recs[2], recs[1]] + recs[3:])) == 1


def test_config_hash_rolling_and_symbolic():
    """H pins the stack's symbol sequence: equal for two outputs whose stacks
    hold the same symbols, different otherwise; a record's config hash after
    each push equals the hash recomputed from the root."""
    og = compile_grammar(grammar_text("expr"))
    a = og.feed_bytes(og.start_config(), b"(a+1*b")
    b = og.feed_bytes(og.start_config(), b"(xy+22*z")
    c = og.feed_bytes(og.start_config(), b"(a+1+b")
    assert og.stack_list(a) != og.stack_list(c)
    assert audit.config_hash(og, a) == audit.config_hash(og, b) != audit.config_hash(og, c)
    # from scratch: H over the symbols, one BLAKE2b per node
    ranks = audit.nonterminal_ranks(og)
    h = 0
    for s in og.stack_list(a)[1:]:
        kind, i = audit.node_symbol(og, s, ranks)
        h = struct.unpack("<Q", hashlib.blake2b(struct.pack("<QII", h, kind, i), digest_size=16).digest()[:8])[0]
    assert h == audit.config_hash(og, a)
    assert audit.config_hash(og, og.start_config()) == 0
