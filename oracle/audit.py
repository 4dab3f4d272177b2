"""Audit chain of the decoding loop (GRID Sec. 6.4) -- TEST INFRASTRUCTURE.

Written from the definitions only (hashlib's BLAKE2b is the hash primitive):
  * node hash: H(root) = 0, H(node) = low 64 bits (little-endian) of
    BLAKE2b-128(u64 H(parent) || u32 kind || u32 id), where (kind, id) is the
    grammar symbol on which the node's state was entered: (0, terminal index)
    or (1, rank of the nonterminal's name in byte order among all nonterminal
    names of the grammar text).  The configuration hash is H(top node).
    (Sec. 6.4 writes the node's payload as its state and goto; LR state numbers
    depend on the table construction -- canonical LR(1) here, LALR(1) in the
    library -- so the entering symbol, which determines the state, is hashed.)
  * mask entry id: the mask row as little-endian 32-bit words in chunks of
    256 words, each hashed with BLAKE2b-128; then BLAKE2b-128 of "GRIDmask" ||
    u32 V || u32 number of chunks || the chunk digests.
  * record: u64 step || u64 config hash || mask id || i32 token || u32 blocked
    (ids < V the mask rejects) || u32 kind || prev (16) -- 60 bytes -- then a
    zero u32 and the record hash BLAKE2b-128 of the 60 bytes: 80 bytes.  The
    first record's prev is the genesis constant BLAKE2b-128("GRID audit chain
    genesis"); a seal (kind 3) carries the stop reason as its token, mode flags
    as its blocked count and the spec fingerprint as its mask id.
  * fingerprints of the inputs (grammar, vocabulary, spec).
"""
from __future__ import annotations

import hashlib
import struct


def b2_128(data: bytes) -> bytes:
    return hashlib.blake2b(data, digest_size=16).digest()


GENESIS = b2_128(b"GRID audit chain genesis")


def nonterminal_ranks(og) -> dict:
    names = sorted({p[0] for p in og.g.productions}, key=lambda n: n.encode())
    return {n: i for i, n in enumerate(names)}


def node_symbol(og, state, ranks) -> tuple:
    X = og.lr.access[state]
    return (1, ranks[X]) if isinstance(X, str) else (0, X)


def config_hash(og, cfg, ranks=None) -> int:
    """H(top node) of the configuration's stack."""
    ranks = ranks or nonterminal_ranks(og)
    states = og.stack_list(cfg)
    h = 0
    for s in states[1:]:
        kind, i = node_symbol(og, s, ranks)
        h = struct.unpack("<Q", b2_128(struct.pack("<QII", h, kind, i))[:8])[0]
    return h


def mask_words(bits) -> list:
    V = len(bits)
    W = (V + 31) // 32
    words = [0] * W
    for t, x in enumerate(bits):
        if x:
            words[t >> 5] |= 1 << (t & 31)
    return words


def mask_id(bits) -> bytes:
    V = len(bits)
    words = mask_words(bits)
    chunks = [words[i:i + 256] for i in range(0, len(words), 256)]
    digs = [b2_128(struct.pack("<%dI" % len(c), *c)) for c in chunks]
    return b2_128(b"GRIDmask" + struct.pack("<II", V, len(chunks)) + b"".join(digs))


def record(step: int, cfg_hash: int, mid: bytes, token: int, blocked: int, kind: int, prev: bytes) -> bytes:
    body = struct.pack("<QQ", step, cfg_hash) + mid + struct.pack("<iII", token, blocked, kind) + prev
    assert len(body) == 60
    return body + b"\0\0\0\0" + b2_128(body)


def record_hash(rec: bytes) -> bytes:
    return rec[64:80]


def grammar_fingerprint(text: str, role, lexicons, max_depth: int = 4096) -> bytes:
    """``role``: None or the list of kept tags (passed comma-joined);
    ``lexicons``: ordered (category, words) pairs."""
    raw = text.encode()
    out = b"GRIDgram" + struct.pack("<Q", len(raw)) + raw
    if role is None:
        out += struct.pack("<Q", 2 ** 64 - 1)
    else:
        r = ",".join(role).encode()
        out += struct.pack("<Q", len(r)) + r
    lex = list(lexicons.items()) if isinstance(lexicons, dict) else list(lexicons)
    out += struct.pack("<Q", len(lex))
    for cat, words in lex:
        c = cat.encode()
        out += struct.pack("<Q", len(c)) + c + struct.pack("<Q", len(words))
        for w in words:
            wb = w if isinstance(w, bytes) else w.encode()
            out += struct.pack("<Q", len(wb)) + wb
    out += struct.pack("<Q", max_depth)
    return b2_128(out)


def vocab_fingerprint(tokens, eos: int, specials) -> bytes:
    out = b"GRIDvoca" + struct.pack("<Qq", len(tokens), eos) + struct.pack("<Q", len(specials))
    out += b"".join(struct.pack("<q", s) for s in specials)
    out += b"".join(struct.pack("<Q", len(t)) + t for t in tokens)
    return b2_128(out)


def spec_fingerprint(gfp: bytes, vfp: bytes) -> bytes:
    return b2_128(b"GRIDspec" + gfp + vfp)


def replay(og, prefix_ids, steps, tokens, eos: int, specials=()):
    """One row's log: the row starts at the configuration of ``prefix_ids``
    (built without records, as a fresh chain starts there), then each
    (token, kind) step appends a record made at the current configuration and
    advances by the token.  Returns (records, final configuration)."""
    ranks = nonterminal_ranks(og)
    cfg = og.config_from_ids(prefix_ids, tokens, eos, specials)
    prev, recs = GENESIS, []
    for k, (tok, kind) in enumerate(steps):
        bits = og.mask(cfg, tokens, eos, specials)
        rec = record(k, config_hash(og, cfg, ranks), mask_id(bits), tok, len(bits) - sum(bits), kind, prev)
        recs.append(rec)
        prev = record_hash(rec)
        cfg = og.advance(cfg, tok, tokens, eos, specials)
        assert cfg is not None, ("token not admitted", k, tok)
    return recs, cfg


def verify(records) -> int:
    """Index of the first record whose step, link or hash is wrong; -1 if none."""
    prev = GENESIS
    for k, rec in enumerate(records):
        step = struct.unpack("<Q", rec[:8])[0]
        if step != k or rec[44:60] != prev or rec[60:64] != b"\0\0\0\0" or rec[64:80] != b2_128(rec[:60]):
            return k
        prev = rec[64:80]
    return -1
