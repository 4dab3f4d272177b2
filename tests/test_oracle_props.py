"""Oracle properties from the paper: the worked example (Sec. 7.1), Prop. 2
(the step-1 mask is non-empty), Prop. 7/8 along random walks (every sampled
token keeps the output viable, no dead ends, EOS only on sentences), role and
schema unreachability (Sec. 7.1, Sec. 8.6 speller), alias/special invariants
(Def. 3, Def. 4) and the lexicon precondition (Prop. 8 (d))."""
import os

import numpy as np
import pytest

from oracle import compile_grammar
from oracle.core import LexiconError
from tests.brute import BruteGrammar
from workloads import grammar_text

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "worked_example_1.txt")


def _load_golden():
    meta, rows = {}, []
    for line in open(GOLDEN, encoding="utf-8"):
        line = line.rstrip("\n")
        if not line or line.startswith("#"):
            continue
        parts = line.split("\t")
        if parts[0] in ("table", "column", "role"):
            meta[parts[0]] = parts[1]
            continue
        dec = lambda s: s.replace("\\x20", " ").encode()
        rows.append((dec(parts[0]), parts[1], int(parts[2])))
    return meta, rows


def test_worked_example_1():
    meta, rows = _load_golden()
    lex = {"TABLE_NAME": meta["table"].split(","), "COLUMN_NAME": meta["column"].split(",")}
    og = compile_grammar(grammar_text("sql"), role=[], lexicons=lex)  # analyst: no DML
    for prefix, tok, want in rows:
        cfg = og.feed_bytes(og.start_config(), prefix)
        assert cfg is not None and og.live_end(cfg), prefix
        got = og.eos_ok(cfg) if tok == "EOS" else og.token_bit(cfg, tok.replace("\\x20", " ").encode())
        assert int(got) == want, (prefix, tok, got, want)


def test_admin_role_positive_control():
    lex = {"TABLE_NAME": ["employees", "orders"], "COLUMN_NAME": ["id"]}
    og = compile_grammar(grammar_text("sql"), role=["dml"], lexicons=lex)
    s = og.start_config()
    for verb in (b"insert", b"update", b"delete", b"select"):
        assert og.token_bit(s, verb)


def test_step1_mask_nonempty_and_specials():
    """Prop. 2: masking needs Prefix(L); the first mask is non-empty.
    Specials and EOS are never set by the trie rule."""
    og = compile_grammar(grammar_text("expr"))
    toks = [b"a", b"1", b"(", b"+", b")", b"a", b"<s>", b"<eos>"]
    m = og.mask(og.start_config(), toks, eos=7, specials=[6])
    assert m[0] == 1 and m[1] == 1 and m[2] == 1 and m[3] == 0 and m[4] == 0
    assert m[5] == m[0]  # alias ids share one verdict
    assert m[6] == 0 and m[7] == 0  # the empty output is not a sentence


def _walk(og, bg, toks, eos, rng, steps):
    cfg = og.start_config()
    out = b""
    for _ in range(steps):
        m = og.mask(cfg, toks, eos)
        ones = [i for i, v in enumerate(m) if v]
        assert ones, ("dead end", out)
        t = ones[int(rng.integers(len(ones)))]
        if t == eos:
            assert bg.in_L(out), out
            return out, True
        nxt = og.advance(cfg, t, toks, eos)
        assert nxt is not None
        out += toks[t]
        assert og.live_end(nxt)
        cfg = nxt
    return out, False


def test_random_walks_expr_and_lexfix():
    rng = np.random.default_rng(23)
    og = compile_grammar(grammar_text("expr"))
    bg = BruteGrammar(grammar_text("expr"))
    toks = [bytes([c]) for c in b"ab1+*() "] + [b"a+", b"(a", b"1)", b") ", b"*(", b" +"] + [b"<eos>"]
    ends = 0
    for _ in range(60):
        _, e = _walk(og, bg, toks, len(toks) - 1, rng, 30)
        ends += e
    assert ends > 0
    lex = {"TABLE_NAME": ["ab", "abc", "ba"], "COLUMN_NAME": ["a", "ab", "c"]}
    og = compile_grammar(grammar_text("lexfix"), lexicons=lex)
    bg = BruteGrammar(grammar_text("lexfix"), lexicons=lex)
    toks = [bytes([c]) for c in b"abcgod,; "] + [b"g a", b"ab o", b"c,", b" ab;", b"o b"] + [b"<eos>"]
    ends = 0
    for _ in range(60):
        _, e = _walk(og, bg, toks, len(toks) - 1, rng, 30)
        ends += e
    assert ends > 0


def test_random_walks_sql_no_dead_ends():
    lex = {"TABLE_NAME": ["employees", "orders"], "COLUMN_NAME": ["id", "name"]}
    og = compile_grammar(grammar_text("sql"), role=[], lexicons=lex)
    bg = BruteGrammar(grammar_text("sql"), role=[], lexicons=lex)
    pieces = [b"select", b" from", b" where", b" *", b" ", b"employees", b"orders", b"id", b"name",
              b" =", b" 1", b";", b"(", b")", b",", b" and", b" or", b"emp", b"loyees", b"'x'",
              b"count", b"(*)", b" in", b" not", b" is", b" null", b" group by", b" order", b" by",
              b".", b" limit", b" 5", b" exists", b"-- c\n", b"ord", b"ers", b"na", b"me"]
    toks = [bytes([c]) for c in b"abcdefghijklmnopqrstuvwxyz_0123456789 ;,().*='<>\n"] + pieces + [b"<eos>"]
    rng = np.random.default_rng(29)
    for _ in range(8):
        _walk(og, bg, toks, len(toks) - 1, rng, 40)


def test_schema_speller_never_spells_a_foreign_identifier():
    """Sec. 8.6 speller, model-free: at the identifier position of
    'select * from ', every token sequence (depth <= 3) admitted step by step
    keeps the pending lexeme a prefix of a lexicon word; every lexicon word is
    reachable (positive control)."""
    words = ["employees", "orders", "emp"]
    og = compile_grammar(grammar_text("sql"), role=[], lexicons={"TABLE_NAME": words, "COLUMN_NAME": ["id"]})
    cfg0 = og.feed_bytes(og.start_config(), b"select * from ")
    pieces = [b"e", b"o", b"s", b"emp", b"loy", b"ees", b"rd", b"ers", b"sal", b"aries", b"r", b"d", b"x"]
    prefixes = {w[:k] for w in words for k in range(len(w) + 1)}
    frontier = [(cfg0, b"")]
    reached = set()
    for _ in range(3):
        nxt = []
        for cfg, spelled in frontier:
            for p in pieces:
                if og.token_bit(cfg, p):
                    c2 = og.feed_bytes(cfg, p)
                    s2 = spelled + p
                    assert s2.decode() in prefixes, s2
                    reached.add(s2)
                    nxt.append((c2, s2))
        frontier = nxt
    assert b"emp" in reached and b"employees" in reached and b"orders" in reached


def test_lexicon_precondition_is_validated():
    with pytest.raises(LexiconError):
        compile_grammar(grammar_text("sql"), lexicons={"TABLE_NAME": ["Official_ratings_(millions)"],
                                                       "COLUMN_NAME": []})
