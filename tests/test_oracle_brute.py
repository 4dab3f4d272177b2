"""Pin the oracle's mask semantics to brute force (Def. 2, Def. 4, EOS gate).

For every byte string s up to a length bound over a small alphabet (plus
random longer strings built from sentence prefixes and mutations), the oracle's
viability of s must equal Prefix(L) membership decided by the independent
recognizer in ``brute.py`` (completion search), and the oracle's EOS gate at s
must equal membership of s in L.
"""
import itertools

import numpy as np
import pytest

from oracle import compile_grammar
from tests.brute import BruteGrammar
from workloads import grammar_text
from workloads.gen import expr_sentence


def _strings(alpha: bytes, max_len: int):
    for L in range(max_len + 1):
        for tup in itertools.product(alpha, repeat=L):
            yield bytes(tup)


# ---------------------------------------------------------------------------
# Expression grammar.  Completion set argument: if s is a viable prefix, then
# appending an operand when one is expected ("a", or " a" / "1" variants; ""
# when s already ends in an operand or ")") and then closing every unclosed
# "(" yields a sentence.  Unclosed parens <= count of "(" in s.
# ---------------------------------------------------------------------------
def _expr_completions(s: bytes):
    k_max = s.count(b"(")
    return [x + b")" * k for x in (b"", b"a", b" a", b"1") for k in range(k_max + 1)]


def _check(og, bg, strings, completions):
    bad = []
    for s in strings:
        cfg = og.feed_bytes(og.start_config(), s)
        v_or = cfg is not None and og.live_end(cfg)
        v_bf = bg.in_prefix_L(s, completions(s))
        if v_or != v_bf:
            bad.append(("viable", s, v_or, v_bf))
        e_or = cfg is not None and og.eos_ok(cfg)
        e_bf = bg.in_L(s)
        if e_or != e_bf:
            bad.append(("eos", s, e_or, e_bf))
        if v_bf is False and e_bf:
            bad.append(("brute-inconsistent", s))
    return bad


def test_expr_exhaustive_short_strings():
    text = grammar_text("expr")
    og = compile_grammar(text)
    bg = BruteGrammar(text)
    strings = list(_strings(b"a1+*() ", 5))
    bad = _check(og, bg, strings, _expr_completions)
    assert not bad, bad[:10]


def test_expr_random_long_prefixes_and_mutations():
    text = grammar_text("expr")
    og = compile_grammar(text)
    bg = BruteGrammar(text)
    rng = np.random.default_rng(5)
    alpha = b"ab1+*() "
    strings = []
    for _ in range(600):
        s = expr_sentence(rng, 4).encode()
        cut = int(rng.integers(0, len(s) + 1))
        s = s[:cut]
        if s and rng.random() < 0.5:
            i = int(rng.integers(0, len(s)))
            s = s[:i] + bytes([alpha[int(rng.integers(len(alpha)))]]) + s[i + 1:]
        strings.append(s[:24])
    bad = _check(og, bg, strings, _expr_completions)
    assert not bad, bad[:10]


# ---------------------------------------------------------------------------
# Lexicon grammar (contextual pick + L3 filter + L2 projection).  Completion
# set argument: a viable pending lexeme is finished into a word of the picked
# category by one of X (suffixes of the lexicon words), and from any parser
# position one tail in Y completes the statement: at the start -> "g a o ab;"
# (or "d ab;"), after GET or ',' -> " a o ab;", after a column -> " o ab;",
# after OF or DEL -> " ab;", after a table -> ";".
# ---------------------------------------------------------------------------
LEX = {"TABLE_NAME": ["ab", "abc", "ba"], "COLUMN_NAME": ["a", "ab", "c"]}
_X = [b"", b"a", b"b", b"c", b"bc"]
_Y = [b"", b";", b" ;", b" ab;", b"ab;", b" o ab;", b"o ab;", b" a o ab;", b"a o ab;",
      b"g a o ab;", b"d ab;"]
_LEX_COMPL = [x + y for x in _X for y in _Y]


@pytest.mark.parametrize("role", [None, []])
def test_lexicon_grammar_exhaustive(role):
    text = grammar_text("lexfix")
    og = compile_grammar(text, role=role, lexicons=LEX)
    bg = BruteGrammar(text, role=role, lexicons=LEX)
    strings = list(_strings(b"abcgod,; ", 4))
    bad = _check(og, bg, strings, lambda s: _LEX_COMPL)
    assert not bad, bad[:10]


def test_lexicon_grammar_random_longer():
    text = grammar_text("lexfix")
    rng = np.random.default_rng(11)
    for role in (None, []):
        og = compile_grammar(text, role=role, lexicons=LEX)
        bg = BruteGrammar(text, role=role, lexicons=LEX)
        strings = []
        for _ in range(400):
            cols = ",".join(["a", "ab", "c"][int(rng.integers(3))] for _ in range(int(rng.integers(1, 4))))
            tab = ["ab", "abc", "ba"][int(rng.integers(3))]
            s = ("g " + cols + " o " + tab + ";").encode() if rng.random() < 0.8 else ("d " + tab + ";").encode()
            s = s[:int(rng.integers(0, len(s) + 1))]
            if s and rng.random() < 0.5:
                i = int(rng.integers(0, len(s)))
                s = s[:i] + bytes([b"abcgod,; "[int(rng.integers(9))]]) + s[i + 1:]
            strings.append(s)
        bad = _check(og, bg, strings, lambda s: _LEX_COMPL)
        assert not bad, bad[:10]


# ---------------------------------------------------------------------------
# Pick grammar: a qualified column TABLE_NAME "." COLUMN_NAME beside a bare
# COLUMN_NAME, so that right after "g" or "," both categories are
# parser-viable and a word in both lexicons ("ab") is decided by the priority
# order alone.  Completion set argument: a viable pending lexeme r is finished
# into a lexicon word r.x, x a suffix of a word (every category lexeme is
# emitted only as a word); the pick of r.x depends on the stack and the word
# only, and leaves the parser at one of eight positions, each finished by a
# tail in Y that starts with a byte ending r.x (variants with and without a
# leading blank): start -> "g a o ab;", after GET or ',' -> "a o ab;", after
# a TABLE_NAME of a column -> ".c o ab;", after '.' -> "c o ab;", after a
# column -> "o ab;", after OF -> "ab;", after the table -> ";", after ';' -> "".
# ---------------------------------------------------------------------------
_XP = [b"", b"a", b"b", b"c", b"ab", b"bc", b"abc", b"ba"]
_YP = [b"", b";", b" ;", b" ab;", b"ab;", b" o ab;", b"o ab;", b" a o ab;", b"a o ab;", b"g a o ab;",
       b".c o ab;", b" .c o ab;", b"c o ab;", b" c o ab;"]
_PICK_COMPL = [x + y for x in _XP for y in _YP]


def brute_verdicts(bg, alpha: bytes, max_len: int, completions):
    """(s, s in Prefix(L), s in L) for every s over ``alpha`` with |s| <= max_len.
    Prefix(L) is prefix-closed, so an extension of a string outside it is
    outside it too (and outside L) without a completion search."""
    out, level = [], [b""]
    for L in range(max_len + 1):
        nxt = []
        for s in level:
            v = bg.in_prefix_L(s, completions(s))
            out.append((s, v, bg.in_L(s) if v else False))
            if v and L < max_len:
                nxt.extend(s + bytes([c]) for c in alpha)
            elif L < max_len:
                stack = [s]
                while stack:  # every extension of s: (False, False)
                    u = stack.pop()
                    for c in alpha:
                        w = u + bytes([c])
                        out.append((w, False, False))
                        if len(w) < max_len:
                            stack.append(w)
        level = nxt
    return out


def _check_verdicts(og, verdicts):
    bad = []
    for s, v_bf, e_bf in verdicts:
        cfg = og.feed_bytes(og.start_config(), s)
        if (cfg is not None and og.live_end(cfg)) != v_bf:
            bad.append(("viable", s))
        if (cfg is not None and og.eos_ok(cfg)) != e_bf:
            bad.append(("eos", s))
    return bad


def test_pick_grammar_exhaustive():
    """Priority order of the contextual pick (Sec. 2; TABLE_NAME before
    COLUMN_NAME as in the worked example of Sec. 7.1) at points where both
    candidates are parser-viable."""
    text = grammar_text("lexpick")
    og = compile_grammar(text, lexicons=LEX)
    bg = BruteGrammar(text, lexicons=LEX)
    verdicts = brute_verdicts(bg, b"abcgo.,; ", 5, lambda s: _PICK_COMPL)
    assert len(verdicts) == sum(9 ** k for k in range(6))
    # the pick is observable: a shared word right after "g" is a table and
    # needs ".", a word of the column lexicon only is a bare column
    v = {s: (a, b) for s, a, b in verdicts}
    assert v[b"g ab"] == (True, False) and v[b"g ab."] == (True, False)
    assert v[b"g ab,"] == (False, False) and v[b"g abo"] == (False, False)
    assert v[b"g a o"] == (True, False) and v[b"g c,"] == (True, False)
    bad = _check_verdicts(og, verdicts)
    assert not bad, bad[:10]


def test_pick_grammar_random_sentences():
    text = grammar_text("lexpick")
    og = compile_grammar(text, lexicons=LEX)
    bg = BruteGrammar(text, lexicons=LEX)
    rng = np.random.default_rng(13)
    strings = []
    for _ in range(500):
        cols = []
        for _ in range(int(rng.integers(1, 4))):
            if rng.random() < 0.5:
                cols.append(["a", "c", "ab"][int(rng.integers(3))])  # "ab" bare: read as a table
            else:
                cols.append(["ab", "abc", "ba"][int(rng.integers(3))] + "." + ["a", "ab", "c"][int(rng.integers(3))])
        s = ("g " + ",".join(cols) + " o " + ["ab", "abc", "ba"][int(rng.integers(3))] + ";").encode()
        s = s[:int(rng.integers(0, len(s) + 1))]
        if s and rng.random() < 0.4:
            i = int(rng.integers(0, len(s)))
            s = s[:i] + bytes([b"abcgo.,; "[int(rng.integers(9))]]) + s[i + 1:]
        strings.append(s)
    bad = _check(og, bg, strings, lambda s: _PICK_COMPL)
    assert not bad, bad[:10]


def test_contextual_pick_shared_word():
    """'ab' is in both lexicons: a column after 'g', a table after 'o'."""
    og = compile_grammar(grammar_text("lexfix"), lexicons=LEX)
    tn = og.g.term_ids["TABLE_NAME"]
    cn = og.g.term_ids["COLUMN_NAME"]
    c = og.feed_bytes(og.start_config(), b"g ab ")
    # the shift of COLUMN_NAME leaves a column-list state on the stack
    st = og.stack_list(c)
    assert og.simulate(c.stack, og.g.term_ids["OF"]) is not None
    c2 = og.feed_bytes(og.start_config(), b"g a o ab ")
    assert c2 is not None and og.eos_ok(og.feed_bytes(c2, b";"))
    assert tn < cn and len(st) >= 2
