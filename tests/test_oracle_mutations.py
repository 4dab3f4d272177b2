"""The oracle's pins catch plausible mistakes (CPU only).

Each case plants one mistake in a freshly compiled oracle -- a dropped step,
a missing condition, a wrong set, an off-by-one -- and checks that the
brute-force verdicts of ``test_oracle_brute`` (or the ``re`` pin of the lexer
DFA) disagree with it.  The unmodified oracle agrees with the same verdicts.
The candidate priority of the contextual pick is pinned on the pick grammar,
where a word of both lexicons meets two parser-viable candidates."""
import functools
import types

import pytest

from oracle import compile_grammar
from oracle.core import Config
from tests.brute import BruteGrammar
from tests.test_oracle_brute import LEX, _LEX_COMPL, _PICK_COMPL, _expr_completions, _strings, brute_verdicts
from workloads import grammar_text


@functools.lru_cache(maxsize=None)
def _brute(name):
    """Brute-force verdicts (viable, in L) of every short string, computed once."""
    if name == "lexpick":
        return brute_verdicts(BruteGrammar(grammar_text("lexpick"), lexicons=LEX), b"abcgo.,; ", 4,
                              lambda s: _PICK_COMPL)
    if name == "expr":
        bg = BruteGrammar(grammar_text("expr"))
        strings, compl = list(_strings(b"a1+*() ", 4)), _expr_completions
    else:
        bg = BruteGrammar(grammar_text("lexfix"), lexicons=LEX)
        strings, compl = list(_strings(b"abcgod,; ", 4)), (lambda s: _LEX_COMPL)
    return [(s, bg.in_prefix_L(s, compl(s)), bg.in_L(s)) for s in strings]


def _disagree(og, name):
    bad = []
    for s, v_bf, e_bf in _brute(name):
        cfg = og.feed_bytes(og.start_config(), s)
        if (cfg is not None and og.live_end(cfg)) != v_bf:
            bad.append(("viable", s))
        if (cfg is not None and og.eos_ok(cfg)) != e_bf:
            bad.append(("eos", s))
    return bad


def _expr_bad(og):
    return _disagree(og, "expr")


def _lex_bad(og):
    return _disagree(og, "lexfix")


def _pick_bad(og):
    return _disagree(og, "lexpick")


def _pick():
    return compile_grammar(grammar_text("lexpick"), lexicons=LEX)


def _expr():
    return compile_grammar(grammar_text("expr"))


def _lex():
    return compile_grammar(grammar_text("lexfix"), lexicons=LEX)


# ---- the mistakes -----------------------------------------------------------
def m_emit_accepts_prefix_of_word(og):
    og.candidates = lambda q, r: [t for t in sorted(og.dfa.acc[q]) if t not in og.categories or r in og.P[t]]


def m_priority_reversed(og):
    og.candidates = lambda q, r: [t for t in sorted(og.dfa.acc[q], reverse=True)
                                  if t not in og.categories or r in og.W[t]]


def m_emit_ignores_lexicon(og):
    og.candidates = lambda q, r: sorted(og.dfa.acc[q])


def m_live_ignores_lexicon_prefix(og):
    def live_end(self, cfg):
        if not cfg.r:
            return True
        for t in sorted(self.dfa.live[cfg.q]):
            if t in self.ignored:
                return True
            s = self.simulate(cfg.stack, t)
            if s is not None and s[0] == "shift":
                return True
        return False
    og.live_end = types.MethodType(live_end, og)


def m_ignored_needs_shift(og):
    def emit(self, stack, q, r):
        for t in self.candidates(q, r):
            s = self.simulate(stack, t)
            if s is not None and s[0] == "shift":
                return s[1]
        return None
    og.emit = types.MethodType(emit, og)


def m_killing_byte_dropped(og):
    def feed(self, cfg, b):
        nq = self.dfa.delta[cfg.q][b]
        if nq != self.DEAD:
            return Config(cfg.stack, nq, cfg.r + bytes([b]))
        if not cfg.r:
            return None
        st = self.emit(cfg.stack, cfg.q, cfg.r)
        return None if st is None else Config(st, self.START, b"")
    og.feed = types.MethodType(feed, og)


def m_eos_skips_finalize(og):
    def eos_ok(self, cfg):
        if cfg.complete:
            return False
        s = self.simulate(cfg.stack, self.END)
        return s is not None and s[0] == "accept"
    og.eos_ok = types.MethodType(eos_ok, og)


def m_reduce_pops_one_short(og):
    A, G, rhs, lhs = og.lr.ACTION, og.lr.GOTO, og.lr.rhs, og.lr.lhs

    def simulate(self, stack, tau):
        st = stack
        for _ in range(10000):
            a = A[st[0]].get(tau)
            if a is None:
                return None
            kind, arg = a
            if kind == "s":
                return ("shift", (arg, st))
            if kind == "acc":
                return ("accept", st)
            for _ in range(max(0, len(rhs[arg]) - 1)):
                st = st[1]
            st = (G[st[0]].get(lhs[arg], 0), st)
        return None
    og.simulate = types.MethodType(simulate, og)


def m_trailing_skips_parser(og):
    def live_end(self, cfg):
        return not cfg.r or any(t not in self.categories or cfg.r in self.P[t] for t in self.dfa.live[cfg.q])
    og.live_end = types.MethodType(live_end, og)


CASES = [
    (m_emit_accepts_prefix_of_word, _lex, _lex_bad),
    (m_emit_ignores_lexicon, _lex, _lex_bad),
    (m_priority_reversed, _pick, _pick_bad),
    (m_live_ignores_lexicon_prefix, _lex, _lex_bad),
    (m_ignored_needs_shift, _expr, _expr_bad),
    (m_killing_byte_dropped, _expr, _expr_bad),
    (m_eos_skips_finalize, _expr, _expr_bad),
    (m_reduce_pops_one_short, _expr, _expr_bad),
    (m_trailing_skips_parser, _expr, _expr_bad),
]


@pytest.mark.parametrize("mutate,make,check", CASES, ids=[c[0].__name__ for c in CASES])
def test_planted_mistake_is_caught(mutate, make, check):
    og = make()
    assert not check(og)  # the oracle as written passes
    mutate(og)
    assert check(og), "pins did not notice %s" % mutate.__name__


def test_dfa_liveness_mistake_is_caught():
    """The lexer DFA's live sets replaced by its accepting sets: the ``re`` pin
    (prefixes of literals are live) disagrees."""
    import re
    og = compile_grammar(grammar_text("sql"))
    og.dfa.live = [set(a) for a in og.dfa.acc]
    q = og.dfa.run(b"sel")
    select = og.g.term_ids["SELECT"]
    assert re.fullmatch(re.escape(b"select"), b"select")
    assert select not in og.dfa.live[q]  # while b"sel" is a prefix of the literal
