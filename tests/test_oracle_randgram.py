"""Pin the oracle on random grammars of the statement family
(``workloads/randgram.py``) against the independent recognizer of
``tests/brute.py``: Python ``re`` longest match, the contextual pick decided
by Earley, and a complete Earley parse.

- EOS gate (Sec. 3.2): for random sentences, their cuts at random bytes,
  single-byte substitutions, insertions and deletions, and joins of two
  pieces, the oracle's EOS verdict equals membership in L.
- Viability (Def. 2): for the same strings, the oracle's verdict equals
  membership in Prefix(L), decided as follows.  In this family every viable
  terminal string has a rendering that lexes back to it (an identifier word
  that is no keyword or lexicon word, a column-only word beside every table
  word), so a string that ends in a blank is in Prefix(L) iff its lexing
  succeeds with every picked terminal scannable by Earley.  A string s is in
  Prefix(L) iff some completion x of its last lexeme keeps s + x + blank so:
  the completion a sentence continues with ends that lexeme as a keyword, a
  lexicon word (x a suffix of one), an identifier (x = "hhhhh" gives one
  that is no word, picked as an identifier as well) or a lexeme that is
  already whole (x empty); the blank ends it with the same emission.
- Each planted mistake of ``test_oracle_mutations`` disagrees with the
  recognizer on these grammars.
"""
import functools

import numpy as np
import pytest

from oracle import compile_grammar
from tests.brute import BruteGrammar
from tests.test_oracle_mutations import (m_eos_skips_finalize, m_emit_accepts_prefix_of_word,
                                         m_emit_ignores_lexicon, m_ignored_needs_shift, m_killing_byte_dropped,
                                         m_live_ignores_lexicon_prefix, m_priority_reversed,
                                         m_reduce_pops_one_short, m_trailing_skips_parser)
from workloads.randgram import LETTERS, RandGrammar, render

SEEDS = [0, 1, 2, 5, 6, 8, 11, 14]
MUTATIONS = [m_emit_accepts_prefix_of_word, m_emit_ignores_lexicon, m_priority_reversed,
             m_live_ignores_lexicon_prefix, m_ignored_needs_shift, m_killing_byte_dropped, m_eos_skips_finalize,
             m_reduce_pops_one_short, m_trailing_skips_parser]


def _strings(g, rng, role, n):
    alpha = g.alphabet()
    sents = [render(g.derive(rng, role, max_depth=int(rng.integers(3, 8))), rng) for _ in range(n)]
    out = []
    for s in sents:
        out.append(s)
        out.append(s[:int(rng.integers(0, len(s) + 1))])
        i = int(rng.integers(0, len(s)))
        c = bytes([alpha[int(rng.integers(len(alpha)))]])
        out.append(s[:i] + c + s[i + 1:])
        out.append(s[:i] + c)  # ends in the changed lexeme: trailing liveness decides
        out.append(s[:i] + c + s[i:])
        out.append(s[:i] + s[i + 1:])
    for k in range(n):
        a, b = sents[k], sents[(k + 1) % n]
        out.append(a[:int(rng.integers(0, len(a) + 1))] + b[int(rng.integers(0, len(b) + 1)):])
    return out


def _completions(g, s):
    """Completions of the last lexeme of s: empty, and when s ends in a run
    of letters r, the rest of every keyword or lexicon word that starts with
    r, and a tail that makes r an identifier that is no word."""
    k = len(s)
    while k and chr(s[k - 1]) in LETTERS:
        k -= 1
    r = s[k:].decode()
    out = [b""]
    if r:
        out.append(b"hhhhh")
        out += [w[len(r):].encode() for w in g.ident_words if w.startswith(r) and len(w) > len(r)]
    return out


@functools.lru_cache(maxsize=None)
def _case(seed):
    """The grammar, its role, the strings and the recognizer's verdicts
    (in L, in Prefix(L)) for one seed, computed once."""
    g = RandGrammar(seed)
    role = [] if seed % 2 else None
    bg = BruteGrammar(g.text(), role=role, lexicons=g.lexicons)
    strs = _strings(g, np.random.default_rng(seed + 31), role, 14)
    verd = [(bg.in_L(s), any(bg.lexes_viably(s + x + b" ") for x in _completions(g, s))) for s in strs]
    return g, role, strs, verd


def _disagreements(og, strs, verd):
    bad = []
    for s, (e_bf, v_bf) in zip(strs, verd):
        try:
            c = og.feed_bytes(og.start_config(), s)
            e_or = c is not None and og.eos_ok(c)
            v_or = c is not None and og.live_end(c)
        except Exception:  # a planted mistake may break the oracle outright
            e_or = v_or = None
        if e_or != e_bf:
            bad.append(("eos", s, e_or, e_bf))
        if v_or != v_bf:
            bad.append(("viable", s, v_or, v_bf))
    return bad


@pytest.mark.parametrize("seed", SEEDS)
def test_random_grammar_eos_and_viability_against_brute(seed):
    g, role, strs, verd = _case(seed)
    og = compile_grammar(g.text(), role, g.lexicons)
    bad = _disagreements(og, strs, verd)
    assert not bad, bad[:5]
    assert sum(e for e, _ in verd) >= 14 and sum(not v for _, v in verd) >= 5  # both verdicts occur


@pytest.mark.parametrize("mutate", MUTATIONS, ids=[m.__name__ for m in MUTATIONS])
def test_planted_mistake_is_caught_on_random_grammars(mutate):
    """Each planted mistake of ``test_oracle_mutations`` disagrees with the
    recognizer somewhere on these grammars."""
    n = 0
    for seed in SEEDS:
        g, role, strs, verd = _case(seed)
        og = compile_grammar(g.text(), role, g.lexicons)
        mutate(og)
        n += len(_disagreements(og, strs, verd))
    assert n > 0, mutate.__name__
