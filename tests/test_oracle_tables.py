"""Pin the oracle's lexer DFA to Python's ``re`` and its LR(1) tables to an
Earley recognizer (both independent of ``oracle/``)."""
import re

import numpy as np
import pytest

from oracle import compile_grammar
from oracle.grammar import EmptyLanguage, Grammar, project
from tests.brute import BruteGrammar
from workloads import grammar_text

SQL_LEX = {"TABLE_NAME": ["employees", "employees_public", "orders"],
           "COLUMN_NAME": ["id", "name", "salary"]}


def _py_regexes(text):
    out = []
    for line in text.splitlines():
        p = line.split(None, 2)
        if len(p) == 3 and p[0] in ("%token", "%ignore"):
            spec = p[2].strip()
            if spec[0] == '"':
                lit = spec[1:-1].encode("latin-1").replace(b"\\\\", b"\\").replace(b'\\"', b'"')
                out.append(("lit", lit, re.compile(re.escape(lit), re.DOTALL)))
            else:
                out.append(("re", None, re.compile(spec[1:-1].encode("latin-1"), re.DOTALL)))
    return out


@pytest.mark.parametrize("name", ["expr", "sql", "lexfix"])
def test_dfa_matches_python_re(name):
    """acc(q(s)) = {tau : R_tau fullmatches s}; live(q(s)) = {tau : some
    extension of s fullmatches R_tau} (literal terminals: s is a prefix of the
    literal; the other regexes here need at most two more bytes from ``ext``)."""
    text = grammar_text(name)
    og = compile_grammar(text, lexicons=SQL_LEX if name == "sql" else None)
    pyr = _py_regexes(text)
    rng = np.random.default_rng(3)
    alpha = b"abcdefghijklmnopqrstuvwxyz_0123456789.'-;,()*=<>!+/% \n\t\"xz"
    ext = [b""] + [bytes([c]) for c in b"a_0.'- \n"] + [bytes([a, b]) for a in b"a0'-\n" for b in b"a0'-\n"]
    seeds = [l for k, l, _ in pyr if k == "lit"] + [b"select", b"emp_1", b"12.5", b"'ab c'", b"-- x", b"  \n"]
    strings = set()
    for _ in range(4000):
        if rng.random() < 0.5:
            s = seeds[int(rng.integers(len(seeds)))]
            s = s[:int(rng.integers(0, len(s) + 1))]
            if rng.random() < 0.5:
                s += bytes([alpha[int(rng.integers(len(alpha)))]])
        else:
            s = bytes(alpha[int(i)] for i in rng.integers(0, len(alpha), size=int(rng.integers(0, 6))))
        strings.add(s)
    for s in strings:
        q = og.dfa.run(s)
        acc = {t for t, (_, _, r) in enumerate(pyr) if r.fullmatch(s)}
        live = set()
        for t, (kind, lit, r) in enumerate(pyr):
            if kind == "lit":
                if lit.startswith(s):
                    live.add(t)
            elif any(r.fullmatch(s + e) for e in ext):
                live.add(t)
        assert set(og.dfa.acc[q]) == acc, (s, og.dfa.acc[q], acc)
        assert set(og.dfa.live[q]) == live, (s, og.dfa.live[q], live)
        assert (q == og.DEAD) == (not live and s != b"")


def _random_terms(bg: BruteGrammar, rng, max_depth):
    """A random sentence (as terminal ids) of the tag-filtered grammar."""
    # shortest-derivation heights so deep branches can terminate
    INF = 10 ** 9
    h = {n: INF for n in bg.nts}
    ch = True
    while ch:
        ch = False
        for l, r in bg.prods:
            v = 1 + max([h[s] if s in bg.nts else 0 for s in r] or [0])
            if v < h[l]:
                h[l] = v
                ch = True

    def expand(sym, d, out):
        if sym not in bg.nts:
            out.append(sym)
            return
        opts = [bg.prods[i][1] for i in bg.by_lhs[sym]]
        opts = [o for o in opts if all(h.get(s, 0) < INF for s in o)]
        if d >= max_depth:
            best = min(max([h[s] if s in bg.nts else 0 for s in o] or [0]) for o in opts)
            opts = [o for o in opts if max([h[s] if s in bg.nts else 0 for s in o] or [0]) == best]
        o = opts[int(rng.integers(len(opts)))]
        for s in o:
            expand(s, d + 1, out)

    out = []
    expand(bg.prods[0][1][0], 0, out)
    return out


@pytest.mark.parametrize("name,role", [("expr", None), ("sql", None), ("sql", []), ("lexfix", None), ("lexfix", [])])
def test_lr1_allowed_sets_match_earley(name, role):
    """For every prefix of random sentences and of their mutations:
    A(sigma) from LR(1) simulation equals Earley's scannable terminal set, the
    first terminal rejected by one is rejected by the other, and ACCEPT via the
    $end reduce chain equals a complete Earley parse."""
    text = grammar_text(name)
    og = compile_grammar(text, role=role, lexicons=SQL_LEX if name == "sql" else None)
    bg = BruteGrammar(text, role=role)
    rng = np.random.default_rng(17)
    nterm = og.n_term
    for it in range(60 if name == "sql" else 200):
        terms = _random_terms(bg, rng, 6 if name == "sql" else 8)
        if it % 2 == 1 and terms:
            i = int(rng.integers(len(terms)))
            k = rng.random()
            t = int(rng.integers(nterm))
            if t in og.ignored:
                t = 0
            if k < 0.4:
                terms[i] = t
            elif k < 0.7:
                terms.insert(i, t)
            else:
                del terms[i]
        scans, _ = bg.terms_viable(terms)
        stack = og.start_config().stack
        alive = True
        for j, t in enumerate(terms):
            A = og.allowed(stack)
            assert A == scans[j], (name, terms[:j + 1], A, scans[j])
            s = og.simulate(stack, t)
            if s is None or s[0] != "shift":
                assert t not in scans[j]
                alive = False
                break
            stack = s[1]
        if alive:
            ok_lr = og.simulate(stack, og.END)
            _, acc = bg.terms_viable(terms)
            assert (ok_lr is not None and ok_lr[0] == "accept") == acc, (name, terms)


def test_reduction_removes_useless_symbols():
    text = """%token A "a"
%token B "b"
%start s
s -> A x
s -> A
x -> B x
y -> B
s -> A z @r
z -> B
"""
    g = Grammar(text)
    prods = project(g, None)
    # x never terminates (non-generating) and y is unreachable
    assert ("s", ("A",)) in prods and ("s", ("A", "z")) in prods and ("z", ("B",)) in prods
    assert all(l not in ("x", "y") for l, _ in prods)
    prods2 = project(g, [])
    assert prods2 == [("s", ("A",))]
    with pytest.raises(EmptyLanguage):
        project(Grammar("%token A \"a\"\n%start s\ns -> A s\n"), None)
