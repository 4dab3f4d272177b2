"""Seeded random grammars for randomized parity.

Each seed draws one grammar of a statement family: statements led by their own
keyword, bodies of expressions, comma lists and optional clauses joined by
separator keywords, a precedence ladder of one to three binary-operator levels
with unary operators, parentheses and function calls, nested statement blocks,
productions tagged for a role, and optionally two identifier categories that
share the identifier regex (a qualified or bare column, so that both are
viable at one point and the declaration order decides a shared word).  The
family is LALR(1) by construction; both compilers still check it.

Keywords are drawn from the identifier alphabet, so a keyword is also an
identifier word and the contextual pick decides between them.  Sentences are
rendered by top-down derivation from the grammar's own production list, with a
depth bound that switches to the shortest productions; identifiers avoid the
keyword spellings so that every rendered sentence is in the language.  Nothing
here lexes or parses.
"""
from __future__ import annotations

import numpy as np

from workloads.gen import GreedyTokenizer

LETTERS = "abcdefgh"
OPS = "+-*/%<>=&|^!~:?"


class RandGrammar:
    """One drawn grammar: terminal declarations, productions, lexicons."""

    def __init__(self, seed: int):
        rng = np.random.default_rng(seed)
        self.seed = seed
        self.terms = []     # (name, "lit"/"re"/"ign", text), in declaration (priority) order
        self.prods = []     # (lhs, [rhs symbols], tag or None)
        self.lit = {}       # terminal name -> its literal spelling
        self.cats = bool(rng.random() < 0.6)
        words = set()

        def word(lo, hi):
            while True:
                w = "".join(LETTERS[int(i)] for i in rng.integers(0, len(LETTERS), size=int(rng.integers(lo, hi + 1))))
                if w not in words:
                    words.add(w)
                    return w

        def kw():
            name = "K%d" % len(self.lit)
            self.lit[name] = word(1, 3)
            return name

        ops = list(rng.permutation(list(OPS)))
        n_lev = int(rng.integers(1, 4))
        n_stmt = int(rng.integers(2, 5))
        # expression ladder: e{i} -> e{i} op e{i+1} | e{i+1} for i < L; e{L} -> op e{L} | p (unary operators)
        lev_ops = [[ops.pop() for _ in range(int(rng.integers(1, 3)))] for _ in range(n_lev)]
        for i, os_ in enumerate(lev_ops):
            for o in os_:
                self.lit.setdefault("O" + str(OPS.index(o)), o)
                self.prods.append(("e%d" % i, ["e%d" % i, "O" + str(OPS.index(o)), "e%d" % (i + 1)], None))
            self.prods.append(("e%d" % i, ["e%d" % (i + 1)], None))
        un = [ops.pop() for _ in range(int(rng.integers(0, 2)))]
        if rng.random() < 0.5:
            un.append(lev_ops[0][0])  # a binary operator that is also unary
        for o in un:
            self.lit.setdefault("O" + str(OPS.index(o)), o)
            self.prods.append(("e%d" % n_lev, ["O" + str(OPS.index(o)), "e%d" % n_lev], None))
        self.prods.append(("e%d" % n_lev, ["p"], None))
        self.prods += [("p", ["ID"], None), ("p", ["NUM"], None), ("p", ["LP", "e0", "RP"], None)]
        if rng.random() < 0.7:
            fn = kw()
            self.prods += [("p", [fn, "LP", "args", "RP"], None), ("args", [], None), ("args", ["al"], None),
                           ("al", ["al", "COMMA", "e0"], None), ("al", ["e0"], None)]
        # statements
        self.prods += [("prog", ["ss"], None), ("ss", ["ss", "st"], None), ("ss", ["st"], None)]
        for j in range(n_stmt):
            lead = kw()
            tag = "adm" if j == n_stmt - 1 and n_stmt > 2 and rng.random() < 0.5 else None
            self.prods.append(("st", ["s%d" % j], tag))
            body = []
            for k in range(int(rng.integers(1, 4))):
                if k:
                    body.append(kw())
                kind = rng.choice(["e", "l", "o", "c"] if self.cats else ["e", "l", "o"])
                if kind == "e":
                    body.append("e0")
                elif kind == "l":
                    lst, el = "l%d_%d" % (j, k), "m%d_%d" % (j, k)
                    self.prods += [(lst, [lst, "COMMA", el], None), (lst, [el], None)]
                    if self.cats and rng.random() < 0.5:
                        self.prods += [(el, ["CO"], None), (el, ["TA", "DOT", "CO"], None)]
                    else:
                        self.prods.append((el, ["e0"], None))
                    body.append(lst)
                elif kind == "o":
                    opt = "o%d_%d" % (j, k)
                    self.prods += [(opt, [], None), (opt, [kw(), "e0"], None)]
                    body.append(opt)
                else:
                    body.append("CO")
            self.prods.append(("s%d" % j, [lead] + body + ["SEMI"], None))
        if rng.random() < 0.7:  # nested blocks: deep stacks
            blk = kw()
            self.prods += [("st", ["b"], None), ("b", [blk, "LP", "ss", "RP"], None)]
        # lexicons: shared words are read as TA (declared first) where both fit
        self.lexicons = {}
        if self.cats:
            ta = [word(1, 3) for _ in range(int(rng.integers(2, 6)))]
            co = [word(1, 3) for _ in range(int(rng.integers(2, 6)))]
            shared = [ta[int(i)] for i in rng.integers(0, len(ta), size=int(rng.integers(1, 3)))]
            self.lexicons = {"TA": sorted(set(ta)), "CO": sorted(set(co) | set(shared))}
        self.ident_words = words  # every keyword and lexicon word: identifiers avoid them
        # declarations, in priority order: keywords, punctuation, categories, identifiers
        for name in sorted(self.lit, key=lambda n: (n[0] != "K", int(n[1:]))):
            self.terms.append((name, "lit", self.lit[name]))
        self.terms += [("LP", "lit", "("), ("RP", "lit", ")"), ("COMMA", "lit", ","), ("SEMI", "lit", ";"),
                       ("DOT", "lit", ".")]
        for name, txt in (("LP", "("), ("RP", ")"), ("COMMA", ","), ("SEMI", ";"), ("DOT", ".")):
            self.lit[name] = txt
        if self.cats:
            self.terms += [("TA", "re", "[%s]+" % LETTERS), ("CO", "re", "[%s]+" % LETTERS)]
        self.terms += [("ID", "re", "[%s]+" % LETTERS), ("NUM", "re", "[0-9]+"), ("WS", "ign", "[ ]+")]
        used = {s for _, r, _ in self.prods for s in r}
        self.terms = [t for t in self.terms if t[0] in used or t[1] == "ign"]
        self.lexicons = {c: w for c, w in self.lexicons.items() if c in used}
        self.cats = bool(self.lexicons)
        self.nts = sorted({p[0] for p in self.prods})
        self._heights()

    # ---- text ---------------------------------------------------------------
    def text(self) -> str:
        out = ["# random statement grammar, seed %d" % self.seed]
        for name, kind, txt in self.terms:
            if kind == "lit":
                out.append('%%token %s "%s"' % (name, txt))
            elif kind == "re":
                out.append("%%token %s /%s/" % (name, txt))
            else:
                out.append("%%ignore %s /%s/" % (name, txt))
        out += ["%%category %s" % c for c in ("TA", "CO") if c in self.lexicons]
        out.append("%start prog")
        for lhs, rhs, tag in self.prods:
            out.append("%s -> %s%s" % (lhs, " ".join(rhs) if rhs else "%empty", " @" + tag if tag else ""))
        return "\n".join(out) + "\n"

    def alphabet(self) -> bytes:
        s = set(LETTERS) | set("0123456789 ")
        for t in self.lit.values():
            s |= set(t)
        return bytes(sorted(ord(c) for c in s))

    # ---- derivation ---------------------------------------------------------
    def _heights(self):
        """Least derivation height of every symbol (terminals 0)."""
        INF = 1 << 30
        h = {n: INF for n in self.nts}
        changed = True
        while changed:
            changed = False
            for lhs, rhs, _ in self.prods:
                v = 1 + max([h.get(s, 0) for s in rhs], default=0)
                if v < h[lhs]:
                    h[lhs] = v
                    changed = True
        self.height = h

    def _prods_of(self, nt, role):
        return [p for p in self.prods if p[0] == nt and (p[2] is None or role is None or p[2] in role)]

    def derive(self, rng, role=None, max_depth=10):
        """A random sentence as a list of (terminal, lexeme text)."""
        out = []

        def go(sym, d):
            if sym not in self.height:
                out.append((sym, self._lexeme(rng, sym, out)))
                return
            ps = self._prods_of(sym, role)
            if d >= max_depth:
                best = min(1 + max([self.height.get(s, 0) for s in p[1]], default=0) for p in ps)
                ps = [p for p in ps if 1 + max([self.height.get(s, 0) for s in p[1]], default=0) == best]
            p = ps[int(rng.integers(0, len(ps)))]
            for s in p[1]:
                go(s, d + 1)

        go("prog", 0)
        return out

    def _lexeme(self, rng, term, before):
        if term in self.lit:
            return self.lit[term]
        if term == "NUM":
            return str(int(rng.integers(0, 1000)))
        if term == "TA":
            return self.lexicons["TA"][int(rng.integers(0, len(self.lexicons["TA"])))]
        if term == "CO":
            if before and before[-1][0] == "DOT":
                pool = self.lexicons["CO"]
            else:  # a bare column: a word that is not also a table (the table reading comes first)
                pool = [w for w in self.lexicons["CO"] if w not in self.lexicons.get("TA", ())] or None
                if pool is None:
                    raise ValueError("no column-only word")
            return pool[int(rng.integers(0, len(pool)))]
        while True:  # ID: a word that is no keyword or lexicon word
            w = "".join(LETTERS[int(i)] for i in rng.integers(0, len(LETTERS), size=int(rng.integers(1, 5))))
            if w not in self.ident_words:
                return w


def render(lexemes, rng) -> bytes:
    """Join lexemes with random blanks; a blank is forced between two words or
    two numbers (which would otherwise merge into one lexeme)."""
    out = []
    prev = None
    for _, t in lexemes:
        if prev is not None:
            merge = (prev[-1].isalpha() and t[0].isalpha()) or (prev[-1].isdigit() and t[0].isdigit())
            n = int(rng.choice([0, 0, 1, 1, 2]))
            out.append(" " * max(n, 1 if merge else 0))
        out.append(t)
        prev = t
    return "".join(out).encode()


def rand_vocab(rng, V: int, alpha: bytes, corpus, n_alias: int = 4):
    """V ids: the alphabet's single bytes, substrings (2-10 bytes) of the
    corpus sentences for half of the rest (spellings that cross lexeme
    boundaries, as merged tokenizer pieces do), random strings (2-5 bytes)
    over the alphabet for the other half, ``n_alias`` duplicate spellings, and
    EOS as the last id."""
    toks = [bytes([c]) for c in alpha]
    seen = set(toks)
    n_rand = V - 1 - len(alpha) - n_alias
    target = len(alpha) + n_rand
    n_sub = n_rand // 2
    tries = 0
    while len(toks) < len(alpha) + n_sub and tries < 50 * V:
        tries += 1
        s = corpus[int(rng.integers(0, len(corpus)))]
        if len(s) < 2:
            continue
        L = int(rng.integers(2, min(10, len(s)) + 1))
        a = int(rng.integers(0, len(s) - L + 1))
        piece = s[a:a + L]
        if piece not in seen:
            seen.add(piece)
            toks.append(piece)
    while len(toks) < target:
        L = int(rng.integers(2, 6))
        s = bytes(alpha[int(i)] for i in rng.integers(0, len(alpha), size=L))
        if s not in seen:
            seen.add(s)
            toks.append(s)
    for _ in range(n_alias):
        toks.append(toks[int(rng.integers(len(alpha), len(toks)))])
    order = rng.permutation(len(toks))
    toks = [toks[i] for i in order]
    eos = len(toks)
    toks.append(b"<eos>")
    return toks, eos


def rand_grammar_workload(seed: int, B: int = 24, V: int = 1500, role=None):
    """One random grammar with a vocabulary of V ids and B prefixes: the empty
    prefix, whole sentences (EOS admitted), and sentences cut at a uniformly
    random byte offset, tokenized by greedy longest match."""
    g = RandGrammar(seed)
    rng = np.random.default_rng(seed + 7919)
    corpus = [render(g.derive(rng, role), rng) for _ in range(120)]
    toks, eos = rand_vocab(rng, V, g.alphabet(), corpus)
    tk = GreedyTokenizer(toks, [eos])
    prefixes, texts = [[]], [b""]
    for k in range(1, B):
        s = render(g.derive(rng, role, max_depth=int(rng.integers(4, 14))), rng)
        cut = len(s) if k % 6 == 1 else int(rng.integers(0, len(s) + 1))
        texts.append(s[:cut])
        prefixes.append(tk.encode(s[:cut]))
    return dict(name="rand_%d" % seed, grammar=g.text(), role=role, lexicons=g.lexicons, tokens=toks, eos=eos,
                specials=[], prefixes=prefixes, texts=texts, B=B, seed=seed, sentences=corpus)
