"""Grammar text, L2 role projection and reduction (GRID Sec. 2, layers L1/L2).

Test infrastructure (see package docstring).

File format, one declaration per line ('#' starts a comment line):
  %token NAME "literal" | %token NAME /regex/   terminal; line order = priority
  %ignore NAME /regex/                           ignored terminal (the set I)
  %category NAME                                 L3 lexicon category
  %start SYMBOL
  lhs -> X Y Z [@tag]                            production ('%empty' = epsilon)

Role projection (Sec. 2, L2): keep the productions whose tag is absent or listed
in the role; then *mandatory* useless-symbol elimination -- drop non-generating
nonterminals, then everything unreachable from the start symbol -- and verify
that the language is non-empty (the start symbol generates).
"""
from __future__ import annotations


class GrammarError(ValueError):
    pass


class EmptyLanguage(GrammarError):
    pass


def _unescape_literal(s: str) -> bytes:
    out = bytearray()
    i = 0
    b = s.encode("latin-1")
    while i < len(b):
        if b[i] == 0x5C and i + 1 < len(b):
            out.append(b[i + 1])
            i += 2
        else:
            out.append(b[i])
            i += 1
    return bytes(out)


class Grammar:
    """Parsed L1 grammar.

    terminals: list of (name, kind in {'token','ignore'}, ('lit', bytes) | ('re', bytes))
    productions: list of (lhs, rhs tuple, tag or None)"""

    def __init__(self, text: str):
        self.terminals = []
        self.categories = []
        self.productions = []
        self.start = None
        for raw in text.splitlines():
            line = raw.strip()
            if not line or line.startswith("#"):
                continue
            if line.startswith("%token") or line.startswith("%ignore"):
                kind = "token" if line.startswith("%token") else "ignore"
                rest = line.split(None, 1)[1]
                name, spec = rest.split(None, 1)
                spec = spec.strip()
                if spec.startswith('"') and spec.endswith('"') and len(spec) >= 2:
                    pat = ("lit", _unescape_literal(spec[1:-1]))
                elif spec.startswith("/") and spec.endswith("/") and len(spec) >= 2:
                    pat = ("re", spec[1:-1].replace("\\/", "/").encode("latin-1"))
                else:
                    raise GrammarError("bad terminal spec: " + line)
                if any(t[0] == name for t in self.terminals):
                    raise GrammarError("duplicate terminal " + name)
                self.terminals.append((name, kind, pat))
            elif line.startswith("%category"):
                self.categories.append(line.split()[1])
            elif line.startswith("%start"):
                self.start = line.split()[1]
            elif "->" in line:
                lhs, rhs = line.split("->", 1)
                lhs = lhs.strip()
                toks = rhs.split()
                tag = None
                if toks and toks[-1].startswith("@"):
                    tag = toks[-1][1:]
                    toks = toks[:-1]
                if toks == ["%empty"]:
                    toks = []
                self.productions.append((lhs, tuple(toks), tag))
            else:
                raise GrammarError("cannot parse line: " + line)
        if self.start is None:
            raise GrammarError("no %start")
        self.term_ids = {t[0]: i for i, t in enumerate(self.terminals)}
        for c in self.categories:
            if c not in self.term_ids:
                raise GrammarError("category is not a terminal: " + c)
        nts = {p[0] for p in self.productions}
        for lhs, rhs, _ in self.productions:
            for s in rhs:
                if s not in nts and s not in self.term_ids:
                    raise GrammarError("unknown symbol " + s)
                if s in self.term_ids and self.terminals[self.term_ids[s]][1] == "ignore":
                    raise GrammarError("ignored terminal used in a production: " + s)


def project(g: Grammar, role):
    """L2 projection + reduction.  ``role`` = None keeps every production,
    otherwise an iterable of kept tags (untagged productions are always kept).
    Returns the reduced production list [(lhs, rhs)]; raises EmptyLanguage."""
    keep = None if role is None else set(role)
    prods = [(l, r) for (l, r, tag) in g.productions if tag is None or keep is None or tag in keep]
    is_term = g.term_ids.__contains__
    # generating nonterminals: fixpoint
    gen = set()
    changed = True
    while changed:
        changed = False
        for l, r in prods:
            if l not in gen and all(is_term(s) or s in gen for s in r):
                gen.add(l)
                changed = True
    if g.start not in gen:
        raise EmptyLanguage("the projected grammar generates no sentence")
    prods = [(l, r) for l, r in prods if l in gen and all(is_term(s) or s in gen for s in r)]
    # reachable from the start symbol: fixpoint
    reach = {g.start}
    changed = True
    while changed:
        changed = False
        for l, r in prods:
            if l in reach:
                for s in r:
                    if not is_term(s) and s not in reach:
                        reach.add(s)
                        changed = True
    return [(l, r) for l, r in prods if l in reach]
