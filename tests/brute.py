"""Independent recognizer used only to pin the oracle.

Shares no code with ``oracle/``: its own reading of the grammar file, Python's
``re`` for the lexeme languages (classic longest match; equal to streaming
maximal munch on accept-closed lexers), the same contextual pick decided by a
textbook Earley recognizer (not an LR parser), and membership in L decided by a
complete Earley parse.  Prefix(L) is decided by searching completions from a
per-grammar candidate set that the calling test argues is sufficient.

Earley runs on the tag-filtered productions without useless-symbol
elimination; the grammars it is used on have no useless symbols after
filtering, so the language and the viable-prefix sets are unchanged.
"""
from __future__ import annotations

import re


def _unesc(s: str) -> bytes:
    out = bytearray()
    b = s.encode("latin-1")
    i = 0
    while i < len(b):
        if b[i] == 0x5C and i + 1 < len(b):
            out.append(b[i + 1])
            i += 2
        else:
            out.append(b[i])
            i += 1
    return bytes(out)


class BruteGrammar:
    def __init__(self, text: str, role=None, lexicons=None):
        self.names = []
        self.rx = []
        self.ignored = set()
        cats = []
        prods = []
        start = None
        for raw in text.splitlines():
            line = raw.strip()
            if not line or line[0] == "#":
                continue
            head = line.split()[0]
            if head in ("%token", "%ignore"):
                _, name, spec = line.split(None, 2)
                spec = spec.strip()
                if spec[0] == '"':
                    pat = re.escape(_unesc(spec[1:-1]))
                else:
                    pat = spec[1:-1].replace("\\/", "/").encode("latin-1")
                if head == "%ignore":
                    self.ignored.add(len(self.names))
                self.names.append(name)
                self.rx.append(re.compile(pat, re.DOTALL))
            elif head == "%category":
                cats.append(line.split()[1])
            elif head == "%start":
                start = line.split()[1]
            else:
                lhs, rhs = line.split("->")
                syms = rhs.split()
                tag = None
                if syms and syms[-1][0] == "@":
                    tag = syms[-1][1:]
                    syms = syms[:-1]
                if syms == ["%empty"]:
                    syms = []
                if tag is None or role is None or tag in set(role):
                    prods.append((lhs.strip(), tuple(syms)))
        ids = {n: i for i, n in enumerate(self.names)}
        self.cats = {ids[c] for c in cats}
        lexicons = lexicons or {}
        self.W = {ids[c]: {w if isinstance(w, bytes) else w.encode() for w in lexicons.get(c, [])}
                  for c in cats}
        self.prods = [("S'", (start,))] + [(l, tuple(ids.get(s, s) for s in r)) for l, r in prods]
        self.nts = {l for l, _ in self.prods}
        self.by_lhs = {}
        for i, (l, _) in enumerate(self.prods):
            self.by_lhs.setdefault(l, []).append(i)
        nullable = set()
        ch = True
        while ch:
            ch = False
            for l, r in self.prods:
                if l not in nullable and all(s in nullable for s in r):
                    nullable.add(l)
                    ch = True
        self.nullable = nullable

    # ---------------- Earley ----------------
    def earley_start(self):
        return [self._close(set([(0, 0, 0)]), 0, [])]

    def _close(self, items, k, sets):
        items = set(items)
        work = list(items)
        cur = items
        while work:
            p, d, o = work.pop()
            l, r = self.prods[p]
            new = []
            if d < len(r):
                X = r[d]
                if X in self.nts:
                    for q in self.by_lhs[X]:
                        new.append((q, 0, k))
                    if X in self.nullable:
                        new.append((p, d + 1, o))
            else:
                src = cur if o == k else sets[o]
                for (p2, d2, o2) in list(src):
                    r2 = self.prods[p2][1]
                    if d2 < len(r2) and r2[d2] == l:
                        new.append((p2, d2 + 1, o2))
            for it in new:
                if it not in cur:
                    cur.add(it)
                    work.append(it)
        return cur

    def scannable(self, sets):
        out = set()
        for p, d, o in sets[-1]:
            r = self.prods[p][1]
            if d < len(r) and r[d] not in self.nts:
                out.add(r[d])
        return out

    def scan(self, sets, t):
        k = len(sets) - 1
        moved = set()
        for p, d, o in sets[-1]:
            r = self.prods[p][1]
            if d < len(r) and r[d] == t:
                moved.add((p, d + 1, o))
        sets.append(self._close(moved, k + 1, sets))
        return sets

    def accepts_terms(self, sets):
        return (0, 1, 0) in sets[-1]

    # ---------------- lexing + membership ----------------
    def in_L(self, s: bytes) -> bool:
        """s in L: lex by longest match with the parser-viable contextual pick
        (viability = Earley can scan the terminal), then a complete parse."""
        sets = self.earley_start()
        pos, n = 0, len(s)
        while pos < n:
            best = 0
            for k in range(1, n - pos + 1):
                piece = s[pos:pos + k]
                if any(r.fullmatch(piece) for r in self.rx):
                    best = k
            if best == 0:
                return False
            lex = s[pos:pos + best]
            picked = None
            scan_ok = self.scannable(sets)
            for t in range(len(self.names)):
                if not self.rx[t].fullmatch(lex):
                    continue
                if t in self.cats and lex not in self.W[t]:
                    continue
                if t in self.ignored or t in scan_ok:
                    picked = t
                    break
            if picked is None:
                return False
            if picked not in self.ignored:
                self.scan(sets, picked)
            pos += best
        return self.accepts_terms(sets)

    def lexes_viably(self, s: bytes) -> bool:
        """The lexing of in_L succeeds to the end of s with every picked
        terminal scannable: the terminal string read so far is a viable
        prefix.  For an s that ends in a blank this is s in Prefix(L) on any
        grammar where each viable terminal string has a rendering that lexes
        back to it."""
        sets = self.earley_start()
        pos, n = 0, len(s)
        while pos < n:
            best = 0
            for k in range(1, n - pos + 1):
                if any(r.fullmatch(s[pos:pos + k]) for r in self.rx):
                    best = k
            if best == 0:
                return False
            lex = s[pos:pos + best]
            scan_ok = self.scannable(sets)
            picked = None
            for t in range(len(self.names)):
                if self.rx[t].fullmatch(lex) and not (t in self.cats and lex not in self.W[t]) \
                        and (t in self.ignored or t in scan_ok):
                    picked = t
                    break
            if picked is None:
                return False
            if picked not in self.ignored:
                self.scan(sets, picked)
            pos += best
        return True

    def in_prefix_L(self, s: bytes, completions) -> bool:
        return any(self.in_L(s + u) for u in completions)

    def terms_viable(self, term_ids):
        """Earley viable-prefix check of a terminal-id sequence; returns the
        list of scannable sets after each prefix (None once it dies)."""
        sets = self.earley_start()
        out = [self.scannable(sets)]
        for t in term_ids:
            if t not in out[-1]:
                return out, False
            self.scan(sets, t)
            out.append(self.scannable(sets))
        return out, self.accepts_terms(sets)
