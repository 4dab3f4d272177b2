"""Seeded generators: identifier names, byte vocabularies, sentences, greedy tokenizer.

All randomness comes from ``numpy.random.default_rng(seed)``.  Nothing here
lexes or parses: sentences are rendered directly from hand-written productions
of the two workload languages (the expression language and the SQL subset), and
the tokenizer is a plain greedy longest-match over the vocabulary's spellings.
"""
from __future__ import annotations

import numpy as np

# --------------------------------------------------------------------------
# identifier names
# --------------------------------------------------------------------------
_ONSETS = ["b", "c", "d", "f", "g", "h", "j", "k", "l", "m", "n", "p", "r", "s",
           "t", "v", "w", "z", "ch", "sh", "th", "br", "cr", "dr", "gr", "pr",
           "st", "tr", "pl", "kl", "sp", "qu"]
_VOWELS = ["a", "e", "i", "o", "u", "ai", "ea", "io", "ou", "ee", "oa"]
_CODAS = ["", "", "", "n", "r", "s", "t", "l", "m", "x", "nd", "st", "rk", "ng"]


def syllables(seed: int = 7, n: int = 320) -> list[str]:
    """A seeded inventory of distinct pronounceable syllables (2-5 letters)."""
    rng = np.random.default_rng(seed)
    out, seen = [], set()
    while len(out) < n:
        s = (_ONSETS[rng.integers(len(_ONSETS))] + _VOWELS[rng.integers(len(_VOWELS))]
             + _CODAS[rng.integers(len(_CODAS))])
        if s not in seen and 2 <= len(s) <= 5:
            seen.add(s)
            out.append(s)
    return out


def snake_names(rng, syl: list[str], count: int, exclude: set, parts=(1, 3)) -> list[str]:
    """``count`` distinct snake_case names of ``parts`` syllable groups, none in ``exclude``."""
    out, seen = [], set(exclude)
    tries = 0
    while len(out) < count:
        tries += 1
        if tries > 200 * count + 10000:
            raise RuntimeError("name space exhausted")
        k = int(rng.integers(parts[0], parts[1] + 1))
        groups = []
        for _ in range(k):
            g = syl[rng.integers(len(syl))]
            if rng.random() < 0.3:
                g += syl[rng.integers(len(syl))]
            groups.append(g)
        name = "_".join(groups)
        if rng.random() < 0.05:
            name += str(int(rng.integers(1, 10)))
        if name in seen or len(name) > 40:
            continue
        seen.add(name)
        out.append(name)
    return out


def make_schema(seed: int, n_tables: int, n_cols: int, keywords, col_pool: int | None = None,
                shared: int = 0):
    """Return (tables, table->columns dict, sorted distinct column words).

    Names never equal a keyword.  Tables and columns are disjoint, except that
    with ``shared`` > 0 that many column names are also table names (real
    catalogs have a column ``order`` beside a table ``order``).  ``col_pool``
    bounds the distinct column names (columns repeat across tables, as real
    catalogs do); ``None`` makes every column name distinct."""
    rng = np.random.default_rng(seed)
    syl = syllables()
    kw = set(keywords)
    tables = snake_names(rng, syl, n_tables, kw, parts=(1, 2))
    pool_n = n_tables * n_cols if col_pool is None else col_pool
    pool = snake_names(rng, syl, pool_n, kw | set(tables), parts=(1, 3))
    if shared:
        pick = rng.choice(len(tables), size=min(shared, len(tables), pool_n), replace=False)
        for k, j in enumerate(sorted(int(x) for x in pick)):
            pool[k] = tables[j]
    cols = {}
    if col_pool is None:
        for i, t in enumerate(tables):
            cols[t] = pool[i * n_cols:(i + 1) * n_cols]
    else:
        for t in tables:
            idx = rng.choice(len(pool), size=n_cols, replace=False)
            cols[t] = [pool[j] for j in idx]
    words = sorted({c for cs in cols.values() for c in cs})
    return tables, cols, words


# --------------------------------------------------------------------------
# sentences
# --------------------------------------------------------------------------
def render(lexemes, rng, ws_rate=0.08, nl_rate=0.03, comment_rate=0.0) -> str:
    """Join lexemes with blanks.  Punctuation that cannot merge with a
    neighbour ( ( ) , ; . ) is sometimes written without a blank; every other
    pair gets at least one blank so no two lexemes run together."""
    tight_after = {"(", "."}
    tight_before = {")", ",", ";", ".", "("}
    out = []
    prev = None
    for lx in lexemes:
        if prev is not None:
            if lx == "." or prev == ".":
                sep = ""
            elif (lx in tight_before or prev in tight_after) and rng.random() < 0.6:
                sep = ""
            else:
                r = rng.random()
                if r < comment_rate:
                    sep = " -- " + "x" * int(rng.integers(0, 6)) + "\n"
                elif r < comment_rate + nl_rate:
                    sep = "\n" + " " * int(rng.integers(0, 5))
                elif r < comment_rate + nl_rate + ws_rate:
                    sep = " " * int(rng.integers(2, 4))
                else:
                    sep = " "
            out.append(sep)
        out.append(lx)
        prev = lx
    return "".join(out)


def expr_sentence(rng, max_depth: int = 8, depth: int = 0) -> str:
    """A random sentence of E -> E+T|T, T -> T*F|F, F -> (E)|id|num with random blanks."""
    lex = _expr_e(rng, max_depth, depth)
    out = []
    for i, t in enumerate(lex):
        if i:
            out.append(" " * int(rng.choice([0, 0, 1, 1, 2])))
        out.append(t)
    return "".join(out)


def _expr_e(rng, md, d):
    terms = [_expr_t(rng, md, d)]
    while rng.random() < 0.4:
        terms.append(_expr_t(rng, md, d))
    out = []
    for i, t in enumerate(terms):
        if i:
            out.append("+")
        out.extend(t)
    return out


def _expr_t(rng, md, d):
    fs = [_expr_f(rng, md, d)]
    while rng.random() < 0.35:
        fs.append(_expr_f(rng, md, d))
    out = []
    for i, f in enumerate(fs):
        if i:
            out.append("*")
        out.extend(f)
    return out


def _expr_f(rng, md, d):
    r = rng.random()
    if d < md and r < 0.3:
        return ["("] + _expr_e(rng, md, d + 1) + [")"]
    if r < 0.65:
        return ["".join(chr(97 + int(x)) for x in rng.integers(0, 26, size=int(rng.integers(1, 4))))]
    return [str(int(rng.integers(0, 1000)))]


class SqlGen:
    """Random statements of the SQL subset, as lexeme lists.

    ``dml`` enables INSERT/UPDATE/DELETE statements (the admin role)."""

    AGG = ["count", "sum", "avg", "min", "max"]
    CMP = ["=", "<>", "!=", "<", ">", "<=", ">="]

    def __init__(self, rng, tables, cols, dml: bool):
        self.rng = rng
        self.tables = tables
        self.cols = cols
        # a column name that is also a table name is written qualified
        # (t.c) where a bare column may stand: there both categories are
        # parser-viable and the earlier-declared TABLE_NAME is picked
        ts = set(tables)
        self.all_cols = sorted({c for cs in cols.values() for c in cs} - ts)
        self.dml = dml

    def _p(self, p):
        return self.rng.random() < p

    def _pick(self, seq):
        return seq[int(self.rng.integers(len(seq)))]

    def table(self):
        return self._pick(self.tables)

    def column(self):
        if self._p(0.2):
            t = self.table()
            return [t, ".", self._pick(self.cols[t])]
        return [self._pick(self.all_cols)]

    def number(self):
        if self._p(0.2):
            return str(int(self.rng.integers(0, 100))) + "." + str(int(self.rng.integers(0, 100)))
        return str(int(self.rng.integers(0, 100000)))

    def string(self):
        n = int(self.rng.integers(0, 8))
        body = "".join(self._pick("abcdefgh ijk") for _ in range(n))
        return "'" + body + "'"

    def primary(self, d):
        r = self.rng.random()
        if d > 0 and r < 0.08:
            return ["("] + self.expr(d - 1) + [")"]
        if d > 0 and r < 0.12:
            return ["("] + self.select(d - 1) + [")"]
        if r < 0.2:
            arg = ["*"] if self._p(0.3) else (["distinct"] + self.expr(0) if self._p(0.2) else self.expr(0))
            return [self._pick(self.AGG), "("] + arg + [")"]
        if r < 0.65:
            return self.column()
        if r < 0.85:
            return [self.number()]
        if r < 0.95:
            return [self.string()]
        return [self._pick(["true", "false", "null"])]

    def factor(self, d):
        if self._p(0.05):
            return ["-"] + self.factor(d)
        return self.primary(d)

    def term(self, d):
        out = self.factor(d)
        while self._p(0.15):
            out += [self._pick(["*", "/", "%"])] + self.factor(d)
        return out

    def arith(self, d):
        out = self.term(d)
        while self._p(0.2):
            out += [self._pick(["+", "-"])] + self.term(d)
        return out

    def pred(self, d):
        r = self.rng.random()
        if d > 0 and r < 0.06:
            return self.arith(d) + (["not"] if self._p(0.3) else []) + ["in", "("] + self.select(d - 1) + [")"]
        if d > 0 and r < 0.09:
            return ["exists", "("] + self.select(d - 1) + [")"]
        if r < 0.15:
            return self.arith(d) + ["is"] + (["not"] if self._p(0.5) else []) + ["null"]
        if r < 0.2:
            return self.arith(d) + ["like", self.string()]
        if r < 0.85:
            return self.arith(d) + [self._pick(self.CMP)] + self.arith(d)
        return self.arith(d)

    def not_expr(self, d):
        if self._p(0.08):
            return ["not"] + self.not_expr(d)
        return self.pred(d)

    def expr(self, d, min_preds: int = 1):
        out = self.not_expr(d)
        n = 1
        while n < min_preds or self._p(0.25):
            out += [self._pick(["and", "and", "or"])] + self.not_expr(d)
            n += 1
        return out

    def select(self, d, where_preds: int = 0):
        out = ["select"]
        if self._p(0.1):
            out.append("distinct")
        if self._p(0.2):
            out.append("*")
        else:
            out += self.expr(0)
            while self._p(0.4):
                out += [","] + self.expr(0)
        out.append("from")
        out += self.table_ref(d)
        while self._p(0.1):
            out += [","] + self.table_ref(d)
        if where_preds or self._p(0.7):
            out += ["where"] + self.expr(d, max(1, where_preds))
        if self._p(0.15):
            out += ["group", "by"] + self.column()
            while self._p(0.3):
                out += [","] + self.column()
            if self._p(0.3):
                out += ["having"] + self.expr(0)
        if self._p(0.2):
            out += ["order", "by"] + self.expr(0) + ([self._pick(["asc", "desc"])] if self._p(0.5) else [])
            while self._p(0.3):
                out += [","] + self.expr(0)
        if self._p(0.15):
            out += ["limit", str(int(self.rng.integers(1, 1000)))]
        return out

    def table_ref(self, d):
        out = [self.table()]
        while self._p(0.15):
            out += ([self._pick(["inner", "left"])] if self._p(0.5) else []) + ["join", self.table(), "on"] + self.expr(0)
        return out

    def statement(self, d: int = 2, where_preds: int = 0):
        if self.dml and self._p(0.35):
            k = int(self.rng.integers(3))
            t = self.table()
            if k == 0:
                cs = [self._pick(self.cols[t]) for _ in range(int(self.rng.integers(1, 4)))]
                out = ["insert", "into", t, "("]
                for i, c in enumerate(cs):
                    out += ([","] if i else []) + [c]
                out += [")", "values", "("]
                for i in range(len(cs)):
                    out += ([","] if i else []) + self.expr(0)
                out += [")"]
            elif k == 1:
                out = ["update", t, "set", self._pick(self.cols[t]), "="] + self.expr(0)
                while self._p(0.3):
                    out += [",", self._pick(self.cols[t]), "="] + self.expr(0)
                if where_preds or self._p(0.7):
                    out += ["where"] + self.expr(d, max(1, where_preds))
            else:
                out = ["delete", "from", t]
                if where_preds or self._p(0.7):
                    out += ["where"] + self.expr(d, max(1, where_preds))
            return out + [";"]
        return self.select(d, where_preds) + [";"]

    def nested_chain(self, depth: int, n_preds: int):
        """``depth`` levels of nesting opened first (parenthesised expressions
        or IN-subqueries), then a left-recursive AND/OR chain of ``n_preds``
        simple predicates; the statement is closed afterwards."""
        out = ["select", self._pick(self.all_cols), "from", self.table(), "where"]
        closers = []
        for _ in range(depth):
            if self._p(0.25):
                out += [self._pick(self.all_cols), "in", "(", "select", self._pick(self.all_cols),
                        "from", self.table(), "where"]
            else:
                out += ["("]
            closers.append(")")
        for i in range(n_preds):
            if i:
                out.append(self._pick(["and", "and", "or"]))
            out += self.arith(0) + [self._pick(self.CMP)] + self.arith(0)
        return out + closers + [";"]


def pick_sentence(rng) -> str:
    """A random sentence of the pick grammar (q -> g cols o TABLE ;, a column
    bare or qualified) over the lexicons TABLE {ab, abc, ba} and COLUMN
    {a, ab, c}, with random blanks.  Bare columns are the column-only words;
    the shared word "ab" appears as a table of a qualified column or after "."."""
    cols = []
    for _ in range(int(rng.integers(1, 4))):
        if rng.random() < 0.5:
            cols.append([["a", "c"][int(rng.integers(2))]])
        else:
            cols.append([["ab", "abc", "ba"][int(rng.integers(3))], ".", ["a", "ab", "c"][int(rng.integers(3))]])
    lex = ["g"]
    for i, c in enumerate(cols):
        if i:
            lex.append(",")
        lex.extend(c)
    lex += ["o", ["ab", "abc", "ba"][int(rng.integers(3))], ";"]
    out = []
    for i, t in enumerate(lex):
        if i:
            out.append(" " * int(rng.choice([0, 0, 1, 2])))
        out.append(t)
    return "".join(out)


# --------------------------------------------------------------------------
# vocabularies
# --------------------------------------------------------------------------
def _zipf_lengths(alpha: float, lo: int, hi: int):
    ls = np.arange(lo, hi + 1)
    w = ls.astype(np.float64) ** (-alpha)
    return ls, w / w.sum()


_PUNCT = "(),;.*=<>!+-/%'"


def sql_vocab(seed: int, V: int, keywords, multiword_frac: float = 0.0,
              sentence_src=None, n_special: int = 2, alias_frac: float = 0.001):
    """A BPE-like byte vocabulary of exactly ``V`` ids.

    Contents: the 256 single bytes (byte-complete), keyword fragments, pieces of
    identifiers built from the shared syllable inventory, blank runs,
    punctuation clusters, digit runs, unrelated printable/high-byte strings and,
    when ``multiword_frac`` > 0, windows of rendered sentences that cross lexeme
    boundaries.  Lengths are 1..16 with P(l) ~ l^-1.1, resampled when a length
    class saturates.  ``alias_frac`` of the ids duplicate an earlier spelling.
    Ids are shuffled; the last ``n_special`` + 1 ids are the special tokens and
    EOS (EOS = V-1).  Returns (list of bytes per id, eos_id, special_ids)."""
    rng = np.random.default_rng(seed)
    syl = syllables()
    kws = list(keywords)
    n_alias = int(round(alias_frac * V))
    n_plain = V - 1 - n_special - n_alias
    spell = [bytes([b]) for b in range(256)]
    seen = set(spell)
    ls, pl = _zipf_lengths(1.1, 1, 16)
    saturated = np.zeros(len(ls), dtype=bool)
    fails = np.zeros(len(ls), dtype=np.int64)
    cats = ["syl", "junk", "kw", "digit", "punct", "ws", "multi"]
    cw = np.array([0.46, 0.2, 0.1, 0.06, 0.09, 0.03, multiword_frac * 3.0])
    cw = cw / cw.sum()
    windows = sentence_src if sentence_src is not None else []

    def gen(cat, L):
        sp = " " if rng.random() < 0.45 else ""
        if cat == "syl":
            s = sp + ("_" if rng.random() < 0.1 else "")
            while len(s) < L:
                s += syl[rng.integers(len(syl))]
                if rng.random() < 0.15:
                    s += "_"
            return s[:L]
        if cat == "kw":
            k = kws[rng.integers(len(kws))]
            s = sp + k
            if rng.random() < 0.5:
                a = int(rng.integers(0, len(s)))
                s = s[a:]
            while len(s) < L:
                s += " " + kws[rng.integers(len(kws))]
            return s[:L]
        if cat == "digit":
            s = sp + "".join(str(int(d)) for d in rng.integers(0, 10, size=L))
            if rng.random() < 0.1 and L > 2:
                s = s[:L - 1] + "."
            return s[:L]
        if cat == "punct":
            return "".join(_PUNCT[rng.integers(len(_PUNCT))] if rng.random() < 0.8 else " " for _ in range(L))
        if cat == "ws":
            if rng.random() < 0.5:
                return " " * L
            return ("\n" + " " * (L - 1))[:L]
        if cat == "junk":
            if rng.random() < 0.3:
                bs = bytes(int(x) for x in rng.integers(128, 256, size=L))
                return bs
            return "".join(chr(int(x)) for x in rng.integers(33, 127, size=L))
        if cat == "multi":
            if not windows:
                return None
            w = windows[rng.integers(len(windows))]
            if len(w) <= L:
                return None
            a = int(rng.integers(0, len(w) - L))
            return w[a:a + L]
        return None

    while len(spell) < n_plain:
        avail = ~saturated
        if not avail.any():
            raise RuntimeError("vocabulary space exhausted")
        p = pl * avail
        li = int(rng.choice(len(ls), p=p / p.sum()))
        L = int(ls[li])
        cat = cats[int(rng.choice(len(cats), p=cw))]
        s = gen(cat, L)
        if s is None:
            continue
        b = s if isinstance(s, bytes) else s.encode("latin-1")
        if len(b) != L or b in seen:
            fails[li] += 1
            if fails[li] > 400:
                saturated[li] = True
            continue
        fails[li] = 0
        seen.add(b)
        spell.append(b)
    for _ in range(n_alias):
        spell.append(spell[int(rng.integers(256, len(spell)))])
    order = rng.permutation(len(spell))
    toks = [spell[i] for i in order]
    specials = []
    for k in range(n_special):
        specials.append(len(toks))
        toks.append(("<|special_%d|>" % k).encode())
    eos = len(toks)
    toks.append(b"<|endoftext|>")
    assert len(toks) == V
    return toks, eos, specials


def expr_vocab(seed: int, V: int = 512, n_alias: int = 5, alpha: bytes = b"abcdefghijklmnopqrstuvwxyz0123456789+*() "):
    """V ids over the alphabet (default [a-z0-9+*() ]): its single bytes,
    distinct random strings of length 2-4 drawn uniformly from it, ``n_alias``
    duplicate spellings, and EOS as the last id.  Returns (tokens, eos_id, [])."""
    rng = np.random.default_rng(seed)
    toks = [bytes([c]) for c in alpha]
    seen = set(toks)
    n_rand = V - 1 - len(alpha) - n_alias
    while len(toks) < len(alpha) + n_rand:
        L = int(rng.integers(2, 5))
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
    return toks, eos, []


# --------------------------------------------------------------------------
# greedy tokenizer
# --------------------------------------------------------------------------
class GreedyTokenizer:
    """Longest-match tokenization over a vocabulary's spellings (special ids and
    EOS excluded); among alias ids of one spelling the smallest id is used."""

    def __init__(self, tokens, exclude):
        ex = set(exclude)
        self.map = {}
        self.maxlen = 1
        for i, t in enumerate(tokens):
            if i in ex or not t:
                continue
            if t not in self.map:
                self.map[t] = i
            self.maxlen = max(self.maxlen, len(t))

    def encode(self, data: bytes, limit: int | None = None):
        out = []
        i, n = 0, len(data)
        while i < n and (limit is None or len(out) < limit):
            for L in range(min(self.maxlen, n - i), 0, -1):
                tid = self.map.get(data[i:i + L])
                if tid is not None:
                    out.append(tid)
                    i += L
                    break
            else:
                raise ValueError("vocabulary is not byte-complete at offset %d" % i)
        return out
