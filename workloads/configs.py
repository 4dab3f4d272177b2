"""The five workload recipes (tiny expression grammar, SQL admin, SQL
SELECT-only headline, long/deep flatness sweep, cold schema).

Each recipe returns a plain dict of inputs; seeds default to 1000 + index.
Prefixes are lists of token ids obtained by rendering a random sentence,
tokenizing it greedily and truncating it (at a byte offset for the tiny
grammar, at a token count for the SQL workloads)."""
from __future__ import annotations

import numpy as np

from . import grammar_text, grammar_keywords
from .gen import (GreedyTokenizer, SqlGen, expr_sentence, expr_vocab, make_schema,
                  pick_sentence, render, sql_vocab)

SQL_V_HEADLINE = 151_936
SQL_V_SWEEP = 128_256
SQL_V_ADMIN = 32_000

_cache: dict = {}


def _sql_vocab_cached(V: int, seed: int, multiword: float):
    key = ("vocab", V, seed, multiword)
    if key not in _cache:
        kws = grammar_keywords(grammar_text("sql"))
        src = None
        if multiword > 0:
            rng = np.random.default_rng(seed + 77)
            tables, cols, _ = make_schema(seed + 78, 50, 12, kws, col_pool=300)
            g = SqlGen(rng, tables, cols, dml=True)
            src = [render(g.statement(2), rng).encode() for _ in range(3000)]
        _cache[key] = sql_vocab(seed, V, kws, multiword_frac=multiword, sentence_src=src)
    return _cache[key]


def _tokenizer_cached(V, toks, exclude):
    key = ("tok", V, len(toks), toks[0], toks[-2])
    if key not in _cache:
        _cache[key] = GreedyTokenizer(toks, exclude)
    return _cache[key]


def tiny_expr(seed: int = 1001, B: int = 64, V: int = 512):
    """Expression grammar, V=512 vocab over [a-z0-9+*() ], 64 prefixes truncated
    at a uniformly random byte offset of a random derivation (nesting <= 8)."""
    rng = np.random.default_rng(seed)
    toks, eos, specials = expr_vocab(seed, V)
    tk = GreedyTokenizer(toks, specials + [eos])
    prefixes, texts = [], []
    for _ in range(B):
        s = expr_sentence(rng, 8).encode()
        cut = int(rng.integers(0, len(s) + 1))
        texts.append(s[:cut])
        prefixes.append(tk.encode(s[:cut]))
    return dict(name="tiny_expr", grammar=grammar_text("expr"), role=None, lexicons={},
                tokens=toks, eos=eos, specials=specials, prefixes=prefixes, texts=texts, B=B,
                seed=seed)


PICK_LEXICONS = {"TABLE_NAME": ["ab", "abc", "ba"], "COLUMN_NAME": ["a", "ab", "c"]}


def tiny_pick(seed: int = 1006, B: int = 64, V: int = 300):
    """Pick grammar (a bare or qualified column, so that both identifier
    categories are parser-viable at one point) with the word "ab" in both
    lexicons; V ids over the alphabet [abcgo.,; ]; B prefixes truncated at a
    uniformly random byte offset of a random sentence."""
    rng = np.random.default_rng(seed)
    toks, eos, specials = expr_vocab(seed, V, n_alias=4, alpha=b"abcgo.,; ")
    tk = GreedyTokenizer(toks, specials + [eos])
    prefixes, texts = [], []
    for _ in range(B):
        s = pick_sentence(rng).encode()
        cut = int(rng.integers(0, len(s) + 1))
        texts.append(s[:cut])
        prefixes.append(tk.encode(s[:cut]))
    return dict(name="tiny_pick", grammar=grammar_text("lexpick"), role=None,
                lexicons={k: list(v) for k, v in PICK_LEXICONS.items()},
                tokens=toks, eos=eos, specials=specials, prefixes=prefixes, texts=texts, B=B, seed=seed)


def forced_pick():
    """Pick grammar with a small vocabulary that is not byte-complete, so that
    some configurations admit exactly one token (jump-forward spans)."""
    toks = [b"g", b" a", b" o", b" ab", b";", b".c", b",", b" ba", b"<eos>"]
    prefixes = [[], [0], [0, 3], [0, 3, 5], [0, 1], [0, 1, 6], [0, 3, 5, 2], [0, 3, 5, 2, 7], [0, 3, 5, 2, 7, 4]]
    return dict(name="forced_pick", grammar=grammar_text("lexpick"), role=None,
                lexicons={k: list(v) for k, v in PICK_LEXICONS.items()},
                tokens=toks, eos=len(toks) - 1, specials=[], prefixes=prefixes, B=len(prefixes), seed=0)


def forced_sql():
    """SQL SELECT-only projection, a one-table one-column schema and a small
    vocabulary of blank-led words (not byte-complete): after "select *" the
    words "from" and the table are forced, after "group" or "order" "by" is."""
    toks = [b" select", b" *", b" from", b" t", b" where", b" x", b" =", b" 1", b";", b" and", b" or", b" (",
            b" )", b" count", b"(", b"*", b")", b" order", b" by", b" group", b"<eos>"]
    prefixes = [[], [0], [0, 1], [0, 1, 2], [0, 1, 2, 3], [0, 5, 2, 3, 4], [0, 5, 2, 3, 17], [0, 5, 2, 3, 19],
                [0, 13], [0, 13, 14, 15], [0, 1, 2, 3, 8]]
    return dict(name="forced_sql", grammar=grammar_text("sql"), role=[],
                lexicons={"TABLE_NAME": ["t"], "COLUMN_NAME": ["x"]},
                tokens=toks, eos=len(toks) - 1, specials=[], prefixes=prefixes, B=len(prefixes), seed=0)


def _sql_prefixes(rng, gen: SqlGen, tk: GreedyTokenizer, lens):
    prefixes, texts = [], []
    for n in lens:
        preds = max(1, n // 10)
        while True:
            text = render(gen.statement(2, where_preds=preds), rng, comment_rate=0.01).encode()
            ids = tk.encode(text)
            if len(ids) >= n or preds > 4 * n:
                break
            preds *= 2
        ids = ids[:n]
        prefixes.append(ids)
        texts.append(b"".join(tk_tokens(tk, ids)))
    return prefixes, texts


def tk_tokens(tk: GreedyTokenizer, ids):
    inv = getattr(tk, "_inv", None)
    if inv is None:
        inv = {v: k for k, v in tk.map.items()}
        tk._inv = inv
    return [inv[i] for i in ids]


def sql_admin(seed: int = 1002, B: int = 32, V: int = SQL_V_ADMIN):
    """SQL grammar, admin role (all productions), schema 20 x 10, V=32,000,
    32 prefixes of U[20,200] tokens."""
    kws = grammar_keywords(grammar_text("sql"))
    tables, cols, words = make_schema(seed, 20, 10, kws, col_pool=120)
    toks, eos, specials = _sql_vocab_cached(V, seed, 0.0)
    tk = GreedyTokenizer(toks, specials + [eos])
    rng = np.random.default_rng(seed + 1)
    lens = [int(x) for x in rng.integers(20, 201, size=B)]
    prefixes, texts = _sql_prefixes(rng, SqlGen(rng, tables, cols, dml=True), tk, lens)
    return dict(name="sql_admin", grammar=grammar_text("sql"), role=["dml"],
                lexicons={"TABLE_NAME": tables, "COLUMN_NAME": words},
                tokens=toks, eos=eos, specials=specials, prefixes=prefixes, texts=texts, B=B,
                seed=seed)


def sql_shared(seed: int = 1007, B: int = 32, V: int = SQL_V_ADMIN, shared: int = 8):
    """SQL admin workload whose schema has ``shared`` column names that are
    also table names (20 x 10 schema, V=32,000, prefixes of U[20,200]
    tokens): where a column may stand, both identifier categories are
    parser-viable and such a word is read as TABLE_NAME, the earlier one."""
    kws = grammar_keywords(grammar_text("sql"))
    tables, cols, words = make_schema(seed, 20, 10, kws, col_pool=60, shared=shared)
    toks, eos, specials = _sql_vocab_cached(V, 1002, 0.0)
    tk = GreedyTokenizer(toks, specials + [eos])
    rng = np.random.default_rng(seed + 1)
    both = sorted(set(tables) & set(words))
    n_end = B // 4
    lens = [int(x) for x in rng.integers(20, 201, size=B - n_end)]
    gen = SqlGen(rng, tables, cols, dml=True)
    prefixes, texts = _sql_prefixes(rng, gen, tk, lens)
    # a quarter of the rows end with a shared word where a column may stand,
    # so that the pending lexeme's two candidates are both parser-viable
    for k in range(n_end):
        head = [["select"], ["select", "*", "from", gen.table(), "where"],
                ["select", gen._pick(gen.all_cols), "from", gen.table(), "order", "by"]][k % 3]
        text = render(head + [both[k % len(both)]], rng).encode()
        ids = tk.encode(text)
        prefixes.append(ids)
        texts.append(b"".join(tk_tokens(tk, ids)))
    return dict(name="sql_shared", grammar=grammar_text("sql"), role=["dml"],
                lexicons={"TABLE_NAME": tables, "COLUMN_NAME": words},
                tokens=toks, eos=eos, specials=specials, prefixes=prefixes, texts=texts, B=B,
                seed=seed, shared=sorted(set(tables) & set(words)))


def sql_select_only(seed: int = 1003, B: int = 32, V: int = SQL_V_HEADLINE,
                    lo: int = 50, hi: int = 2000, prefix_seed: int | None = None):
    """Headline workload: SQL grammar under the SELECT-only projection (DML
    productions removed), schema 200 x 30, V=151,936 with ~3% multi-word tokens,
    B=32 prefixes of U[50,2000] tokens, fp32 logits N(0,3)."""
    kws = grammar_keywords(grammar_text("sql"))
    tables, cols, words = make_schema(seed, 200, 30, kws, col_pool=3000)
    toks, eos, specials = _sql_vocab_cached(V, 1003, 0.03)
    tk = _tokenizer_cached(V, toks, specials + [eos])
    rng = np.random.default_rng(seed + 1 if prefix_seed is None else prefix_seed)
    lens = [int(x) for x in rng.integers(lo, hi + 1, size=B)]
    prefixes, texts = _sql_prefixes(rng, SqlGen(rng, tables, cols, dml=False), tk, lens)
    return dict(name="sql_select_only", grammar=grammar_text("sql"), role=[],
                lexicons={"TABLE_NAME": tables, "COLUMN_NAME": words},
                tokens=toks, eos=eos, specials=specials, prefixes=prefixes, texts=texts, B=B,
                seed=seed, logits_dtype="f32", logits_std=3.0)


def sql_sweep_cell(n: int, depth: int, seed: int = 1004, B: int = 32, V: int = SQL_V_SWEEP):
    """One cell of the flatness sweep: admin role, schema 200 x 30, V=128,256,
    B=32 prefixes of exactly ``n`` tokens whose first part opens ``depth``
    nesting levels (parentheses or IN-subqueries) and whose rest is a
    left-recursive AND/OR chain, truncated mid-chain."""
    kws = grammar_keywords(grammar_text("sql"))
    tables, cols, words = make_schema(seed, 200, 30, kws, col_pool=3000)
    toks, eos, specials = _sql_vocab_cached(V, seed, 0.0)
    tk = GreedyTokenizer(toks, specials + [eos])
    rng = np.random.default_rng(seed * 1000 + n * 7 + depth)
    gen = SqlGen(rng, tables, cols, dml=True)
    prefixes, texts = [], []
    for _ in range(B):
        preds = max(2, n // 6)
        while True:
            text = render(gen.nested_chain(depth, preds), rng).encode()
            ids = tk.encode(text, limit=n + 1)
            if len(ids) > n:
                break
            preds *= 2
        ids = ids[:n]
        prefixes.append(ids)
        texts.append(b"".join(tk_tokens(tk, ids)))
    return dict(name="sql_sweep_n%d_d%d" % (n, depth), grammar=grammar_text("sql"), role=["dml"],
                lexicons={"TABLE_NAME": tables, "COLUMN_NAME": words},
                tokens=toks, eos=eos, specials=specials, prefixes=prefixes, texts=texts, B=B,
                seed=seed, n=n, depth=depth)


def sql_cold_schema(seed: int = 1005, B: int = 256, V: int = SQL_V_HEADLINE,
                    lo: int = 50, hi: int = 2000):
    """Cold-schema workload: a fresh schema of 1,000 tables x 50 distinct
    columns (50k identifiers), SELECT-only role, the headline V=151,936
    vocabulary, B=256 prefixes of U[50,2000] tokens, bf16 logits N(0,3)."""
    kws = grammar_keywords(grammar_text("sql"))
    tables, cols, words = make_schema(seed, 1000, 50, kws, col_pool=None)
    toks, eos, specials = _sql_vocab_cached(V, 1003, 0.03)
    tk = GreedyTokenizer(toks, specials + [eos])
    rng = np.random.default_rng(seed + 1)
    lens = [int(x) for x in rng.integers(lo, hi + 1, size=B)]
    prefixes, texts = _sql_prefixes(rng, SqlGen(rng, tables, cols, dml=False), tk, lens)
    return dict(name="sql_cold_schema", grammar=grammar_text("sql"), role=[],
                lexicons={"TABLE_NAME": tables, "COLUMN_NAME": words},
                tokens=toks, eos=eos, specials=specials, prefixes=prefixes, texts=texts, B=B,
                seed=seed, logits_dtype="bf16", logits_std=3.0)


def logits(seed: int, B: int, V: int, std: float = 3.0):
    """fp32 logits ~ N(0, std^2), shape [B, V], as a numpy array."""
    rng = np.random.default_rng(seed + 99)
    return (rng.standard_normal((B, V), dtype=np.float32) * np.float32(std)).astype(np.float32)


# --------------------------------------------------------------------------
# many lexicon categories: the edges of the 16-bit class-code space
# --------------------------------------------------------------------------
MANYCAT_KEYWORDS = ["ab", "bad", "cab", "dace", "ebb", "deed", "aced", "bead", "cede", "dab", "beaded",
                    "decade", "acceded", "abed", "ace", "ebbed", "added", "adde", "cabbed", "dabbed", "bade"]


def manycat_grammar(n_cat: int, n_kw: int) -> str:
    """A list language whose items are n_cat lexicon categories C0.. sharing the
    identifier regex /[a-e]+/, qualified pairs C(2k) "." C(2k+1), a call
    C0 "(" args ")" and keyword-led items; the n_kw keywords are words over the
    same letters, each adding lexer states.  A CI class id ranges over
    2 x lexer states x 2^n_cat values, so the number of categories and
    keywords moves the spec across the edges of the 16-bit code space."""
    kws = MANYCAT_KEYWORDS[:n_kw]
    out = ["# %d lexicon categories over one regex, %d keywords (generated)" % (n_cat, n_kw)]
    out += ['%%token K%d "%s"' % (i, k) for i, k in enumerate(kws)]
    out += ["%%token C%d /[a-e]+/" % c for c in range(n_cat)]
    out += ['%token COMMA ","', '%token SEMI ";"', '%token DOT "."', '%token LP "("', '%token RP ")"',
            "%ignore WS /[ ]+/"]
    out += ["%%category C%d" % c for c in range(n_cat)]
    out += ["%start prog", "", "prog -> items SEMI", "items -> items COMMA item", "items -> item"]
    out += ["item -> C%d" % c for c in range(n_cat)]
    out += ["item -> C%d DOT C%d" % (c, c + 1) for c in range(0, n_cat - 1, 2)]
    out += ["item -> C0 LP args RP"]
    out += ["item -> K%d C%d" % (i, i % n_cat) for i in range(len(kws))]
    out += ["args -> args COMMA C1", "args -> C2"]
    return "\n".join(out) + "\n"


def manycat(n_cat: int, n_kw: int, seed: int = 1008, B: int = 16, n_multi: int = 10000):
    """Many-category workload.  Lexicons: 12 words over a-e of length 2-5 per
    category (keywords excluded), pairwise disjoint, plus 6 words shared by
    several categories that sentences never use.  Vocabulary: every string of
    length 1-2 over [abcde,;.() ], then ``n_multi`` distinct random strings of
    2-4 pieces (letter runs, keywords, punctuation, blanks), EOS last.
    Prefixes: random sentences (items from single-lexicon words, blanks
    between lexemes) tokenized greedily and cut at a random byte offset."""
    rng = np.random.default_rng(seed)
    letters = "abcde"
    kws = MANYCAT_KEYWORDS[:n_kw]
    taken = set(MANYCAT_KEYWORDS)

    def rand_word(lo=2, hi=5):
        return "".join(letters[int(i)] for i in rng.integers(0, 5, size=int(rng.integers(lo, hi + 1))))

    own = []
    for _ in range(n_cat):
        ws = []
        while len(ws) < 12:
            w = rand_word()
            if w not in taken:
                taken.add(w)
                ws.append(w)
        own.append(ws)
    shared = []
    while len(shared) < 6:
        w = rand_word()
        if w not in taken:
            taken.add(w)
            shared.append(w)
    lexicons = {}
    for c in range(n_cat):
        extra = [shared[k] for k in range(6) if (c + k) % 3 == 0]
        lexicons["C%d" % c] = sorted(own[c] + extra)
    alpha = "abcde,;.() "
    toks = [a for a in alpha] + [a + b for a in alpha for b in alpha]
    seen = set(toks)
    pieces = [lambda: rand_word(1, 4), lambda: kws[int(rng.integers(len(kws)))] if kws else "a",
              lambda: ",;.()"[int(rng.integers(5))], lambda: " "]
    while len(toks) < len(alpha) * (len(alpha) + 1) + n_multi:
        s = "".join(pieces[int(rng.choice(4, p=[0.45, 0.1, 0.3, 0.15]))]() for _ in range(int(rng.integers(2, 5))))
        if s not in seen:
            seen.add(s)
            toks.append(s)
    tokens = [t.encode() for t in toks]
    eos = len(tokens)
    tokens.append(b"<eos>")

    def item():
        k = int(rng.integers(4))
        if k == 0:
            c = int(rng.integers(n_cat))
            return [own[c][int(rng.integers(12))]]
        if k == 1:
            c = 2 * int(rng.integers(n_cat // 2))
            return [own[c][int(rng.integers(12))], ".", own[c + 1][int(rng.integers(12))]]
        if k == 2:
            args = [own[2][int(rng.integers(12))]] + [own[1][int(rng.integers(12))]
                                                     for _ in range(int(rng.integers(0, 3)))]
            return [own[0][int(rng.integers(12))], "("] + sum(([a, ","] for a in args), [])[:-1] + [")"]
        i = int(rng.integers(len(kws)))
        return [kws[i], own[i % n_cat][int(rng.integers(12))]]

    tk = GreedyTokenizer(tokens, [eos])
    prefixes, texts = [], []
    for _ in range(B):
        lexemes = []
        for j in range(int(rng.integers(1, 6))):
            if j:
                lexemes.append(",")
            lexemes += item()
        lexemes.append(";")
        s = " ".join(lexemes).encode()
        cut = int(rng.integers(0, len(s) + 1))
        texts.append(s[:cut])
        prefixes.append(tk.encode(s[:cut]))
    return dict(name="manycat%d" % n_cat, grammar=manycat_grammar(n_cat, n_kw), role=None, lexicons=lexicons,
                tokens=tokens, eos=eos, specials=[], prefixes=prefixes, texts=texts, B=B, seed=seed)
