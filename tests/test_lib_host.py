"""CPU-only checks of libgrid: the shared library loads, exports every symbol
that include/grid.h declares, and its host-side compiler reports the
documented errors (no GPU call is made here)."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2607_11951_gb300 import grid as G
from workloads import grammar_text

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built():
    if not os.path.exists(G.library_path()):
        import paper_2607_11951_gb300 as pkg
        pkg.build()
    G.lib()


def _declared():
    text = open(os.path.join(ROOT, "include", "grid.h")).read()
    return sorted(set(re.findall(r"^\s*(?:int|void|size_t|int64_t)\s+(grid_[a-z0-9_]+)\s*\(", text, re.M)))


def test_exports_every_declared_symbol():
    names = _declared()
    assert len(names) >= 16
    L = ctypes.CDLL(G.library_path())
    for n in names:
        assert hasattr(L, n), n
    assert sorted(G.EXPORTED) == sorted(n for n in names if n in G.EXPORTED)


def _err(text, role=None, lex=None):
    with pytest.raises(G.GridError) as e:
        G.Grammar(text, role, lex)
    return e.value.code


def test_compile_ok_and_sizes():
    g = G.Grammar(grammar_text("sql"), [], {"TABLE_NAME": ["t1"], "COLUMN_NAME": ["c1"]})
    info = g.info()
    assert info["terminals"] == 60 and info["categories"] == 2 and info["lalr_states"] > 50
    g2 = G.Grammar(grammar_text("sql"), ["dml"], {"TABLE_NAME": ["t1"], "COLUMN_NAME": ["c1"]})
    assert g2.info()["lalr_states"] > info["lalr_states"]  # projection removed DML states


def test_lalr_conflict_detected():
    # LR(1) but not LALR(1): merging the two 'c' states gives a reduce/reduce conflict
    text = """%token A "a"
%token B "b"
%token C "c"
%token D "d"
%token E "e"
%ignore WS /[ ]+/
%start s
s -> A x D
s -> B y D
s -> A y E
s -> B x E
x -> C
y -> C
"""
    assert _err(text) == -3
    # the same grammar with one pair removed is LALR(1)
    ok = text.replace("s -> B x E\n", "")
    G.Grammar(ok)


def test_empty_language_and_projection():
    text = """%token A "a"
%ignore WS /[ ]+/
%start s
s -> A @r
"""
    assert _err(text, role=[]) == -4
    G.Grammar(text, role_keep=["r"])


def test_lexicon_not_in_regex():
    assert _err(grammar_text("sql"), [], {"TABLE_NAME": ["Official_ratings_(millions)"], "COLUMN_NAME": []}) == -5


def test_lexer_preconditions():
    # "ab" accepting, "abc" live but not accepting, "abcd" accepting: not accept-closed
    text = """%token X "ab"
%token Y "abcd"
%ignore WS /[ ]+/
%start s
s -> X
s -> Y
"""
    assert _err(text) == -6
    # a blank extends a non-ignored lexeme: not blank-delimited
    text2 = """%token X /a[ a]*/
%ignore WS /[ ]+/
%start s
s -> X
"""
    assert _err(text2) == -6


def test_parse_errors():
    assert _err("%token A \"a\"\n%ignore WS /[ ]+/\n%start s\ns -> B\n") == -2
    assert _err("%token A /(a/\n%ignore WS /[ ]+/\n%start s\ns -> A\n") == -2


def test_vocab_errors_and_info():
    v = G.Vocab([bytes([b]) for b in range(256)] + [b"ab", b"ab", b"<eos>"], 258)
    info = v.info()
    assert info["spellings"] == 257 and info["byte_complete"] == 1
    with pytest.raises(G.GridError):
        G.Vocab([b"a", b"", b"<eos>"], 2)
    with pytest.raises(G.GridError):
        G.Vocab([b"a", b"<eos>"], 5)


def test_lexicon_trie_and_vocab_sizes_against_python():
    # the identifier trie has one node per distinct prefix of the lexicon words
    # (the empty prefix is the root), whichever category they belong to, and
    # the vocabulary keeps one spelling per distinct non-excluded token
    rng = np.random.default_rng(5)
    alpha = b"abcdefghijklmnopqrstuvwxyz_0123456789"
    def word():
        n = int(rng.integers(1, 12))
        w = bytes([alpha[int(rng.integers(0, 26))]]) + bytes(alpha[int(i)] for i in rng.integers(0, len(alpha), n - 1))
        return w
    tables = [word() for _ in range(300)]
    cols = [word() for _ in range(700)] + tables[:50] + [b"a", b"ab", b"abc"]
    g = G.Grammar(grammar_text("sql"), [], {"TABLE_NAME": tables, "COLUMN_NAME": cols})
    prefixes = {w[:k] for w in tables + cols for k in range(len(w) + 1)}
    assert g.info()["lexicon_nodes"] == len(prefixes)
    toks = [word() for _ in range(3000)] + [b"\x00", b"\xff", b"a\x00", b"<eos>", b"<pad>"]
    toks += toks[:100]  # aliases
    eos, specials = toks.index(b"<eos>"), [toks.index(b"<pad>")]
    v = G.Vocab(toks, eos, specials)
    kept = {t for i, t in enumerate(toks) if i != eos and i not in specials}
    info = v.info()
    assert info["spellings"] == len(kept)
    assert info["bytes"] == sum(len(t) for t in kept)


def test_lexicon_trie_arrays_against_python_bfs():
    """The identifier trie's arrays equal a trie built here by breadth-first
    numbering with children in byte order: child ranges, edge bytes, child
    ids, and the prefix / word category masks, for a random lexicon with
    shared prefixes, words in both categories and one-letter words."""
    rng = np.random.default_rng(9)
    alpha = b"abcdefghij_0123"
    def word():
        n = int(rng.integers(1, 7))
        return bytes([alpha[int(rng.integers(0, 10))]]) + bytes(alpha[int(i)] for i in rng.integers(0, len(alpha), n - 1))
    tables = sorted({word() for _ in range(120)})
    cols = sorted({word() for _ in range(200)} | set(tables[:30]) | {b"a", b"b"})
    g = G.Grammar(grammar_text("sql"), [], {"TABLE_NAME": tables, "COLUMN_NAME": cols})
    cstart, cbyte, cnode, pc, wc = G.grid_grammar_lexicon_trie(g.h)
    # reference trie: BFS from the root, children by byte
    cats = {0: tables, 1: cols}
    strings = sorted({w[:k] for c in cats.values() for w in c for k in range(len(w) + 1)}, key=lambda x: (len(x), x))
    children = {}
    for x in strings[1:]:
        children.setdefault(x[:-1], []).append(x)
    order, seen = [b""], 0
    while seen < len(order):
        x = order[seen]
        seen += 1
        order.extend(sorted(children.get(x, []), key=lambda y: y[-1]))
    idx = {x: i for i, x in enumerate(order)}
    assert len(order) == len(pc)
    want_start, want_byte, want_node = [0], [], []
    for x in order:
        for y in sorted(children.get(x, []), key=lambda y: y[-1]):
            want_byte.append(y[-1])
            want_node.append(idx[y])
        want_start.append(len(want_byte))
    assert cstart.tolist() == want_start
    assert cbyte.tolist() == want_byte and cnode.tolist() == want_node
    for x in order:
        p = sum(1 << c for c, ws in cats.items() if any(w.startswith(x) for w in ws))
        w = sum(1 << c for c, ws in cats.items() if x in set(ws))
        assert pc[idx[x]] == p and wc[idx[x]] == w, x


def test_manycat_grammars_straddle_the_class_code_space():
    """The many-category workloads sit on the two sides of the 16-bit class
    code space (the GPU parity test relies on it): 2 x lexer states x
    2^categories class ids reach 65,531 with ten categories and stay below it,
    within 1,024 ids of the top, with nine; the sentences of both parse."""
    from oracle import compile_grammar
    from paper_2607_11951_gb300 import grid as G
    from workloads import configs
    for n_cat, n_kw, over in ((10, 9, True), (9, 21, False)):
        wl = configs.manycat(n_cat, n_kw, B=6)
        info = G.Grammar(wl["grammar"], wl["role"], wl["lexicons"]).info()
        assert info["categories"] == n_cat
        ncls = (2 * info["dfa_states"]) << n_cat
        assert (ncls >= 65531) == over, (n_cat, info["dfa_states"], ncls)
        if not over:
            assert 65535 - 5 - ncls < 1024
        og = compile_grammar(wl["grammar"], wl["role"], wl["lexicons"])
        for p in wl["prefixes"]:
            cfg = og.config_from_ids(p, wl["tokens"], wl["eos"], wl["specials"])
            assert cfg is not None and og.live_end(cfg)


_VOID_FREE = ("grid_grammar_free", "grid_vocab_free", "grid_spec_free", "grid_configs_free", "grid_cache_free")


@pytest.mark.parametrize("name", [n for n in G.EXPORTED if n != "grid_last_error" and n not in _VOID_FREE])
def test_entry_point_refuses_null_handles_without_a_device(name):
    """Every call with NULL handles and pointers returns GRID_E_INVALID_ARG
    and names itself in the thread's error message, before any CUDA call (no
    GPU in this process); the free functions accept NULL."""
    L = G.lib()
    f = getattr(L, name)
    ints = (ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t, ctypes.c_uint32)
    args = [1 if a in ints else None for a in f.argtypes]
    assert f(*args) == -1, name
    buf = ctypes.create_string_buffer(256)
    L.grid_last_error(buf, 256)
    assert buf.value.decode().startswith(name + ":"), buf.value
    for free in _VOID_FREE:
        getattr(L, free)(None)


def test_apply_mask_argument_checks_on_the_host():
    """grid_apply_mask refuses a bad row count, vocabulary size, row stride or
    logits type, and more than 65,535 rows, before it launches anything (the
    pointers here are never dereferenced)."""
    L = G.lib()
    m, lg = ctypes.c_void_p(256), ctypes.c_void_p(512)
    F32, BF16 = G.GRID_DTYPE_F32, G.GRID_DTYPE_BF16
    for B, V, stride, dt in [(0, 10, 10, F32), (2, 0, 10, F32), (2, 10, 9, BF16), (2, 10, 10, 7), (-1, 10, 10, F32)]:
        assert L.grid_apply_mask(m, lg, dt, B, V, stride, None) == -1, (B, V, stride, dt)
    assert L.grid_apply_mask(m, lg, F32, 65536, 10, 10, None) == -8  # GRID_E_TOO_LARGE
    assert L.grid_apply_mask(None, lg, F32, 1, 10, 10, None) == -1
