"""Random grammars of the statement family (``workloads/randgram.py``), CPU
only.  Every rendered sentence is in the language by the oracle's EOS gate
(Sec. 3.2) and every cut of one is a viable prefix (Def. 2), so the prefixes
the GPU tests build are valid; and libgrid's host compiler accepts each
grammar under both role projections (Sec. 2, L2) with the oracle's terminal
count and the same minimised lexer DFA size."""
import os

import numpy as np
import pytest

from oracle import compile_grammar
from paper_2607_11951_gb300 import grid as G
from workloads.randgram import RandGrammar, render

SEEDS = list(range(24))


@pytest.fixture(scope="module", autouse=True)
def built():
    if not os.path.exists(G.library_path()):
        import paper_2607_11951_gb300 as pkg
        pkg.build()
    G.lib()


def test_family_covers_its_features():
    """Across the seeds: identifier categories, role-tagged statements, nested
    blocks, function calls and unary operators all occur."""
    gs = [RandGrammar(s) for s in SEEDS]
    assert sum(g.cats for g in gs) >= 6
    assert sum(any(p[2] for p in g.prods) for g in gs) >= 4
    assert sum(any(p[0] == "b" for p in g.prods) for g in gs) >= 8
    assert sum(any(p[0] == "args" for p in g.prods) for g in gs) >= 8
    assert sum(any(len(p[1]) == 2 and p[1][0].startswith("O") for p in g.prods) for g in gs) >= 6  # unary


@pytest.mark.parametrize("seed", SEEDS)
def test_random_grammar_sentences_and_compilers(seed):
    g = RandGrammar(seed)
    for role in (None, []):
        og = compile_grammar(g.text(), role, g.lexicons)
        info = G.Grammar(g.text(), role, g.lexicons).info()
        assert info["terminals"] == og.n_term + 1  # the library counts $end
        assert info["dfa_states"] == len(og.dfa.delta)
        assert info["categories"] == len(g.lexicons)
        rng = np.random.default_rng(seed)
        for _ in range(25):
            s = render(g.derive(rng, role), rng)
            c = og.feed_bytes(og.start_config(), s)
            assert c is not None and og.eos_ok(c), s
            cut = int(rng.integers(0, len(s)))
            c = og.feed_bytes(og.start_config(), s[:cut])
            assert c is not None and og.live_end(c), s[:cut]


def test_random_workloads_are_seeded_and_well_formed():
    """The same seed gives the same workload; prefixes are greedy
    tokenizations of their texts; the vocabulary is byte-complete over the
    grammar's alphabet with EOS last; the first row is the empty prefix."""
    from workloads.randgram import rand_grammar_workload
    a = rand_grammar_workload(3, B=12, V=800, role=[])
    b = rand_grammar_workload(3, B=12, V=800, role=[])
    assert a["grammar"] == b["grammar"] and a["tokens"] == b["tokens"] and a["prefixes"] == b["prefixes"]
    toks = a["tokens"]
    assert len(toks) == 800 and a["eos"] == 799 and toks[-1] == b"<eos>"
    alpha = RandGrammar(3).alphabet()
    assert all(bytes([c]) in toks for c in alpha)
    assert a["prefixes"][0] == [] and a["texts"][0] == b""
    for p, t in zip(a["prefixes"], a["texts"]):
        assert b"".join(toks[i] for i in p) == t
