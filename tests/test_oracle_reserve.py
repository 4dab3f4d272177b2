"""The oracle's token-denominated reserve (Sec. 5 Prop. 9, Sec. 6.1 step 3),
pinned to brute force: the cheapest terminal completion of a stack equals the
minimum, over every terminal string up to a length bound that drives the
parser to ACCEPT, of its summed rendering costs; and the completion the cost
model writes (extension, separator, renderings) is a sentence of L according
to the independent Earley recognizer, with exactly `reserve` tokens."""
import numpy as np
import pytest

from oracle import compile_grammar
from oracle.reserve import Reserve
from tests.brute import BruteGrammar
from tests.test_oracle_brute import LEX
from workloads import configs, grammar_text


def _brute_completion(og, R, stack, max_len):
    """(cost, terminal string) of the cheapest completion with at most
    max_len terminals, by exhaustive search over viable terminal strings."""
    best = (float("inf"), None)
    frontier = [(stack, ())]
    for L in range(max_len + 1):
        nxt = []
        for st, x in frontier:
            a = og.simulate(st, og.END)
            if a is not None and a[0] == "accept":
                c = sum(R.cost[t] for t in x)
                if c < best[0]:
                    best = (c, x)
            if L == max_len:
                continue
            for t in R.cost:
                s2 = og.simulate(st, t)
                if s2 is not None and s2[0] == "shift":
                    nxt.append((s2[1], x + (t,)))
        frontier = nxt
    return best


def _written(R, cfg):
    """The bytes and token count of one cheapest completion, built from the
    cost model's definition with a brute-force terminal string."""
    og = R.og
    INF = float("inf")
    opts = []
    if not cfg.r:
        opts.append((b"", 0x20, cfg.stack))
    else:
        s = R.sep(cfg.q)
        st = og.emit(cfg.stack, cfg.q, cfg.r) if s is not None else None
        if st is not None:
            opts.append((b"", s, st))
        for tau in sorted(og.dfa.live[cfg.q]):
            if tau in og.ignored or (tau in og.categories and cfg.r not in og.P[tau]):
                continue
            y = R.extension(cfg.q, cfg.r, tau)
            if y is None:
                continue
            q2 = og.dfa.run(cfg.r + y)
            s = R.sep(q2)
            st = og.emit(cfg.stack, q2, cfg.r + y) if s is not None else None
            if st is not None:
                opts.append((y, s, st))
    best = None
    for y, s, st in opts:
        c, x = _brute_completion(og, R, st, 6)
        if x is None:
            continue
        tot = len(y) + (1 if c > 0 and s != 0x20 else 0) + c + 1
        data = y + (bytes([s]) if c > 0 and s != 0x20 else b"") + b"".join(
            b"".join(R.tokens[i] for i in R.render[t]) for t in x)
        if best is None or tot < best[0]:
            best = (tot, data)
    return best


CASES = [
    ("expr", None, None, [b"", b"a", b"(", b"(a+", b"((1*", b"12", b"a+b*(c", b"(a) ", b"((a)+1)*"]),
    ("lexpick", None, LEX, [b"", b"g", b"g a", b"g ab", b"g ab.", b"g a,ba.c o", b"g a o a", b"g c o ab;"]),
    ("lexfix", None, LEX, [b"", b"g", b"g ab", b"d ", b"d ab", b"g a,c o ba"]),
]


@pytest.mark.parametrize("name,role,lex,prefixes", CASES, ids=[c[0] for c in CASES])
def test_reserve_matches_brute_force(name, role, lex, prefixes):
    text = grammar_text(name)
    og = compile_grammar(text, role=role, lexicons=lex)
    bg = BruteGrammar(text, role=role, lexicons=lex)
    # a vocabulary of all single bytes of the grammar's alphabet plus a few
    # multi-byte spellings (the renderings use the longest ones)
    alpha = sorted(set(b"".join(prefixes) + b" ()+*a1.,;gocbd" + b"abc"))
    toks = [bytes([c]) for c in alpha] + [b" a", b" (", b"ab", b" ab", b" o", b")", b";"]
    toks = list(dict.fromkeys(toks)) + [b"<eos>"]
    eos = len(toks) - 1
    R = Reserve(og, toks, eos)
    n = 0
    for pre in prefixes:
        cfg = og.feed_bytes(og.start_config(), pre)
        assert cfg is not None and og.live_end(cfg), pre
        res = R.reserve(cfg)
        best = _written(R, cfg)
        assert best is not None and res == best[0], (pre, res, best)
        # the written completion is a sentence, by the independent recognizer
        assert bg.in_L(pre + best[1]), (pre, best[1])
        n += res > 1
    assert n >= 2


def test_reserve_tokens_replay_in_the_oracle():
    """On the SQL grammar (no brute force there): every configuration of the
    admin workload has a reserve, and rendering costs are the greedy token
    counts of a blank plus the terminal's lexeme."""
    wl = configs.sql_admin(B=6)
    og = compile_grammar(wl["grammar"], wl["role"], wl["lexicons"])
    R = Reserve(og, wl["tokens"], wl["eos"], wl["specials"])
    for t, toks in R.render.items():
        assert len(toks) == R.cost[t] and b"".join(wl["tokens"][i] for i in toks).startswith(b" ")
    for p in wl["prefixes"]:
        cfg = og.config_from_ids(p, wl["tokens"], wl["eos"], wl["specials"])
        r = R.reserve(cfg)
        assert r is not None and r >= 1
