"""Jump-forward forced spans (Sec. 6.1 step 6) in the oracle, pinned to the
brute-force recognizer: a span is the run of configurations whose mask,
decided token by token by completion search, admits exactly one id."""
from oracle import compile_grammar
from tests.brute import BruteGrammar
from tests.test_oracle_brute import LEX, _PICK_COMPL
from workloads import configs, grammar_text


def _brute_mask(bg, text, toks, eos):
    out = []
    for i, t in enumerate(toks):
        if i == eos:
            out.append(int(bg.in_L(text)))
        else:
            out.append(int(bg.in_prefix_L(text + t, _PICK_COMPL)))
    return out


def test_forced_span_matches_brute_force_on_pick_grammar():
    wl = configs.forced_pick()
    toks, eos = wl["tokens"], wl["eos"]
    og = compile_grammar(wl["grammar"], wl["role"], wl["lexicons"])
    bg = BruteGrammar(grammar_text("lexpick"), lexicons=LEX)
    seen_forced = 0
    for pre in wl["prefixes"]:
        text = b"".join(toks[i] for i in pre)
        # brute-force span: extend while the brute mask is a singleton
        span, done = [], False
        while len(span) < 16 and not done:
            m = _brute_mask(bg, text, toks, eos)
            if sum(m) != 1:
                break
            t = m.index(1)
            span.append(t)
            if t == eos:
                done = True
            else:
                text += toks[t]
        cfg = og.config_from_ids(pre, toks, eos)
        got, _ = og.forced_span(cfg, toks, eos)
        assert got == span, (pre, got, span)
        seen_forced += len(span) > 0
    assert seen_forced >= 3


def test_forced_span_properties_sql():
    """Every forced token was the only admitted one, and the span stops at a
    mask with zero or several bits (or at max_span)."""
    wl = configs.forced_sql()
    toks, eos = wl["tokens"], wl["eos"]
    og = compile_grammar(wl["grammar"], wl["role"], wl["lexicons"])
    lens = []
    for pre in wl["prefixes"]:
        cfg = og.config_from_ids(pre, toks, eos)
        span, end = og.forced_span(cfg, toks, eos, max_span=8)
        c = cfg
        for t in span:
            m = og.mask(c, toks, eos)
            assert sum(m) == 1 and m[t] == 1
            c = og.advance(c, t, toks, eos)
        assert og.stack_list(c) == og.stack_list(end) and c.r == end.r
        if len(span) < 8:
            assert sum(og.mask(end, toks, eos)) != 1 or end.complete
        lens.append(len(span))
    assert max(lens) >= 2 and min(lens) == 0
    # max_span bounds the run
    cfg = og.config_from_ids(wl["prefixes"][2], toks, eos)
    assert og.forced_span(cfg, toks, eos, max_span=1)[0] == og.forced_span(cfg, toks, eos)[0][:1]
