"""Configurations and the exact mask M(kappa) -- test infrastructure.

Follows GRID Sec. 2 (maximal munch with contextual resolution, L3 lexicons),
Sec. 3.2 (Def. 1 configuration, Def. 2 viable prefix, allowed terminals by
simulation, EOS gating) and Sec. 4.1 (Def. 4 the mask), in the readings listed
below.  Everything is per token and per byte; the stack is the persistent chain
of Def. 1 (a node is (state, parent)), so trying a token never copies it.

Readings where the paper is silent (shared with the CUDA path, both written
from this list):
  * Maximal munch runs over the regex union automaton, lexicon-blind.  When a
    byte kills the automaton, the pending lexeme r is emitted; its candidates
    are the terminals accepting r, where a category terminal c also needs
    r in W_c.  The first candidate in priority (declaration) order that is
    ignored, or whose simulated reduce chain reaches SHIFT, wins; if none does,
    or r is empty, the byte is rejected (no backtracking).  The killing byte is
    then fed from the start state.  Grammars guarantee that the automaton is
    accept-closed (no live non-accepting state after an accepting one), so the
    last accept is always the whole of r.
  * Trailing liveness (Def. 2): r is empty, or some terminal live at q(r) is
    ignored or allowed, where a category terminal c also needs r in Prefix(W_c).
  * EOS (Sec. 3.2): r is empty or finalizes by the same candidate pick; after
    shifting that terminal on a scratch stack, the reduce chain of $end reaches
    ACCEPT.
  * Special tokens and EOS are never set by the trie rule; EOS only by the gate.
"""
from __future__ import annotations

from dataclasses import dataclass

from .grammar import Grammar, project
from .lr1 import LR1
from .regex import UnionDFA, literal_ast, parse_regex


class LexiconError(ValueError):
    pass


@dataclass(frozen=True)
class Config:
    """Def. 1: kappa = (sigma, rho).  ``stack`` is a persistent chain
    (state, parent) with None below the bottom; ``q`` is the DFA state of the
    pending lexeme ``r`` (1 = start when r is empty).  ``complete`` is set once
    EOS has been accepted."""
    stack: tuple
    q: int
    r: bytes
    complete: bool = False


class OracleGrammar:
    def __init__(self, text: str, role=None, lexicons=None):
        g = Grammar(text)
        self.g = g
        self.n_term = len(g.terminals)
        self.END = self.n_term
        asts = [literal_ast(p[1]) if p[0] == "lit" else parse_regex(p[1]) for _, _, p in g.terminals]
        self.dfa = UnionDFA(asts)
        self.ignored = frozenset(i for i, t in enumerate(g.terminals) if t[1] == "ignore")
        self.categories = frozenset(g.term_ids[c] for c in g.categories)
        prods = project(g, role)
        self.lr = LR1(prods, g.start, self.n_term, g.term_ids)
        lexicons = lexicons or {}
        self.W = {}
        self.P = {}
        for c in self.categories:
            name = g.terminals[c][0]
            words = [w if isinstance(w, bytes) else w.encode() for w in lexicons.get(name, [])]
            for w in words:
                # precondition (d) of Prop. 8: W_c is a subset of R_c
                if c not in self.dfa.acc[self.dfa.run(w)]:
                    raise LexiconError("lexicon word %r is not in the regex of %s" % (w, name))
            self.W[c] = frozenset(words)
            self.P[c] = frozenset(w[:k] for w in words for k in range(len(w) + 1))
        self.START = 1
        self.DEAD = 0

    # ---- parser simulation (Sec. 3.2, "allowed terminals by simulation") ----
    def simulate(self, stack, tau):
        """Run the reduce chain for terminal ``tau`` on a virtual copy of the
        persistent stack.  Returns ('shift', new_stack), ('accept', stack) or None."""
        A, G, rhs, lhs = self.lr.ACTION, self.lr.GOTO, self.lr.rhs, self.lr.lhs
        st = stack
        while True:
            a = A[st[0]].get(tau)
            if a is None:
                return None
            kind, arg = a
            if kind == "s":
                return ("shift", (arg, st))
            if kind == "acc":
                return ("accept", st)
            for _ in range(len(rhs[arg])):
                st = st[1]
            st = (G[st[0]][lhs[arg]], st)

    def allowed(self, stack):
        """A(sigma) = {tau : simulate(sigma, tau) reaches SHIFT}."""
        out = set()
        for t in range(self.n_term):
            if t not in self.ignored:
                s = self.simulate(stack, t)
                if s is not None and s[0] == "shift":
                    out.add(t)
        return out

    # ---- lexer ----
    def candidates(self, q, r):
        """Emission candidates of lexeme r in priority order."""
        return [t for t in sorted(self.dfa.acc[q]) if t not in self.categories or r in self.W[t]]

    def emit(self, stack, q, r):
        """Finalize pending lexeme r on ``stack``: the highest-priority
        parser-viable candidate wins.  Returns the new stack or None."""
        for t in self.candidates(q, r):
            if t in self.ignored:
                return stack
            s = self.simulate(stack, t)
            if s is not None and s[0] == "shift":
                return s[1]
        return None

    def feed(self, cfg: Config, b: int):
        """Feed one byte; None if the output stops being a viable prefix."""
        nq = self.dfa.delta[cfg.q][b]
        if nq != self.DEAD:
            return Config(cfg.stack, nq, cfg.r + bytes([b]))
        if not cfg.r:
            return None
        st = self.emit(cfg.stack, cfg.q, cfg.r)
        if st is None:
            return None
        nq = self.dfa.delta[self.START][b]
        if nq == self.DEAD:
            return None
        return Config(st, nq, bytes([b]))

    def live_end(self, cfg: Config) -> bool:
        """Def. 2, operational: the trailing partial lexeme is live for some
        allowed-or-ignored terminal (with the lexicon-prefix condition)."""
        if not cfg.r:
            return True
        for t in sorted(self.dfa.live[cfg.q]):
            if t in self.categories and cfg.r not in self.P[t]:
                continue
            if t in self.ignored:
                return True
            s = self.simulate(cfg.stack, t)
            if s is not None and s[0] == "shift":
                return True
        return False

    def eos_ok(self, cfg: Config) -> bool:
        """EOS gating (Sec. 3.2): w is a complete sentence."""
        if cfg.complete:
            return False
        st = cfg.stack
        if cfg.r:
            st = self.emit(st, cfg.q, cfg.r)
            if st is None:
                return False
        s = self.simulate(st, self.END)
        return s is not None and s[0] == "accept"

    # ---- configurations ----
    def start_config(self) -> Config:
        return Config((0, None), self.START, b"")

    def feed_bytes(self, cfg: Config, data: bytes):
        for b in data:
            cfg = self.feed(cfg, b)
            if cfg is None:
                return None
        return cfg

    def viable(self, data: bytes, cfg: Config | None = None) -> bool:
        """Is ``data`` (appended to cfg's output) a viable prefix?"""
        c = self.feed_bytes(cfg or self.start_config(), data)
        return c is not None and self.live_end(c)

    def token_bit(self, cfg: Config, tok: bytes) -> bool:
        if cfg.complete or not tok:
            return False
        c = self.feed_bytes(cfg, tok)
        return c is not None and self.live_end(c)

    def mask(self, cfg: Config, tokens, eos: int, specials=(), ids=None):
        """Def. 4 over token ids: returns a list of 0/1 (or only for ``ids``)."""
        sp = set(specials)
        rng = range(len(tokens)) if ids is None else ids
        out = []
        for i in rng:
            if i == eos:
                out.append(1 if self.eos_ok(cfg) else 0)
            elif i in sp:
                out.append(0)
            else:
                out.append(1 if self.token_bit(cfg, tokens[i]) else 0)
        return out

    def advance(self, cfg: Config, tok_id: int, tokens, eos: int, specials=()):
        """Advance by one sampled token (Sec. 6.1 step 7); None if the token is
        not in the mask."""
        if cfg.complete:
            return None
        if tok_id == eos:
            return Config(cfg.stack, cfg.q, cfg.r, True) if self.eos_ok(cfg) else None
        if tok_id in set(specials):
            return None
        c = self.feed_bytes(cfg, tokens[tok_id])
        if c is None or not self.live_end(c):
            return None
        return c

    def forced_span(self, cfg: Config, tokens, eos: int, specials=(), max_span: int = 16):
        """Jump-forward (Sec. 6.1 step 6): while the mask of the configuration
        has exactly one bit set (over token ids, EOS included), that token is
        forced: append it and advance.  Returns (span ids, final config)."""
        span = []
        while len(span) < max_span and not cfg.complete:
            m = self.mask(cfg, tokens, eos, specials)
            if sum(m) != 1:
                break
            t = m.index(1)
            nxt = self.advance(cfg, t, tokens, eos, specials)
            if nxt is None:
                break
            span.append(t)
            cfg = nxt
        return span, cfg

    def config_from_ids(self, ids, tokens, eos: int, specials=()):
        cfg = self.start_config()
        for t in ids:
            cfg = self.advance(cfg, t, tokens, eos, specials)
            if cfg is None:
                return None
        return cfg

    def stack_list(self, cfg: Config):
        out = []
        st = cfg.stack
        while st is not None:
            out.append(st[0])
            st = st[1]
        return out[::-1]


def compile_grammar(text: str, role=None, lexicons=None) -> OracleGrammar:
    return OracleGrammar(text, role, lexicons)
