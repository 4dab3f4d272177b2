"""Token-denominated reserve completion (GRID Sec. 5, Prop. 9, Termination;
Sec. 6.1 step 3) -- TEST INFRASTRUCTURE.

Prop. 9 asks for a reserve counted in vocabulary tokens, per configuration,
summed over the stack, answering Write(shortest legal completion + EOS).  The
reading taken here (shared with the CUDA path, written from this text):

  * rendering of a terminal tau: a blank and lexeme l(tau), split greedily
    into vocabulary tokens (longest spelling first); c(tau) = its token count.
    l(tau) is the shortest (then bytewise smallest) string whose first
    emission candidate is tau -- for a category, a word of its lexicon; the
    search for other terminals stops at 32 bytes.
  * the pending lexeme r ends as it stands, or after an extension y: for a
    terminal tau live at r, the shortest (then smallest) y with r.y a lexeme
    of tau (a category: r.y a word of its lexicon; otherwise a path of the
    lexer automaton to a state accepting tau); its bytes are written as
    single-byte tokens.  Then r (or r.y) is emitted by the contextual pick and
    ended by the state's separator: the blank when, after it, the lexer is
    where a fresh blank would leave it (that blank is the first rendering's),
    else the smallest byte that does so, written as its own token when a
    rendering follows.
  * the terminal completion x of the resulting stack minimising the sum of
    c(tau) over x, such that the stack followed by x reaches ACCEPT.
  * cost = |y| + [separator token] + sum c(tau) + 1 (EOS).
The cheapest terminal completion is computed by uniform-cost search over
parser stacks, where a step completes one kernel item [A -> alpha . beta] of
the top state: beta's cheapest yield is written, alpha is popped and the goto
on A pushed (any completion decomposes into such steps); the goal is the
accept item.
"""
from __future__ import annotations

import heapq


class Reserve:
    def __init__(self, og, tokens, eos, specials=()):
        self.og = og
        self.tokens = tokens
        self.eos = eos
        ex = set(specials) | {eos}
        self.id_of = {}
        for i, t in enumerate(tokens):
            if i not in ex and t and t not in self.id_of:
                self.id_of[t] = i
        self.maxlen = max(len(t) for t in self.id_of) if self.id_of else 1
        self.nt = og.n_term
        self.render = {}
        self.cost = {}
        for tau in range(self.nt):
            if tau in og.ignored:
                continue
            lex = self._lexeme(tau)
            if lex is None:
                continue
            toks = self.greedy(b" " + lex)
            if toks is not None:
                self.render[tau] = toks
                self.cost[tau] = len(toks)
        self._min_yields()

    # ---- lexemes and tokens ----
    def first_candidate(self, s: bytes):
        q = self.og.dfa.run(s)
        if q == self.og.DEAD:
            return None
        c = self.og.candidates(q, s)
        return c[0] if c else None

    def _lexeme(self, tau):
        og = self.og
        if tau in og.categories:
            for w in sorted(og.W[tau], key=lambda w: (len(w), w)):
                if self.first_candidate(w) == tau:
                    return w
            return None
        # breadth-first over strings in (length, bytes) order; strings that are
        # not prefixes of any lexicon word are merged by automaton state
        seen = set()
        level = [b""]
        allP = set().union(*og.P.values()) if og.P else set()
        for _ in range(32):
            nxt = []
            for s in level:
                for b in range(256):
                    t = s + bytes([b])
                    q = og.dfa.run(t)
                    if q == og.DEAD:
                        continue
                    key = (q, t if t in allP else None)
                    if key in seen:
                        continue
                    seen.add(key)
                    if self.first_candidate(t) == tau:
                        return t
                    nxt.append(t)
            level = nxt
            if not level:
                break
        return None

    def greedy(self, s: bytes):
        out, i = [], 0
        while i < len(s):
            for L in range(min(self.maxlen, len(s) - i), 0, -1):
                t = self.id_of.get(s[i:i + L])
                if t is not None:
                    out.append(t)
                    i += L
                    break
            else:
                return None
        return out

    def sep(self, q):
        og = self.og
        d = og.dfa.delta

        def ok(b):
            r = d[og.START][b]
            if r == og.DEAD:
                return False
            x = d[q][b]
            if x != og.DEAD and x != r:
                return False
            return bool(og.dfa.acc[r] & og.ignored) and og.dfa.live[r] <= og.ignored
        if ok(0x20):
            return 0x20
        for b in range(256):
            if ok(b):
                return b
        return None

    def extension(self, q, r: bytes, tau):
        """Shortest (then smallest) y, |y| >= 1, making r.y a lexeme of tau."""
        og = self.og
        if tau in og.categories:
            ws = [w for w in og.W[tau] if w.startswith(r) and len(w) > len(r)]
            return min(ws, key=lambda w: (len(w), w))[len(r):] if ws else None
        d = og.dfa.delta
        seen = {q}
        level = [(q, b"")]
        while level:
            nxt = []
            for s, y in level:
                for b in range(256):
                    x = d[s][b]
                    if x == og.DEAD or x in seen:
                        continue
                    seen.add(x)
                    if tau in og.dfa.acc[x]:
                        return y + bytes([b])
                    nxt.append((x, y + bytes([b])))
            level = nxt
        return None

    # ---- cheapest terminal completion of a stack ----
    def _min_yields(self):
        og, lr = self.og, self.og.lr
        INF = float("inf")
        nts = {l for l in lr.lhs}
        mc = {A: INF for A in nts}
        changed = True
        while changed:
            changed = False
            for p, A in enumerate(lr.lhs):
                c = sum(self.cost.get(X, INF) if not isinstance(X, str) else mc[X] for X in lr.rhs[p])
                if c < mc[A]:
                    mc[A] = c
                    changed = True
        self.mc = mc

    def beta_cost(self, p, d):
        lr = self.og.lr
        INF = float("inf")
        return sum(self.cost.get(X, INF) if not isinstance(X, str) else self.mc[X] for X in lr.rhs[p][d:])

    def completion_cost(self, stack):
        """Cheapest sum of c(tau) over terminal completions of the stack."""
        og, lr = self.og, self.og.lr
        INF = float("inf")
        pq = [(0, 0, stack)]
        best = {stack: 0}
        n = 1
        while pq:
            c, _, st = heapq.heappop(pq)
            if best.get(st, INF) < c:
                continue
            depth = 0
            x = st
            while x is not None:
                depth += 1
                x = x[1]
            for (p, d), _la in lr.kernel_states[st[0]]:
                bc = self.beta_cost(p, d)
                if bc == INF:
                    continue
                if p == 0:
                    if (d == 0 and depth == 1) or (d == 1 and depth == 2):
                        return c + bc
                    continue
                if d >= depth:
                    continue
                below = st
                for _ in range(d):
                    below = below[1]
                g = lr.GOTO[below[0]].get(lr.lhs[p])
                if g is None:
                    continue
                nst = (g, below)
                nc = c + bc
                if nc < best.get(nst, INF):
                    best[nst] = nc
                    heapq.heappush(pq, (nc, n, nst))
                    n += 1
        return INF

    def reserve(self, cfg):
        """The reserve of a configuration: the token count of its completion
        plus EOS (0 for a completed row), or None when there is none."""
        og = self.og
        if cfg.complete:
            return 0
        INF = float("inf")
        best = INF
        options = []
        if not cfg.r:
            options.append((b"", 0x20, cfg.stack))
        else:
            s = self.sep(cfg.q)
            if s is not None:
                st = og.emit(cfg.stack, cfg.q, cfg.r)
                if st is not None:
                    options.append((b"", s, st))
            live = [t for t in sorted(og.dfa.live[cfg.q])
                    if t not in og.ignored and (t not in og.categories or cfg.r in og.P[t])]
            for tau in live:
                y = self.extension(cfg.q, cfg.r, tau)
                if y is None or len(y) > 64:
                    continue
                q2 = og.dfa.run(cfg.r + y)
                s = self.sep(q2)
                if s is None:
                    continue
                st = og.emit(cfg.stack, q2, cfg.r + y)
                if st is None:
                    continue
                if any(bytes([b]) not in self.id_of for b in y):
                    continue
                options.append((y, s, st))
        for y, s, st in options:
            C = self.completion_cost(st)
            if C == INF:
                continue
            if C > 0 and s != 0x20 and bytes([s]) not in self.id_of:
                continue
            tot = len(y) + (1 if (C > 0 and s != 0x20) else 0) + C + 1
            best = min(best, tot)
        return None if best == INF else best
