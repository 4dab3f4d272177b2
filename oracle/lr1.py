"""Canonical LR(1) tables (Knuth's construction) -- test infrastructure.

GRID runs an LALR(1) parser (Sec. 2); the oracle uses the canonical LR(1)
automaton of the same reduced grammar instead.  Both have the correct-prefix
property that Prop. 3 relies on (an LR parser never shifts a terminal that
cannot continue a sentence), so "simulate(sigma, tau) reaches SHIFT" and
"the reduce chain of $end reaches ACCEPT" decide the same sets; the oracle
keeps the textbook construction with no merging and no default reductions.

Items are (production, dot) cores paired with lookahead sets; a state is
identified by its kernel items with their lookahead sets (this is the canonical
LR(1) collection written with lookahead sets instead of one item per lookahead).
"""
from __future__ import annotations


class LRConflict(ValueError):
    pass


class LR1:
    """ACTION[s]: dict terminal_id -> ('s', state) | ('r', prod) | ('acc', None);
    GOTO[s]: dict nonterminal -> state.  Production 0 is S' -> start."""

    def __init__(self, prods, start: str, n_term: int, term_ids):
        self.END = n_term  # $end
        P = [("$S'", (start,))] + list(prods)
        self.prods = P
        nts = sorted({l for l, _ in P})
        self.is_nt = set(nts)
        tid = dict(term_ids)

        def sym(s):
            return s if s in self.is_nt else tid[s]

        self.rhs = [tuple(sym(s) for s in r) for _, r in P]
        self.lhs = [l for l, _ in P]
        by_lhs = {}
        for i, l in enumerate(self.lhs):
            by_lhs.setdefault(l, []).append(i)
        # nullable and FIRST (fixpoints)
        nullable = set()
        first = {n: set() for n in nts}
        changed = True
        while changed:
            changed = False
            for i, r in enumerate(self.rhs):
                l = self.lhs[i]
                for s in r:
                    if s in self.is_nt:
                        add = first[s] - first[l]
                        if add:
                            first[l] |= add
                            changed = True
                        if s not in nullable:
                            break
                    else:
                        if s not in first[l]:
                            first[l].add(s)
                            changed = True
                        break
                else:
                    if l not in nullable:
                        nullable.add(l)
                        changed = True

        def first_seq(seq, la):
            out = set()
            for s in seq:
                if s in self.is_nt:
                    out |= first[s]
                    if s not in nullable:
                        return out
                else:
                    out.add(s)
                    return out
            return out | la

        def closure(kernel):
            items = {}
            for core, la in kernel:
                items[core] = set(la)
            work = list(items.keys())
            while work:
                core = work.pop()
                p, d = core
                r = self.rhs[p]
                if d < len(r) and r[d] in self.is_nt:
                    la = first_seq(r[d + 1:], items[core])
                    for q in by_lhs[r[d]]:
                        c2 = (q, 0)
                        cur = items.get(c2)
                        if cur is None:
                            items[c2] = set(la)
                            work.append(c2)
                        elif not la <= cur:
                            cur |= la
                            work.append(c2)
            return items

        init = frozenset([((0, 0), frozenset([self.END]))])
        index = {init: 0}
        states = [init]
        # the grammar symbol on which each state is entered (a nonterminal
        # name or a terminal id; None for the start state)
        self.access = [None]
        self.kernel_states = states  # kernel items (core, lookaheads) of each state
        self.ACTION = []
        self.GOTO = []
        k = 0
        while k < len(states):
            items = closure(states[k])
            act, gto = {}, {}
            trans = {}
            for (p, d), la in items.items():
                r = self.rhs[p]
                if d < len(r):
                    trans.setdefault(r[d], {})
                    tk = trans[r[d]]
                    tk[(p, d + 1)] = tk.get((p, d + 1), frozenset()) | frozenset(la)
            for X, kern in trans.items():
                key = frozenset(kern.items())
                if key not in index:
                    index[key] = len(states)
                    states.append(key)
                    self.access.append(X)
                j = index[key]
                if X in self.is_nt:
                    gto[X] = j
                else:
                    act[X] = ("s", j)
            for (p, d), la in items.items():
                if d == len(self.rhs[p]):
                    for a in la:
                        new = ("acc", None) if p == 0 else ("r", p)
                        old = act.get(a)
                        if old is not None and old != new:
                            raise LRConflict("conflict in state %d on terminal %d: %r vs %r" % (k, a, old, new))
                        act[a] = new
            self.ACTION.append(act)
            self.GOTO.append(gto)
            k += 1
        self.n_states = len(states)
