"""Regular lexeme languages R_tau (GRID Sec. 2, layer L1): regex text -> Thompson
NFA -> subset-construction DFA for the union automaton of all terminals.

Test infrastructure (see package docstring).  Regex syntax: literal bytes,
escapes \\n \\t \\r \\xHH and \\<punct>, classes [...] with ranges and a leading
^ for negation, grouping ( ), alternation |, and the postfix operators * + ?.
Literal terminals ("select") are the concatenation of their bytes.

The DFA is the plain subset construction (no minimisation): a DFA state is the
frozenset of NFA states reachable on its input; the empty set is the dead state.
acc(q) = terminals whose accept state is in q; live(q) = terminals for which an
accepting state is reachable from q (the "live for some terminal" notion of
Def. 2).
"""
from __future__ import annotations


class RegexError(ValueError):
    pass


def _parse(pattern: bytes):
    pos = [0]
    n = len(pattern)

    def peek():
        return pattern[pos[0]] if pos[0] < n else None

    def take():
        c = pattern[pos[0]]
        pos[0] += 1
        return c

    def escape_byte():
        c = take()
        if c == ord("n"):
            return 10
        if c == ord("t"):
            return 9
        if c == ord("r"):
            return 13
        if c == ord("x"):
            h = pattern[pos[0]:pos[0] + 2]
            pos[0] += 2
            return int(h, 16)
        return c

    def parse_alt():
        branches = [parse_cat()]
        while peek() == ord("|"):
            take()
            branches.append(parse_cat())
        return ("alt", branches) if len(branches) > 1 else branches[0]

    def parse_cat():
        items = []
        while peek() is not None and peek() not in (ord("|"), ord(")")):
            items.append(parse_rep())
        return ("cat", items)

    def parse_rep():
        node = parse_atom()
        while peek() in (ord("*"), ord("+"), ord("?")):
            op = take()
            node = ({ord("*"): "star", ord("+"): "plus", ord("?"): "opt"}[op], node)
        return node

    def parse_atom():
        c = take()
        if c == ord("("):
            node = parse_alt()
            if peek() != ord(")"):
                raise RegexError("missing )")
            take()
            return node
        if c == ord("["):
            neg = False
            if peek() == ord("^"):
                take()
                neg = True
            chars = set()
            first = True
            while True:
                if peek() is None:
                    raise RegexError("missing ]")
                if peek() == ord("]") and not first:
                    take()
                    break
                first = False
                a = take()
                if a == ord("\\"):
                    a = escape_byte()
                if peek() == ord("-") and pos[0] + 1 < n and pattern[pos[0] + 1] != ord("]"):
                    take()
                    b = take()
                    if b == ord("\\"):
                        b = escape_byte()
                    chars.update(range(a, b + 1))
                else:
                    chars.add(a)
            if neg:
                chars = set(range(256)) - chars
            return ("set", frozenset(chars))
        if c == ord("\\"):
            return ("set", frozenset([escape_byte()]))
        if c in (ord("*"), ord("+"), ord("?"), ord("|"), ord(")")):
            raise RegexError("unexpected operator")
        return ("set", frozenset([c]))

    node = parse_alt()
    if pos[0] != n:
        raise RegexError("trailing input")
    return node


def literal_ast(lit: bytes):
    return ("cat", [("set", frozenset([c])) for c in lit])


def parse_regex(pattern: bytes):
    return _parse(pattern)


class NFA:
    """Thompson NFA: eps[s] = list of eps targets, edges[s] = list of (byteset, target)."""

    def __init__(self):
        self.eps = []
        self.edges = []

    def new(self):
        self.eps.append([])
        self.edges.append([])
        return len(self.eps) - 1

    def build(self, node):
        """Return (start, accept) for the sub-automaton of ``node``."""
        kind = node[0]
        if kind == "set":
            s, a = self.new(), self.new()
            self.edges[s].append((node[1], a))
            return s, a
        if kind == "cat":
            s = self.new()
            cur = s
            for item in node[1]:
                i_s, i_a = self.build(item)
                self.eps[cur].append(i_s)
                cur = i_a
            return s, cur
        if kind == "alt":
            s, a = self.new(), self.new()
            for br in node[1]:
                b_s, b_a = self.build(br)
                self.eps[s].append(b_s)
                self.eps[b_a].append(a)
            return s, a
        if kind in ("star", "plus", "opt"):
            s, a = self.new(), self.new()
            i_s, i_a = self.build(node[1])
            self.eps[s].append(i_s)
            if kind in ("star", "opt"):
                self.eps[s].append(a)
            self.eps[i_a].append(a)
            if kind in ("star", "plus"):
                self.eps[i_a].append(i_s)
            return s, a
        raise RegexError("bad node")


class UnionDFA:
    """Union automaton over all terminals (subset construction over bytes).

    States are numbered 0 = dead, 1 = start.  ``delta[q][b]`` is the next state,
    ``acc[q]`` / ``live[q]`` are frozensets of terminal ids."""

    def __init__(self, asts):
        nfa = NFA()
        start = nfa.new()
        accept_of = {}
        for tid, ast in enumerate(asts):
            s, a = nfa.build(ast)
            nfa.eps[start].append(s)
            accept_of[a] = tid
        self.nfa = nfa

        def closure(states):
            stack = list(states)
            seen = set(states)
            while stack:
                x = stack.pop()
                for y in nfa.eps[x]:
                    if y not in seen:
                        seen.add(y)
                        stack.append(y)
            return frozenset(seen)

        dead = frozenset()
        init = closure([start])
        index = {dead: 0, init: 1}
        order = [dead, init]
        delta = [[0] * 256, None]
        work = [init]
        while work:
            S = work.pop()
            row = [0] * 256
            moves = {}
            for x in S:
                for bs, y in nfa.edges[x]:
                    for b in bs:
                        moves.setdefault(b, set()).add(y)
            cache = {}
            for b, ys in moves.items():
                key = frozenset(ys)
                T = cache.get(key)
                if T is None:
                    T = closure(ys)
                    cache[key] = T
                if T not in index:
                    index[T] = len(order)
                    order.append(T)
                    delta.append(None)
                    work.append(T)
                row[b] = index[T]
            delta[index[S]] = row
        self.delta = delta
        self.n_states = len(order)
        self.acc = [frozenset(accept_of[x] for x in S if x in accept_of) for S in order]
        # live[q]: terminals with an accepting state reachable from q (reverse search).
        preds = [set() for _ in order]
        for q in range(self.n_states):
            for b in range(256):
                preds[delta[q][b]].add(q)
        live = [set() for _ in order]
        for tid in range(len(asts)):
            stack = [q for q in range(self.n_states) if tid in self.acc[q]]
            seen = set(stack)
            while stack:
                q = stack.pop()
                for p in preds[q]:
                    if p not in seen:
                        seen.add(p)
                        stack.append(p)
            for q in seen:
                if q != 0:
                    live[q].add(tid)
        self.live = [frozenset(s) for s in live]

    def run(self, data: bytes, q: int = 1) -> int:
        for b in data:
            q = self.delta[q][b]
        return q
