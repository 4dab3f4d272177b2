// Host-side compiler of libgrid: grammar text -> role projection -> reduction
// -> LALR(1); terminal regexes -> minimised union DFA; schema lexicons ->
// identifier trie; tokenizer spellings -> DFS-ordered byte trie.
//
// GRID Sec. 2 (three grammar layers, maximal munch with contextual
// resolution, L2 reducedness, L3 precondition W_c subset of R_c), Fig. 1
// (offline pipeline), Def. 3 (token trie with alias classes).
//
// The LALR(1) tables are built from the LR(0) collection with the classic
// spontaneous-generation / propagation computation of lookaheads; the lexer is
// Thompson NFA -> subset construction -> Moore minimisation -> byte classes.

#include <algorithm>
#include <array>
#include <cstring>
#include <map>
#include <set>
#include <sstream>
#include <string>
#include <unordered_map>
#include <vector>

#include "grid_blake2b.cuh"
#include "grid_internal.h"

namespace grid {

static thread_local std::string g_last_error;

int set_error(int code, const std::string& msg) {
  g_last_error = msg;
  return code;
}

namespace {

// ---------------------------------------------------------------------------
// small bitsets
// ---------------------------------------------------------------------------
struct Bytes256 {
  uint64_t w[4] = {0, 0, 0, 0};
  void set(int b) { w[b >> 6] |= 1ull << (b & 63); }
  bool has(int b) const { return (w[b >> 6] >> (b & 63)) & 1; }
};

struct Bits128 {
  uint64_t w[2] = {0, 0};
  void set(int b) { w[b >> 6] |= 1ull << (b & 63); }
  bool has(int b) const { return (w[b >> 6] >> (b & 63)) & 1; }
  bool merge(const Bits128& o) {
    uint64_t a = w[0] | o.w[0], b = w[1] | o.w[1];
    bool ch = (a != w[0]) || (b != w[1]);
    w[0] = a;
    w[1] = b;
    return ch;
  }
  bool operator<(const Bits128& o) const { return w[0] != o.w[0] ? w[0] < o.w[0] : w[1] < o.w[1]; }
  bool operator==(const Bits128& o) const { return w[0] == o.w[0] && w[1] == o.w[1]; }
};

// ---------------------------------------------------------------------------
// Thompson NFA built directly while parsing each regex
// ---------------------------------------------------------------------------
struct Nfa {
  std::vector<std::vector<int>> eps;
  std::vector<std::vector<std::pair<Bytes256, int>>> edge;
  int add() {
    eps.emplace_back();
    edge.emplace_back();
    return (int)eps.size() - 1;
  }
};

struct Frag {
  int s, a;
};

struct RegexParser {
  Nfa& n;
  const std::string& p;
  size_t i = 0;
  std::string err;
  RegexParser(Nfa& nfa, const std::string& pat) : n(nfa), p(pat) {}

  bool at_end() const { return i >= p.size(); }
  int peek() const { return at_end() ? -1 : (unsigned char)p[i]; }

  Frag single(const Bytes256& b) {
    Frag f{n.add(), n.add()};
    n.edge[f.s].push_back({b, f.a});
    return f;
  }
  Frag empty() {
    int s = n.add();
    return {s, s};
  }
  Frag cat(Frag x, Frag y) {
    n.eps[x.a].push_back(y.s);
    return {x.s, y.a};
  }

  int escape() {
    if (at_end()) {
      err = "dangling escape";
      return 0;
    }
    int c = (unsigned char)p[i++];
    switch (c) {
      case 'n': return 10;
      case 't': return 9;
      case 'r': return 13;
      case 'x': {
        if (i + 2 > p.size()) {
          err = "bad \\x escape";
          return 0;
        }
        int v = (int)std::strtol(p.substr(i, 2).c_str(), nullptr, 16);
        i += 2;
        return v;
      }
      default: return c;
    }
  }

  Frag alt() {
    Frag f = seq();
    while (peek() == '|') {
      ++i;
      Frag g = seq();
      Frag h{n.add(), n.add()};
      n.eps[h.s].push_back(f.s);
      n.eps[h.s].push_back(g.s);
      n.eps[f.a].push_back(h.a);
      n.eps[g.a].push_back(h.a);
      f = h;
    }
    return f;
  }

  Frag seq() {
    Frag f = empty();
    while (!at_end() && peek() != '|' && peek() != ')') {
      if (!err.empty()) return f;
      f = cat(f, rep());
    }
    return f;
  }

  Frag rep() {
    Frag f = atom();
    while (peek() == '*' || peek() == '+' || peek() == '?') {
      int op = p[i++];
      Frag h{n.add(), n.add()};
      n.eps[h.s].push_back(f.s);
      if (op != '+') n.eps[h.s].push_back(h.a);
      n.eps[f.a].push_back(h.a);
      if (op != '?') n.eps[f.a].push_back(f.s);
      f = h;
    }
    return f;
  }

  Frag atom() {
    if (at_end()) {
      err = "unexpected end of regex";
      return empty();
    }
    int c = (unsigned char)p[i++];
    if (c == '(') {
      Frag f = alt();
      if (peek() != ')') {
        err = "missing )";
        return f;
      }
      ++i;
      return f;
    }
    if (c == '[') {
      bool neg = false;
      if (peek() == '^') {
        neg = true;
        ++i;
      }
      Bytes256 b;
      bool first = true;
      for (;;) {
        if (at_end()) {
          err = "missing ]";
          return empty();
        }
        if (peek() == ']' && !first) {
          ++i;
          break;
        }
        first = false;
        int lo = (unsigned char)p[i++];
        if (lo == '\\') lo = escape();
        if (peek() == '-' && i + 1 < p.size() && p[i + 1] != ']') {
          ++i;
          int hi = (unsigned char)p[i++];
          if (hi == '\\') hi = escape();
          for (int x = lo; x <= hi; ++x) b.set(x);
        } else {
          b.set(lo);
        }
      }
      if (neg) {
        Bytes256 nb;
        for (int x = 0; x < 256; ++x)
          if (!b.has(x)) nb.set(x);
        b = nb;
      }
      return single(b);
    }
    if (c == '\\') {
      Bytes256 b;
      b.set(escape());
      return single(b);
    }
    if (c == '*' || c == '+' || c == '?' || c == '|' || c == ')') {
      err = "unexpected operator in regex";
      return empty();
    }
    Bytes256 b;
    b.set(c);
    return single(b);
  }
};

// ---------------------------------------------------------------------------
// grammar text
// ---------------------------------------------------------------------------
struct Terminal {
  std::string name;
  bool ignored;
  bool literal;
  std::string pattern;
};

struct RawProd {
  std::string lhs;
  std::vector<std::string> rhs;
  std::string tag;
};

struct RawGrammar {
  std::vector<Terminal> terms;
  std::vector<std::string> cats;
  std::vector<RawProd> prods;
  std::string start;
};

std::string trim(const std::string& s) {
  size_t a = s.find_first_not_of(" \t\r");
  if (a == std::string::npos) return "";
  size_t b = s.find_last_not_of(" \t\r");
  return s.substr(a, b - a + 1);
}

std::vector<std::string> split_ws(const std::string& s) {
  std::istringstream is(s);
  std::vector<std::string> out;
  std::string w;
  while (is >> w) out.push_back(w);
  return out;
}

int parse_grammar_text(const std::string& text, RawGrammar& g) {
  std::istringstream in(text);
  std::string raw;
  int lineno = 0;
  while (std::getline(in, raw)) {
    ++lineno;
    std::string line = trim(raw);
    if (line.empty() || line[0] == '#') continue;
    auto fail = [&](const std::string& why) {
      return set_error(GRID_E_PARSE, "grammar line " + std::to_string(lineno) + ": " + why);
    };
    if (line.rfind("%token", 0) == 0 || line.rfind("%ignore", 0) == 0) {
      bool ign = line.rfind("%ignore", 0) == 0;
      std::string rest = trim(line.substr(ign ? 7 : 6));
      size_t sp = rest.find_first_of(" \t");
      if (sp == std::string::npos) return fail("terminal without pattern");
      Terminal t;
      t.name = rest.substr(0, sp);
      std::string spec = trim(rest.substr(sp));
      t.ignored = ign;
      if (spec.size() >= 2 && spec.front() == '"' && spec.back() == '"') {
        t.literal = true;
        std::string body = spec.substr(1, spec.size() - 2), lit;
        for (size_t k = 0; k < body.size(); ++k) {
          if (body[k] == '\\' && k + 1 < body.size()) {
            lit.push_back(body[k + 1]);
            ++k;
          } else {
            lit.push_back(body[k]);
          }
        }
        t.pattern = lit;
      } else if (spec.size() >= 2 && spec.front() == '/' && spec.back() == '/') {
        t.literal = false;
        std::string body = spec.substr(1, spec.size() - 2), pat;
        for (size_t k = 0; k < body.size(); ++k) {
          if (body[k] == '\\' && k + 1 < body.size() && body[k + 1] == '/') {
            pat.push_back('/');
            ++k;
          } else {
            pat.push_back(body[k]);
          }
        }
        t.pattern = pat;
      } else {
        return fail("terminal pattern must be \"literal\" or /regex/");
      }
      if (t.pattern.empty()) return fail("empty terminal pattern");
      for (auto& o : g.terms)
        if (o.name == t.name) return fail("duplicate terminal " + t.name);
      g.terms.push_back(t);
    } else if (line.rfind("%category", 0) == 0) {
      auto w = split_ws(line);
      if (w.size() != 2) return fail("bad %category");
      g.cats.push_back(w[1]);
    } else if (line.rfind("%start", 0) == 0) {
      auto w = split_ws(line);
      if (w.size() != 2) return fail("bad %start");
      g.start = w[1];
    } else {
      size_t ar = line.find("->");
      if (ar == std::string::npos) return fail("unrecognised line");
      RawProd p;
      p.lhs = trim(line.substr(0, ar));
      if (p.lhs.empty() || p.lhs.find_first_of(" \t") != std::string::npos) return fail("bad lhs");
      auto w = split_ws(line.substr(ar + 2));
      if (!w.empty() && w.back()[0] == '@') {
        p.tag = w.back().substr(1);
        w.pop_back();
      }
      if (w.size() == 1 && w[0] == "%empty") w.clear();
      p.rhs = w;
      g.prods.push_back(p);
    }
  }
  if (g.start.empty()) return set_error(GRID_E_PARSE, "grammar has no %start");
  if (g.terms.empty()) return set_error(GRID_E_PARSE, "grammar has no terminals");
  return GRID_OK;
}

// ---------------------------------------------------------------------------
// lexer: union DFA over all terminals
// ---------------------------------------------------------------------------
int build_lexer(const RawGrammar& rg, HostGrammar& h) {
  Nfa nfa;
  int start = nfa.add();
  std::vector<int> accept_of_state;  // NFA state -> terminal or -1
  std::vector<int> term_accept(rg.terms.size());
  for (size_t t = 0; t < rg.terms.size(); ++t) {
    const Terminal& tm = rg.terms[t];
    Frag f;
    if (tm.literal) {
      RegexParser rp(nfa, tm.pattern);
      f = rp.empty();
      for (unsigned char ch : tm.pattern) {
        Bytes256 b;
        b.set(ch);
        f = rp.cat(f, rp.single(b));
      }
    } else {
      RegexParser rp(nfa, tm.pattern);
      f = rp.alt();
      if (rp.err.empty() && !rp.at_end()) rp.err = "trailing characters";
      if (!rp.err.empty()) return set_error(GRID_E_PARSE, "regex of " + tm.name + ": " + rp.err);
    }
    nfa.eps[start].push_back(f.s);
    term_accept[t] = f.a;
  }
  const int NN = (int)nfa.eps.size();
  accept_of_state.assign(NN, -1);
  for (size_t t = 0; t < term_accept.size(); ++t) {
    if (accept_of_state[term_accept[t]] < 0) accept_of_state[term_accept[t]] = (int)t;
  }
  // several terminals never share an NFA accept state: each fragment has its own.
  auto closure = [&](std::vector<int> v) {
    std::vector<char> seen(NN, 0);
    std::vector<int> st = v;
    for (int x : v) seen[x] = 1;
    while (!st.empty()) {
      int x = st.back();
      st.pop_back();
      for (int y : nfa.eps[x])
        if (!seen[y]) {
          seen[y] = 1;
          st.push_back(y);
          v.push_back(y);
        }
    }
    std::sort(v.begin(), v.end());
    return v;
  };
  std::map<std::vector<int>, int> index;
  std::vector<std::vector<int>> sets;
  std::vector<std::array<int, 256>> delta;
  sets.push_back({});  // dead
  index[{}] = 0;
  delta.push_back({});
  delta[0].fill(0);
  std::vector<int> init = closure({start});
  index[init] = 1;
  sets.push_back(init);
  delta.push_back({});
  for (size_t k = 1; k < sets.size(); ++k) {
    std::vector<std::vector<int>> tgt(256);
    for (int x : sets[k])
      for (auto& e : nfa.edge[x])
        for (int b = 0; b < 256; ++b)
          if (e.first.has(b)) tgt[b].push_back(e.second);
    std::array<int, 256> row;
    std::map<std::vector<int>, int> local;
    for (int b = 0; b < 256; ++b) {
      if (tgt[b].empty()) {
        row[b] = 0;
        continue;
      }
      std::vector<int> key = tgt[b];
      std::sort(key.begin(), key.end());
      key.erase(std::unique(key.begin(), key.end()), key.end());
      auto lit = local.find(key);
      int id;
      if (lit != local.end()) {
        id = lit->second;
      } else {
        std::vector<int> cl = closure(key);
        auto it = index.find(cl);
        if (it == index.end()) {
          id = (int)sets.size();
          index[cl] = id;
          sets.push_back(cl);
          delta.push_back({});
        } else {
          id = it->second;
        }
        local[key] = id;
      }
      row[b] = id;
    }
    delta[k] = row;
    if (sets.size() > 60000) return set_error(GRID_E_TOO_LARGE, "lexer DFA exceeds 60000 states");
  }
  const int Q0 = (int)sets.size();
  std::vector<Bits128> acc0(Q0);
  for (int q = 0; q < Q0; ++q)
    for (int x : sets[q])
      if (accept_of_state[x] >= 0) acc0[q].set(accept_of_state[x]);

  // Moore minimisation: start from the partition by accepted-terminal set.
  std::vector<int> blk(Q0);
  {
    std::map<Bits128, int> m;
    for (int q = 0; q < Q0; ++q) {
      auto it = m.find(acc0[q]);
      if (it == m.end()) it = m.emplace(acc0[q], (int)m.size()).first;
      blk[q] = it->second;
    }
    int nb = (int)m.size();
    for (;;) {
      std::map<std::vector<int>, int> sig;
      std::vector<int> nblk(Q0);
      for (int q = 0; q < Q0; ++q) {
        std::vector<int> key(257);
        key[0] = blk[q];
        for (int b = 0; b < 256; ++b) key[b + 1] = blk[delta[q][b]];
        auto it = sig.find(key);
        if (it == sig.end()) it = sig.emplace(key, (int)sig.size()).first;
        nblk[q] = it->second;
      }
      int nn = (int)sig.size();
      blk.swap(nblk);
      if (nn == nb) break;
      nb = nn;
    }
  }
  // renumber: dead -> 0, start -> 1, the rest by first visit from the start.
  std::vector<int> newid(Q0, -1), rep;
  std::unordered_map<int, int> blk2new;
  auto visit = [&](int q) {
    auto it = blk2new.find(blk[q]);
    if (it != blk2new.end()) return it->second;
    int id = (int)rep.size();
    blk2new[blk[q]] = id;
    rep.push_back(q);
    return id;
  };
  visit(0);
  visit(1);
  for (size_t k = 0; k < rep.size(); ++k) {
    int q = rep[k];
    for (int b = 0; b < 256; ++b) visit(delta[q][b]);
  }
  if (blk[0] == blk[1]) return set_error(GRID_E_PARSE, "lexer accepts nothing");
  const int Q = (int)rep.size();
  std::vector<std::array<int, 256>> nd(Q);
  for (int k = 0; k < Q; ++k)
    for (int b = 0; b < 256; ++b) nd[k][b] = blk2new[blk[delta[rep[k]][b]]];
  // byte classes
  std::map<std::vector<int>, int> colmap;
  for (int b = 0; b < 256; ++b) {
    std::vector<int> col(Q);
    for (int q = 0; q < Q; ++q) col[q] = nd[q][b];
    auto it = colmap.find(col);
    if (it == colmap.end()) it = colmap.emplace(col, (int)colmap.size()).first;
    h.byte_class[b] = (uint8_t)it->second;
  }
  const int C = (int)colmap.size();
  if ((long)Q * C > (1l << 26) || Q > 65535) return set_error(GRID_E_TOO_LARGE, "lexer DFA too large");
  h.Q = Q;
  h.C = C;
  h.next.assign((size_t)Q * C, 0);
  for (int q = 0; q < Q; ++q)
    for (int b = 0; b < 256; ++b) h.next[(size_t)q * C + h.byte_class[b]] = (uint16_t)nd[q][b];
  h.acc.assign((size_t)Q * 4, 0);
  h.live.assign((size_t)Q * 4, 0);
  for (int q = 0; q < Q; ++q) {
    const Bits128& a = acc0[rep[q]];
    for (int t = 0; t < 128; ++t)
      if (a.has(t)) h.acc[q * 4 + (t >> 5)] |= 1u << (t & 31);
  }
  // live: reverse reachability from accepting states, per terminal.
  std::vector<std::vector<int>> preds(Q);
  for (int q = 0; q < Q; ++q) {
    std::set<int> seen;
    for (int b = 0; b < 256; ++b)
      if (seen.insert(nd[q][b]).second) preds[nd[q][b]].push_back(q);
  }
  for (size_t t = 0; t < rg.terms.size(); ++t) {
    std::vector<char> mark(Q, 0);
    std::vector<int> st;
    for (int q = 0; q < Q; ++q)
      if ((h.acc[q * 4 + (t >> 5)] >> (t & 31)) & 1) {
        mark[q] = 1;
        st.push_back(q);
      }
    while (!st.empty()) {
      int q = st.back();
      st.pop_back();
      for (int p : preds[q])
        if (!mark[p]) {
          mark[p] = 1;
          st.push_back(p);
        }
    }
    for (int q = 1; q < Q; ++q)
      if (mark[q]) h.live[q * 4 + (t >> 5)] |= 1u << (t & 31);
  }
  // P-LEX: accept-closed (every live successor of an accepting state accepts)
  for (int q = 1; q < Q; ++q) {
    bool accq = h.acc[q * 4] | h.acc[q * 4 + 1] | h.acc[q * 4 + 2] | h.acc[q * 4 + 3];
    if (!accq) continue;
    for (int b = 0; b < 256; ++b) {
      int r = nd[q][b];
      if (r == kDead) continue;
      bool accr = h.acc[r * 4] | h.acc[r * 4 + 1] | h.acc[r * 4 + 2] | h.acc[r * 4 + 3];
      if (!accr)
        return set_error(GRID_E_LEXER_PRECONDITION,
                         "lexer is not accept-closed: byte " + std::to_string(b) +
                             " leads from an accepting state to a live non-accepting one");
    }
  }
  // P-DELIM: a blank kills every accepting state of a non-ignored terminal,
  // and starts an ignored lexeme.
  for (int q = 1; q < Q; ++q) {
    bool nonign = false;
    for (int w = 0; w < 4; ++w)
      if (h.acc[q * 4 + w] & ~h.ignored[w]) nonign = true;
    if (nonign && nd[q][0x20] != kDead)
      return set_error(GRID_E_LEXER_PRECONDITION,
                       "lexer is not blank-delimited: a blank extends a non-ignored lexeme");
  }
  {
    int q = nd[kStart][0x20];
    bool ok = false;
    for (int w = 0; w < 4; ++w)
      if (q != kDead && (h.acc[q * 4 + w] & h.ignored[w])) ok = true;
    if (!ok)
      return set_error(GRID_E_LEXER_PRECONDITION, "no ignored terminal accepts a single blank");
  }
  return GRID_OK;
}

// ---------------------------------------------------------------------------
// role projection + reduction + LALR(1)
// ---------------------------------------------------------------------------
struct Prod {
  int lhs;               // nonterminal index
  std::vector<int> rhs;  // symbol ids: < T1 terminal, >= T1 nonterminal (id - T1)
};

int build_parser(const RawGrammar& rg, const char* role_keep, HostGrammar& h) {
  const int nterm = (int)rg.terms.size();
  const int T1 = nterm + 1;
  std::unordered_map<std::string, int> tid;
  for (int t = 0; t < nterm; ++t) tid[rg.terms[t].name] = t;
  std::set<std::string> nts;
  for (auto& p : rg.prods) nts.insert(p.lhs);
  for (auto& p : rg.prods)
    for (auto& s : p.rhs) {
      auto it = tid.find(s);
      if (it == tid.end()) {
        if (!nts.count(s)) return set_error(GRID_E_PARSE, "unknown symbol " + s);
      } else if (rg.terms[it->second].ignored) {
        return set_error(GRID_E_PARSE, "ignored terminal " + s + " used in a production");
      }
    }
  if (!nts.count(rg.start)) return set_error(GRID_E_PARSE, "start symbol has no production");
  // L2: production subset
  std::set<std::string> keep;
  bool keep_all = role_keep == nullptr;
  if (!keep_all) {
    std::string r(role_keep), cur;
    for (char c : r + ",") {
      if (c == ',') {
        if (!trim(cur).empty()) keep.insert(trim(cur));
        cur.clear();
      } else {
        cur.push_back(c);
      }
    }
  }
  std::vector<const RawProd*> P0;
  for (auto& p : rg.prods)
    if (p.tag.empty() || keep_all || keep.count(p.tag)) P0.push_back(&p);
  // useless-symbol elimination: generating, then reachable
  auto isT = [&](const std::string& s) { return tid.count(s) > 0; };
  std::set<std::string> gen;
  for (bool ch = true; ch;) {
    ch = false;
    for (auto* p : P0) {
      if (gen.count(p->lhs)) continue;
      bool ok = true;
      for (auto& s : p->rhs)
        if (!isT(s) && !gen.count(s)) ok = false;
      if (ok) {
        gen.insert(p->lhs);
        ch = true;
      }
    }
  }
  if (!gen.count(rg.start))
    return set_error(GRID_E_EMPTY_LANGUAGE, "the role-projected grammar generates no sentence");
  std::vector<const RawProd*> P1;
  for (auto* p : P0) {
    bool ok = gen.count(p->lhs) > 0;
    for (auto& s : p->rhs)
      if (!isT(s) && !gen.count(s)) ok = false;
    if (ok) P1.push_back(p);
  }
  std::set<std::string> reach{rg.start};
  for (bool ch = true; ch;) {
    ch = false;
    for (auto* p : P1)
      if (reach.count(p->lhs))
        for (auto& s : p->rhs)
          if (!isT(s) && reach.insert(s).second) ch = true;
  }
  // number nonterminals: 0 = S', then by first appearance as lhs
  std::unordered_map<std::string, int> ntid;
  std::vector<Prod> P;
  P.push_back({0, {T1 + 1}});  // S' -> start (start gets index 1 below)
  ntid["$S'"] = 0;
  ntid[rg.start] = 1;
  for (auto* p : P1)
    if (reach.count(p->lhs) && !ntid.count(p->lhs)) ntid.emplace(p->lhs, (int)ntid.size());
  for (auto* p : P1) {
    if (!reach.count(p->lhs)) continue;
    Prod q;
    q.lhs = ntid[p->lhs];
    for (auto& s : p->rhs) q.rhs.push_back(isT(s) ? tid[s] : T1 + ntid[s]);
    if (q.rhs.size() > 250) return set_error(GRID_E_TOO_LARGE, "production longer than 250 symbols");
    P.push_back(q);
  }
  const int NNT = (int)ntid.size();
  const int NP = (int)P.size();
  std::vector<std::vector<int>> by_lhs(NNT);
  for (int i = 0; i < NP; ++i) by_lhs[P[i].lhs].push_back(i);
  // nullable + FIRST over terminals
  std::vector<char> nullable(NNT, 0);
  std::vector<Bits128> first(NNT);
  for (bool ch = true; ch;) {
    ch = false;
    for (auto& p : P) {
      bool alln = true;
      for (int s : p.rhs) {
        if (s < T1) {
          if (!first[p.lhs].has(s)) {
            first[p.lhs].set(s);
            ch = true;
          }
          alln = false;
          break;
        }
        if (first[p.lhs].merge(first[s - T1])) ch = true;
        if (!nullable[s - T1]) {
          alln = false;
          break;
        }
      }
      if (alln && !nullable[p.lhs]) {
        nullable[p.lhs] = 1;
        ch = true;
      }
    }
  }
  // LR(0) collection; items packed as p*256 + dot
  auto item = [](int p, int d) { return p * 256 + d; };
  auto closure0 = [&](const std::vector<int>& kernel) {
    std::vector<int> out = kernel;
    std::vector<char> added(NNT, 0);
    for (size_t k = 0; k < out.size(); ++k) {
      int p = out[k] / 256, d = out[k] % 256;
      if (d < (int)P[p].rhs.size() && P[p].rhs[d] >= T1) {
        int B = P[p].rhs[d] - T1;
        if (!added[B]) {
          added[B] = 1;
          for (int q : by_lhs[B]) out.push_back(item(q, 0));
        }
      }
    }
    return out;
  };
  std::vector<std::vector<int>> kernels;
  std::map<std::vector<int>, int> kindex;
  std::vector<std::map<int, int>> trans;  // state -> symbol -> state
  kernels.push_back({item(0, 0)});
  kindex[kernels[0]] = 0;
  for (size_t s = 0; s < kernels.size(); ++s) {
    std::vector<int> cl = closure0(kernels[s]);
    std::map<int, std::vector<int>> next;
    for (int it : cl) {
      int p = it / 256, d = it % 256;
      if (d < (int)P[p].rhs.size()) next[P[p].rhs[d]].push_back(item(p, d + 1));
    }
    std::map<int, int> tr;
    for (auto& kv : next) {
      std::vector<int> k = kv.second;
      std::sort(k.begin(), k.end());
      auto f = kindex.find(k);
      int id;
      if (f == kindex.end()) {
        id = (int)kernels.size();
        kindex[k] = id;
        kernels.push_back(k);
      } else {
        id = f->second;
      }
      tr[kv.first] = id;
    }
    trans.push_back(tr);
    if (kernels.size() > 32000) return set_error(GRID_E_TOO_LARGE, "more than 32000 LALR states");
  }
  const int S = (int)kernels.size();
  // LR(1) closure of items with lookahead sets; '#' is bit T1 (T1 <= 127).
  const int HASH = T1;
  auto first_seq = [&](const std::vector<int>& rhs, int from, const Bits128& la) {
    Bits128 out;
    for (int k = from; k < (int)rhs.size(); ++k) {
      int s = rhs[k];
      if (s < T1) {
        out.set(s);
        return out;
      }
      out.merge(first[s - T1]);
      if (!nullable[s - T1]) return out;
    }
    out.merge(la);
    return out;
  };
  auto closure1 = [&](const std::vector<std::pair<int, Bits128>>& kern) {
    std::map<int, Bits128> cl;
    std::vector<int> work;
    for (auto& kv : kern) {
      cl[kv.first].merge(kv.second);
      work.push_back(kv.first);
    }
    while (!work.empty()) {
      int it = work.back();
      work.pop_back();
      int p = it / 256, d = it % 256;
      if (d >= (int)P[p].rhs.size() || P[p].rhs[d] < T1) continue;
      Bits128 la = first_seq(P[p].rhs, d + 1, cl[it]);
      for (int q : by_lhs[P[p].rhs[d] - T1]) {
        auto f = cl.find(item(q, 0));
        if (f == cl.end()) {
          cl[item(q, 0)] = la;
          work.push_back(item(q, 0));
        } else if (f->second.merge(la)) {
          work.push_back(item(q, 0));
        }
      }
    }
    return cl;
  };
  // lookahead propagation
  std::vector<std::vector<Bits128>> la(S);
  for (int s = 0; s < S; ++s) la[s].resize(kernels[s].size());
  auto kpos = [&](int s, int it) {
    auto& k = kernels[s];
    return (int)(std::lower_bound(k.begin(), k.end(), it) - k.begin());
  };
  struct Edge {
    int s0, k0, s1, k1;
  };
  std::vector<Edge> edges;
  for (int s = 0; s < S; ++s) {
    for (size_t k = 0; k < kernels[s].size(); ++k) {
      Bits128 h0;
      h0.set(HASH);
      auto cl = closure1({{kernels[s][k], h0}});
      for (auto& kv : cl) {
        int p = kv.first / 256, d = kv.first % 256;
        if (d >= (int)P[p].rhs.size()) continue;
        int X = P[p].rhs[d];
        int j = trans[s].at(X);
        int kk = kpos(j, item(p, d + 1));
        Bits128 spont = kv.second;
        if (spont.has(HASH)) {
          edges.push_back({s, (int)k, j, kk});
          spont.w[HASH >> 6] &= ~(1ull << (HASH & 63));
        }
        la[j][kk].merge(spont);
      }
    }
  }
  la[0][0].set(nterm);  // $end
  for (bool ch = true; ch;) {
    ch = false;
    for (auto& e : edges)
      if (la[e.s1][e.k1].merge(la[e.s0][e.k0])) ch = true;
  }
  // the symbol entering each state, for the audit's node hash
  {
    std::vector<std::string> ntname(NNT);
    for (auto& kv : ntid) ntname[kv.second] = kv.first;
    std::map<std::string, int> rank;  // nts is ordered by name (bytes)
    for (auto& n : nts) rank.emplace(n, (int)rank.size());
    h.acc_sym.assign(S, 0xFFFFFFFFu);
    for (int s = 1; s < S; ++s) {
      const int it = kernels[s][0], p = it / 256, d = it % 256;  // every kernel item of s > 0 has d >= 1
      const int X = P[p].rhs[d - 1];
      h.acc_sym[s] = X < T1 ? (uint32_t)X : ((1u << 16) | (uint32_t)rank.at(ntname[X - T1]));
    }
  }
  // kernel items and productions for the reserve completion
  h.kitem_off.assign(1, 0);
  h.kitem_p.clear();
  h.kitem_d.clear();
  for (int s = 0; s < S; ++s) {
    for (int it : kernels[s]) {
      h.kitem_p.push_back(it / 256);
      h.kitem_d.push_back(it % 256);
    }
    h.kitem_off.push_back((int32_t)h.kitem_p.size());
  }
  h.prod_off.assign(1, 0);
  h.prod_rhs.clear();
  for (auto& pr : P) {
    for (int x : pr.rhs) h.prod_rhs.push_back(x);
    h.prod_off.push_back((int32_t)h.prod_rhs.size());
  }
  // tables
  h.T1 = T1;
  h.S = S;
  h.NNT = NNT;
  h.P = NP;
  h.action.assign((size_t)S * T1, 0);
  h.go.assign((size_t)S * NNT, 0xFFFF);
  h.plen.resize(NP);
  h.plhs.resize(NP);
  for (int i = 0; i < NP; ++i) {
    h.plen[i] = (uint8_t)P[i].rhs.size();
    h.plhs[i] = (uint16_t)P[i].lhs;
  }
  auto sym_name = [&](int s) { return s < nterm ? rg.terms[s].name : std::string("$end"); };
  for (int s = 0; s < S; ++s) {
    std::vector<std::pair<int, Bits128>> kern;
    for (size_t k = 0; k < kernels[s].size(); ++k) kern.push_back({kernels[s][k], la[s][k]});
    auto cl = closure1(kern);
    for (auto& kv : trans[s]) {
      if (kv.first < T1)
        h.action[(size_t)s * T1 + kv.first] = (int16_t)(kv.second + 1);
      else
        h.go[(size_t)s * NNT + (kv.first - T1)] = (uint16_t)kv.second;
    }
    for (auto& kv : cl) {
      int p = kv.first / 256, d = kv.first % 256;
      if (d != (int)P[p].rhs.size()) continue;
      for (int a = 0; a < T1; ++a) {
        if (!kv.second.has(a)) continue;
        int16_t want = (p == 0) ? kAccept : (int16_t)(-(p + 1));
        int16_t& cell = h.action[(size_t)s * T1 + a];
        if (cell != 0 && cell != want) {
          std::string what = cell > 0 && cell != kAccept ? "shift/reduce" : "reduce/reduce";
          return set_error(GRID_E_LALR_CONFLICT, what + " conflict in LALR state " + std::to_string(s) +
                                                     " on terminal " + sym_name(a));
        }
        cell = want;
      }
    }
  }
  return GRID_OK;
}

// ---------------------------------------------------------------------------
// L3 lexicons -> identifier trie over the union of all W_c
// ---------------------------------------------------------------------------
int build_lexicons(const RawGrammar& rg, const grid_lexicon* lex, int n_lex, HostGrammar& h) {
  std::unordered_map<std::string, int> tid;
  for (int t = 0; t < (int)rg.terms.size(); ++t) tid[rg.terms[t].name] = t;
  if (rg.cats.size() > 32) return set_error(GRID_E_TOO_LARGE, "more than 32 categories");
  h.n_cat = (int)rg.cats.size();
  h.cat_term.clear();
  for (auto& c : rg.cats) {
    auto it = tid.find(c);
    if (it == tid.end()) return set_error(GRID_E_PARSE, "category " + c + " is not a terminal");
    if (rg.terms[it->second].ignored) return set_error(GRID_E_PARSE, "category " + c + " is ignored");
    h.cat_term.push_back(it->second);
    h.catmask[it->second >> 5] |= 1u << (it->second & 31);
  }
  // every word, checked against its category's regex, with its category
  struct Word {
    const uint8_t* p;
    int len, cat;
  };
  std::vector<Word> all;
  {
    size_t n = 0;
    for (int i = 0; i < n_lex; ++i) n += (size_t)std::max(0, lex[i].n_words);
    all.reserve(n);
  }
  for (int i = 0; i < n_lex; ++i) {
    const grid_lexicon& L = lex[i];
    if (!L.category) return set_error(GRID_E_INVALID_ARG, "lexicon without category");
    int cat = -1;
    for (int c = 0; c < h.n_cat; ++c)
      if (rg.cats[c] == L.category) cat = c;
    if (cat < 0) return set_error(GRID_E_INVALID_ARG, std::string("unknown lexicon category ") + L.category);
    if (L.n_words < 0 || (L.n_words > 0 && (!L.words || !L.offsets)))
      return set_error(GRID_E_INVALID_ARG, "bad lexicon arrays");
    const int term = h.cat_term[cat];
    for (int w = 0; w < L.n_words; ++w) {
      int64_t a = L.offsets[w], b = L.offsets[w + 1];
      if (b <= a) return set_error(GRID_E_INVALID_ARG, "empty or negative-length lexicon word");
      if (b - a > (1 << 30)) return set_error(GRID_E_TOO_LARGE, "lexicon word longer than 2^30 bytes");
      // W_c subset of R_c: the word must reach a state accepting the category
      int q = kStart;
      for (int64_t k = a; k < b && q != kDead; ++k) q = h.next[(size_t)q * h.C + h.byte_class[L.words[k]]];
      if (q == kDead || !((h.acc[q * 4 + (term >> 5)] >> (term & 31)) & 1))
        return set_error(GRID_E_LEXICON_NOT_IN_REGEX,
                         "lexicon word '" + std::string((const char*)L.words + a, (size_t)(b - a)) +
                             "' is not in the regex of " + rg.cats[cat]);
      all.push_back(Word{L.words + a, (int)(b - a), cat});
    }
  }
  // the trie in preorder from the words in byte order: a word adds nodes only
  // after its longest common prefix with the word before it, so each node's
  // children appear in increasing byte order
  {
    // sort on the first 8 bytes as a big-endian key (zero padded: where two
    // keys differ they order as the words do), the full comparison only on
    // equal keys
    std::vector<std::pair<uint64_t, int>> kv(all.size());
    for (size_t i = 0; i < all.size(); ++i) {
      uint64_t key = 0;
      for (int k = 0; k < 8; ++k) key = (key << 8) | (k < all[i].len ? all[i].p[k] : 0u);
      kv[i] = {key, (int)i};
    }
    std::sort(kv.begin(), kv.end(), [&](const std::pair<uint64_t, int>& x, const std::pair<uint64_t, int>& y) {
      if (x.first != y.first) return x.first < y.first;
      const Word &a = all[x.second], &b = all[y.second];
      const int c = std::memcmp(a.p, b.p, (size_t)std::min(a.len, b.len));
      return c != 0 ? c < 0 : a.len < b.len;
    });
    std::vector<Word> sorted(all.size());
    for (size_t i = 0; i < all.size(); ++i) sorted[i] = all[kv[i].second];
    all.swap(sorted);
  }
  size_t bytes = 1;
  for (const Word& w : all) bytes += (size_t)w.len;  // bounds the node count
  std::vector<int> parent{-1};
  std::vector<uint8_t> edge{0};
  std::vector<uint32_t> pc(1, 0), wc(1, 0);
  parent.reserve(bytes);
  edge.reserve(bytes);
  pc.reserve(bytes);
  wc.reserve(bytes);
  std::vector<int> path{0};  // path[d]: the current word's node at depth d
  const Word* prev = nullptr;
  for (const Word& w : all) {
    int l = 0;
    if (prev)
      while (l < prev->len && l < w.len && prev->p[l] == w.p[l]) ++l;
    path.resize(l + 1);
    for (int k = l; k < w.len; ++k) {
      path.push_back((int)parent.size());
      parent.push_back(path[k]);
      edge.push_back(w.p[k]);
      pc.push_back(0);
      wc.push_back(0);
    }
    const uint32_t bit = 1u << w.cat;
    for (int k = 0; k <= w.len; ++k) pc[path[k]] |= bit;
    wc[path[w.len]] |= bit;
    prev = &w;
  }
  // the flat arrays in BFS order with children sorted by byte.  Nodes of one
  // depth appear in preorder in the order of their prefixes, which is also
  // their BFS order, so BFS numbering is preorder stably sorted by depth; the
  // children of a node then get consecutive BFS ids, and listing edges by
  // their parents' BFS ids lists them by their children's: edge e leads to
  // BFS node e + 1.
  const int N = (int)parent.size();
  std::vector<int> depth(N, 0), at;  // at[d]: next BFS id at depth d
  int maxd = 0;
  for (int v = 1; v < N; ++v) {
    depth[v] = depth[parent[v]] + 1;  // parents come before children in preorder
    maxd = std::max(maxd, depth[v]);
  }
  at.assign(maxd + 2, 0);
  for (int v = 0; v < N; ++v) ++at[depth[v] + 1];
  for (int d = 0; d <= maxd; ++d) at[d + 1] += at[d];
  std::vector<int> bfs(N);
  for (int v = 0; v < N; ++v) bfs[v] = at[depth[v]]++;
  h.LN = N;
  h.lx_cstart.assign(N + 1, 0);
  h.lx_cbyte.assign(std::max(0, N - 1), 0);
  h.lx_cnode.resize(std::max(0, N - 1));
  h.lx_pcats.assign(N, 0);
  h.lx_wcats.assign(N, 0);
  for (int v = 0; v < N; ++v) {
    const int k = bfs[v];
    h.lx_pcats[k] = pc[v];
    h.lx_wcats[k] = wc[v];
    if (v > 0) {
      h.lx_cbyte[k - 1] = edge[v];
      ++h.lx_cstart[bfs[parent[v]] + 1];  // child counts, summed below
    }
  }
  for (int k = 0; k < N; ++k) h.lx_cstart[k + 1] += h.lx_cstart[k];
  for (int e = 0; e < N - 1; ++e) h.lx_cnode[e] = e + 1;
  return GRID_OK;
}

// Tables of the reserve completion that depend on the grammar and lexicons
// only (Sec. 5, Prop. 9; see include/grid.h, grid_reserve).
int build_completion_tables(const RawGrammar& rg, HostGrammar& h) {
  const int Q = h.Q, T1 = h.T1, LN = h.LN, NC = std::max(1, h.n_cat);
  auto has = [](const std::vector<uint32_t>& v, int q, int t) { return (v[(size_t)q * 4 + (t >> 5)] >> (t & 31)) & 1u; };
  auto step = [&](int q, int b) { return (int)h.next[(size_t)q * h.C + h.byte_class[b]]; };
  auto is_cat = [&](int t) { return (h.catmask[t >> 5] >> (t & 31)) & 1u; };
  auto is_ign = [&](int t) { return (h.ignored[t >> 5] >> (t & 31)) & 1u; };
  // the emission candidates of a lexeme at DFA state q with lexicon word
  // categories wc: its first one (lowest terminal index), or -1
  auto first_cand = [&](int q, uint32_t wc) {
    for (int t = 0; t < h.n_term; ++t) {
      if (!has(h.acc, q, t)) continue;
      if (is_cat(t)) {
        int c = -1;
        for (int k = 0; k < h.n_cat; ++k)
          if (h.cat_term[k] == t) c = k;
        if (c < 0 || !((wc >> c) & 1u)) continue;
      }
      return t;
    }
    return -1;
  };
  // lexicon trie: parent, edge byte and DFA state of every node (BFS ids)
  std::vector<int> par(LN, -1), qn(LN, kStart);
  std::vector<uint8_t> eb(LN, 0);
  for (int n = 0; n < LN; ++n)
    for (int e = h.lx_cstart[n]; e < h.lx_cstart[n + 1]; ++e) {
      const int ch = h.lx_cnode[e];
      par[ch] = n;
      eb[ch] = h.lx_cbyte[e];
      qn[ch] = qn[n] == kDead ? kDead : step(qn[n], h.lx_cbyte[e]);
    }
  // shortest word below each node per category (children in byte order, so
  // the first child reaching the minimum gives the smallest word)
  h.lx_wdist.assign((size_t)LN * NC, 0xFFFF);
  h.lx_wbyte.assign((size_t)LN * NC, 0);
  for (int n = LN - 1; n >= 0; --n)
    for (int c = 0; c < h.n_cat; ++c) {
      uint16_t& d = h.lx_wdist[(size_t)n * NC + c];
      if ((h.lx_wcats[n] >> c) & 1u) {
        d = 0;
        continue;
      }
      for (int e = h.lx_cstart[n]; e < h.lx_cstart[n + 1]; ++e) {
        const uint16_t dc = h.lx_wdist[(size_t)h.lx_cnode[e] * NC + c];
        if (dc != 0xFFFF && dc + 1 < d) {
          d = (uint16_t)(dc + 1);
          h.lx_wbyte[(size_t)n * NC + c] = h.lx_cbyte[e];
        }
      }
    }
  // shortest accepting continuation per (DFA state, terminal), smallest first byte
  h.dfa_tdist.assign((size_t)Q * T1, 0xFF);
  h.dfa_tbyte.assign((size_t)Q * T1, 0);
  for (int q = 1; q < Q; ++q)
    for (int t = 0; t < h.n_term; ++t)
      if (has(h.acc, q, t)) h.dfa_tdist[(size_t)q * T1 + t] = 0;
  {
    // breadth-first from the accepting states over reversed transitions, per
    // terminal; then the first byte: the smallest one whose successor is one
    // step closer (byte classes visited in order of their smallest byte)
    std::vector<int> cls_first(h.C, -1), order;
    for (int b = 0; b < 256; ++b)
      if (cls_first[h.byte_class[b]] < 0) {
        cls_first[h.byte_class[b]] = b;
        order.push_back(h.byte_class[b]);
      }
    std::vector<std::vector<int>> rev(Q);
    for (int q = 1; q < Q; ++q)
      for (int c = 0; c < h.C; ++c) {
        const int r = h.next[(size_t)q * h.C + c];
        if (r != kDead) rev[r].push_back(q);
      }
    std::vector<int> queue;
    for (int t = 0; t < h.n_term; ++t) {
      queue.clear();
      for (int q = 1; q < Q; ++q)
        if (h.dfa_tdist[(size_t)q * T1 + t] == 0) queue.push_back(q);
      for (size_t k = 0; k < queue.size(); ++k) {
        const int r = queue[k];
        const uint8_t dr = h.dfa_tdist[(size_t)r * T1 + t];
        if (dr >= 0xFE) continue;
        for (int q : rev[r])
          if (h.dfa_tdist[(size_t)q * T1 + t] == 0xFF) {
            h.dfa_tdist[(size_t)q * T1 + t] = (uint8_t)(dr + 1);
            queue.push_back(q);
          }
      }
      for (int q = 1; q < Q; ++q) {
        const uint8_t d = h.dfa_tdist[(size_t)q * T1 + t];
        if (d == 0 || d == 0xFF) continue;
        for (int c : order) {
          const int r = h.next[(size_t)q * h.C + c];
          if (r != kDead && h.dfa_tdist[(size_t)r * T1 + t] == d - 1) {
            h.dfa_tbyte[(size_t)q * T1 + t] = (uint8_t)cls_first[c];
            break;
          }
        }
      }
    }
  }
  // separator per state: a byte after which the lexer is where it would be
  // had the pending lexeme been emitted and the byte started an ignored
  // lexeme that stays ignored (the byte ends the lexeme, or extends an
  // ignored one into that same state, as a blank after a blank); the blank
  // when it qualifies
  h.sep_byte.assign(Q, -1);
  auto sep_ok = [&](int q, int b) {
    const int r = step(kStart, b);
    if (r == kDead) return false;
    const int x = step(q, b);
    if (x != kDead && x != r) return false;
    bool acc_ign = false, live_other = false;
    for (int t = 0; t < h.n_term; ++t) {
      if (has(h.acc, r, t) && is_ign(t)) acc_ign = true;
      if (has(h.live, r, t) && !is_ign(t)) live_other = true;
    }
    return acc_ign && !live_other;
  };
  for (int q = 1; q < Q; ++q) {
    if (sep_ok(q, ' ')) {
      h.sep_byte[q] = ' ';
      continue;
    }
    for (int b = 0; b < 256; ++b)
      if (sep_ok(q, b)) {
        h.sep_byte[q] = (int16_t)b;
        break;
      }
  }
  // the lexeme rendering each non-ignored terminal: the shortest (then
  // smallest) string whose first emission candidate is the terminal; for a
  // category a word of its lexicon
  h.render_lex.assign(T1, std::string());
  std::vector<char> done(T1, 0);
  auto word_of = [&](int n) {
    std::string w;
    for (int x = n; x > 0; x = par[x]) w.push_back((char)eb[x]);
    std::reverse(w.begin(), w.end());
    return w;
  };
  int cat_todo = h.n_cat;
  for (int n = 1; n < LN && cat_todo > 0; ++n) {  // BFS order: by length, then bytes
    if (!h.lx_wcats[n] || qn[n] == kDead) continue;
    const int t = first_cand(qn[n], h.lx_wcats[n]);
    if (t >= 0 && is_cat(t) && !done[t]) {
      done[t] = 1;
      h.render_lex[t] = word_of(n);
      --cat_todo;
    }
  }
  // literal terminals: their literal, if it is their own first candidate
  for (int t = 0; t < h.n_term; ++t) {
    if (is_ign(t) || is_cat(t) || !rg.terms[t].literal) continue;
    done[t] = 1;
    const std::string& lit = rg.terms[t].pattern;
    int q = kStart, lx = LN > 0 ? 0 : -1;
    for (unsigned char b : lit) {
      q = q == kDead ? kDead : step(q, b);
      int nl = -1;
      if (lx >= 0)
        for (int e = h.lx_cstart[lx]; e < h.lx_cstart[lx + 1]; ++e)
          if (h.lx_cbyte[e] == b) nl = h.lx_cnode[e];
      lx = nl;
    }
    if (q != kDead && first_cand(q, lx >= 0 ? h.lx_wcats[lx] : 0u) == t) h.render_lex[t] = lit;
  }
  {
    // the other terminals: breadth-first over (DFA state, lexicon node) pairs
    // in byte order, up to 32 bytes
    int todo = 0;
    for (int t = 0; t < h.n_term; ++t)
      if (!is_ign(t) && !is_cat(t) && !done[t]) ++todo;
    struct Node {
      int q, lx;
      std::string s;
    };
    std::vector<Node> level{{kStart, LN > 0 ? 0 : -1, std::string()}};
    std::unordered_map<int64_t, char> seen;
    seen[(int64_t)kStart * (LN + 1) + (LN > 0 ? 1 : 0)] = 1;
    for (int len = 1; len <= 32 && todo > 0 && !level.empty(); ++len) {
      std::vector<Node> nxt;
      for (const Node& nd : level)
        for (int b = 0; b < 256; ++b) {
          const int r = step(nd.q, b);
          if (r == kDead) continue;
          int lx = -1;
          if (nd.lx >= 0)
            for (int e = h.lx_cstart[nd.lx]; e < h.lx_cstart[nd.lx + 1]; ++e)
              if (h.lx_cbyte[e] == b) lx = h.lx_cnode[e];
          const int64_t key = (int64_t)r * (LN + 1) + (lx + 1);
          if (seen.count(key)) continue;
          seen[key] = 1;
          Node m{r, lx, nd.s + (char)b};
          const int t = first_cand(r, lx >= 0 ? h.lx_wcats[lx] : 0u);
          if (t >= 0 && !is_cat(t) && !is_ign(t) && !done[t]) {
            done[t] = 1;
            h.render_lex[t] = m.s;
            --todo;
          }
          nxt.push_back(std::move(m));
        }
      level.swap(nxt);
    }
  }
  return GRID_OK;
}

}  // namespace
}  // namespace grid

using namespace grid;

extern "C" size_t grid_last_error(char* buf, size_t n) {
  const std::string& e = g_last_error;
  if (buf && n) {
    size_t k = std::min(n - 1, e.size());
    std::memcpy(buf, e.data(), k);
    buf[k] = 0;
  }
  return e.size();
}

extern "C" int grid_compile(const char* grammar_text, size_t len, const char* role_keep,
                            const grid_lexicon* lex, int32_t n_lex, const grid_options* opt,
                            grid_grammar** out) {
  if (!grammar_text || !out || n_lex < 0 || (n_lex > 0 && !lex))
    return set_error(GRID_E_INVALID_ARG, "grid_compile: bad arguments");
  *out = nullptr;
  RawGrammar rg;
  int rc = parse_grammar_text(std::string(grammar_text, len), rg);
  if (rc) return rc;
  if (rg.terms.size() > 126) return set_error(GRID_E_TOO_LARGE, "more than 126 terminals");
  auto* g = new grid_grammar();
  HostGrammar& h = g->h;
  h.n_term = (int)rg.terms.size();
  h.T1 = h.n_term + 1;
  for (int t = 0; t < h.n_term; ++t) {
    h.term_names.push_back(rg.terms[t].name);
    if (rg.terms[t].ignored) h.ignored[t >> 5] |= 1u << (t & 31);
  }
  if (opt && opt->max_depth > 0) h.max_depth = opt->max_depth;
  if (h.max_depth < 2 || h.max_depth > (1 << 20)) {
    delete g;
    return set_error(GRID_E_INVALID_ARG, "max_depth out of range");
  }
  if ((rc = build_lexer(rg, h)) || (rc = build_parser(rg, role_keep, h)) ||
      (rc = build_lexicons(rg, lex, n_lex, h)) || (rc = build_completion_tables(rg, h))) {
    delete g;
    return rc;
  }
  {
    // fingerprint of the inputs (the audit seal names the artifacts by it):
    // BLAKE2b-128 of "GRIDgram", the text, the role list (all ones when
    // absent), the lexicons in call order and max_depth, lengths as u64
    Blake2b b;
    b.init(16);
    b.update("GRIDgram", 8);
    b.put_u64(len);
    b.update(grammar_text, len);
    if (role_keep) {
      const size_t n = std::strlen(role_keep);
      b.put_u64(n);
      b.update(role_keep, n);
    } else {
      b.put_u64(~0ull);
    }
    b.put_u64((uint64_t)n_lex);
    for (int i = 0; i < n_lex; ++i) {
      const size_t n = std::strlen(lex[i].category);
      b.put_u64(n);
      b.update(lex[i].category, n);
      b.put_u64((uint64_t)lex[i].n_words);
      for (int w = 0; w < lex[i].n_words; ++w) {
        const int64_t a = lex[i].offsets[w], z = lex[i].offsets[w + 1];
        b.put_u64((uint64_t)(z - a));
        b.update(lex[i].words + a, (size_t)(z - a));
      }
    }
    b.put_u64((uint64_t)h.max_depth);
    b.final(h.fingerprint);
  }
  *out = g;
  return GRID_OK;
}

extern "C" void grid_grammar_free(grid_grammar* g) { delete g; }

extern "C" int grid_grammar_info(const grid_grammar* g, int64_t out[8]) {
  if (!g || !out) return set_error(GRID_E_INVALID_ARG, "grid_grammar_info: bad arguments");
  const HostGrammar& h = g->h;
  out[0] = h.T1;
  out[1] = h.S;
  out[2] = h.NNT;
  out[3] = h.P;
  out[4] = h.Q;
  out[5] = h.C;
  out[6] = h.LN;
  out[7] = h.n_cat;
  return GRID_OK;
}

extern "C" int grid_grammar_lexicon_trie(const grid_grammar* g, int32_t* cstart, uint8_t* cbyte, int32_t* cnode,
                                        uint32_t* pcats, uint32_t* wcats, int64_t n_nodes) {
  if (!g || !cstart || !pcats || !wcats || n_nodes != g->h.LN || (n_nodes > 1 && (!cbyte || !cnode)))
    return set_error(GRID_E_INVALID_ARG, "grid_grammar_lexicon_trie: bad arguments (n_nodes must be the node count)");
  const HostGrammar& h = g->h;
  std::copy(h.lx_cstart.begin(), h.lx_cstart.end(), cstart);
  std::copy(h.lx_cbyte.begin(), h.lx_cbyte.end(), cbyte);
  std::copy(h.lx_cnode.begin(), h.lx_cnode.end(), cnode);
  std::copy(h.lx_pcats.begin(), h.lx_pcats.end(), pcats);
  std::copy(h.lx_wcats.begin(), h.lx_wcats.end(), wcats);
  return GRID_OK;
}

extern "C" int grid_load_vocab(const uint8_t* bytes, const int64_t* offsets, int32_t V, int32_t eos_id,
                               const int32_t* special_ids, int32_t n_special, grid_vocab** out) {
  if (!out || !offsets || V <= 0 || n_special < 0 || (n_special > 0 && !special_ids))
    return set_error(GRID_E_INVALID_ARG, "grid_load_vocab: bad arguments");
  *out = nullptr;
  if (eos_id < 0 || eos_id >= V) return set_error(GRID_E_VOCAB, "eos_id out of range");
  std::vector<char> excluded(V, 0);
  excluded[eos_id] = 1;
  for (int i = 0; i < n_special; ++i) {
    if (special_ids[i] < 0 || special_ids[i] >= V) return set_error(GRID_E_VOCAB, "special id out of range");
    excluded[special_ids[i]] = 1;
  }
  if (offsets[0] != 0) return set_error(GRID_E_VOCAB, "offsets[0] must be 0");
  for (int t = 0; t < V; ++t)
    if (offsets[t + 1] < offsets[t]) return set_error(GRID_E_VOCAB, "offsets must be non-decreasing");
  if (offsets[V] > (int64_t)1 << 30) return set_error(GRID_E_TOO_LARGE, "vocabulary bytes exceed 2^30");
  if (offsets[V] > 0 && !bytes) return set_error(GRID_E_INVALID_ARG, "bytes is NULL");
  // the non-excluded ids in spelling order (bytes compared unsigned, shorter
  // first on a common prefix, equal spellings by id), sorted in place on the
  // caller's buffer
  std::vector<int> ids;
  ids.reserve(V);
  for (int t = 0; t < V; ++t) {
    if (excluded[t]) continue;
    if (offsets[t + 1] == offsets[t])
      return set_error(GRID_E_VOCAB, "token " + std::to_string(t) + " has an empty spelling");
    ids.push_back(t);
  }
  auto spell_cmp = [&](int x, int y) {
    const int64_t nx = offsets[x + 1] - offsets[x], ny = offsets[y + 1] - offsets[y];
    const int c = std::memcmp(bytes + offsets[x], bytes + offsets[y], (size_t)std::min(nx, ny));
    return c != 0 ? c : (nx != ny ? (nx < ny ? -1 : 1) : 0);
  };
  {
    // sort on the first 8 bytes as a big-endian key (zero padded: where two
    // keys differ they order as the spellings do), the full comparison only
    // on equal keys
    std::vector<std::pair<uint64_t, int>> kv(ids.size());
    for (size_t i = 0; i < ids.size(); ++i) {
      const int t = ids[i];
      const int64_t n = std::min<int64_t>(8, offsets[t + 1] - offsets[t]);
      uint64_t key = 0;
      for (int64_t k = 0; k < 8; ++k) key = (key << 8) | (k < n ? bytes[offsets[t] + k] : 0u);
      kv[i] = {key, t};
    }
    std::sort(kv.begin(), kv.end(), [&](const std::pair<uint64_t, int>& x, const std::pair<uint64_t, int>& y) {
      if (x.first != y.first) return x.first < y.first;
      const int c = spell_cmp(x.second, y.second);
      return c != 0 ? c < 0 : x.second < y.second;
    });
    for (size_t i = 0; i < ids.size(); ++i) ids[i] = kv[i].second;
  }
  auto* v = new grid_vocab();
  HostVocab& h = v->h;
  h.V = V;
  h.eos = eos_id;
  h.spell_of_id.assign(V, -1);
  h.spell_off.reserve(ids.size() + 1);
  h.spell_off.push_back(0);
  for (size_t i = 0; i < ids.size(); ++i) {
    const int t = ids[i];
    if (i == 0 || spell_cmp(ids[i - 1], t) != 0) {
      h.spell_bytes.insert(h.spell_bytes.end(), bytes + offsets[t], bytes + offsets[t + 1]);
      h.spell_off.push_back((int32_t)h.spell_bytes.size());
    }
    h.spell_of_id[t] = (int32_t)h.spell_off.size() - 2;
  }
  h.NS = (int)h.spell_off.size() - 1;
  h.first_of_byte.assign(257, h.NS);
  for (int s = h.NS - 1; s >= 0; --s) h.first_of_byte[h.spell_bytes[h.spell_off[s]]] = s;
  for (int b = 255; b >= 0; --b)
    if (h.first_of_byte[b] > h.first_of_byte[b + 1]) h.first_of_byte[b] = h.first_of_byte[b + 1];
  int singles = 0;
  for (int s = 0; s < h.NS; ++s)
    if (h.spell_off[s + 1] - h.spell_off[s] == 1) ++singles;
  h.byte_complete = singles == 256;
  {
    // fingerprint of the inputs: BLAKE2b-128 of "GRIDvoca", V, eos, the
    // special ids in call order and every spelling, lengths as u64
    Blake2b b;
    b.init(16);
    b.update("GRIDvoca", 8);
    b.put_u64((uint64_t)V);
    b.put_u64((uint64_t)(int64_t)eos_id);
    b.put_u64((uint64_t)n_special);
    for (int i = 0; i < n_special; ++i) b.put_u64((uint64_t)(int64_t)special_ids[i]);
    for (int t = 0; t < V; ++t) {
      b.put_u64((uint64_t)(offsets[t + 1] - offsets[t]));
      b.update(bytes + offsets[t], (size_t)(offsets[t + 1] - offsets[t]));
    }
    b.final(h.fingerprint);
  }
  *out = v;
  return GRID_OK;
}

extern "C" void grid_vocab_free(grid_vocab* v) { delete v; }

extern "C" int grid_vocab_info(const grid_vocab* v, int64_t out[4]) {
  if (!v || !out) return set_error(GRID_E_INVALID_ARG, "grid_vocab_info: bad arguments");
  out[0] = v->h.V;
  out[1] = v->h.NS;
  out[2] = v->h.byte_complete ? 1 : 0;
  out[3] = (int64_t)v->h.spell_bytes.size();
  return GRID_OK;
}
