// Jump-forward forced spans (GRID Sec. 6.1, step 6 of the per-token hot
// path): while a row's mask admits exactly one token id, that token is
// forced; it is appended to the row's span and the row is advanced by it,
// without sampling.  Everything runs on the device: per span position one
// mask step, one kernel that finds each row's forced token (or stops the
// row), and one parser step whose no-op token (-1) leaves stopped rows alone.

#include <cstring>

#include "grid_state.cuh"

namespace grid {
namespace {

// aux layout (B ints each): tok, stop, adv_status, fail
__global__ void k_force_init(int32_t* __restrict__ span, int32_t* __restrict__ span_len, int32_t* __restrict__ aux,
                             int B, int max_span) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < B * max_span) span[i] = -1;
  if (i < B) {
    span_len[i] = 0;
    aux[i] = -1;
    aux[B + i] = 0;
    aux[2 * B + i] = GRID_ST_OK;
    aux[3 * B + i] = GRID_ST_OK;
  }
}

// One warp per row, after the mask step of span position `pos`: a row whose
// previous forced token could not be advanced, whose mask step reported a
// status, or whose mask does not hold exactly one bit stops; otherwise its
// one admitted id is appended and becomes the row's next token.
__global__ void k_force(const uint32_t* __restrict__ mask, int W, const int32_t* __restrict__ status,
                        int32_t* __restrict__ span, int32_t* __restrict__ span_len, int32_t* __restrict__ aux, int B,
                        int pos, int max_span) {
  const int b = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (b >= B) return;
  int32_t* tok = aux;
  int32_t* stop = aux + B;
  const int32_t* adv = aux + 2 * B;
  int32_t* fail = aux + 3 * B;
  const bool was_stopped = stop[b] != 0;
  __syncwarp();
  if (was_stopped) {
    if (lane == 0) tok[b] = -1;
    return;
  }
  if (pos > 0 && adv[b] != GRID_ST_OK) {
    if (lane == 0) {
      fail[b] = adv[b];
      stop[b] = 1;
      tok[b] = -1;
    }
    return;
  }
  if (status[b] != GRID_ST_OK) {
    if (lane == 0) {
      stop[b] = 1;
      tok[b] = -1;
    }
    return;
  }
  const uint32_t* row = mask + (size_t)b * W;
  int cnt = 0, first = -1;
  for (int w = lane; w < W; w += 32) {
    const uint32_t x = row[w];
    cnt += __popc(x);
    if (x && first < 0) first = 32 * w + __ffs(x) - 1;
  }
  cnt = __reduce_add_sync(0xffffffffu, cnt);
  // the lowest set bit over the lanes (each lane's first is its lowest)
  const int cand = first < 0 ? 0x7FFFFFFF : first;
  const int id = __reduce_min_sync(0xffffffffu, cand);
  if (lane == 0) {
    if (cnt == 1) {
      span[(size_t)b * max_span + pos] = id;
      span_len[b] = pos + 1;
      tok[b] = id;
    } else {
      stop[b] = 1;
      tok[b] = -1;
    }
  }
}

// After the final mask step: a row whose last forced token could not be
// advanced reports that advance's status.
__global__ void k_force_final(int32_t* __restrict__ d_status, const int32_t* __restrict__ aux, int B, int ran) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const int32_t* stop = aux + B;
  const int32_t* adv = aux + 2 * B;
  const int32_t* fail = aux + 3 * B;
  if (fail[b] != GRID_ST_OK)
    d_status[b] = fail[b];
  else if (ran && !stop[b] && adv[b] != GRID_ST_OK)
    d_status[b] = adv[b];
}

}  // namespace
}  // namespace grid

using namespace grid;

extern "C" int grid_forced_span(const grid_spec* s, grid_configs* c, int32_t max_span, uint32_t* d_mask,
                                int32_t* d_span, int32_t* d_span_len, int32_t* d_status, uint8_t* d_records,
                                void* stream) {
  if (!s || !c || !d_mask || (!d_span && max_span > 0) || !d_span_len || !d_status || max_span < 0 || max_span > 4096)
    return set_error(GRID_E_INVALID_ARG, "grid_forced_span: bad arguments");
  const bool audit = c->c.hs != nullptr;
  if (audit != (d_records != nullptr) && max_span > 0)
    return set_error(GRID_E_INVALID_ARG, audit ? "grid_forced_span: audit is on: pass the records of the forced tokens"
                                               : "grid_forced_span: records given but audit is not enabled");
  cudaStream_t st = (cudaStream_t)stream;
  const int B = c->B;
  const MaskScratch m{c->ctx, c->rng, c->sel, c->verd0, c->verd1, c->A2, c->vcbits,
                      c->surv, c->vsurv, c->cap, c->vcap, c->words_v};
  const int n = std::max(B * std::max(max_span, 1), B);
  k_force_init<<<(n + 255) / 256, 256, 0, st>>>(d_span, d_span_len, c->aux, B, max_span);
  GRID_CUDA(cudaGetLastError());
  int rc;
  for (int pos = 0; pos < max_span; ++pos) {
    if ((rc = launch_masks(s, c->c, m, B, d_mask, d_status, st, nullptr))) return rc;
    k_force<<<(B + 3) / 4, 128, 0, st>>>(d_mask, s->t.W, d_status, d_span, d_span_len, c->aux, B, pos, max_span);
    GRID_CUDA(cudaGetLastError());
    // every interior token of a span is audited (kind 1), at the configuration
    // its mask was computed at, before the advance
    if (audit && (rc = audit_append(s, c, d_mask, c->aux, 1u, d_records + (size_t)pos * 80, (long long)max_span * 80, st)))
      return rc;
    if ((rc = launch_advance(s, c->c, c->c, B, c->aux, 1, c->aux + 2 * B, 0, st))) return rc;
  }
  if ((rc = launch_masks(s, c->c, m, B, d_mask, d_status, st, nullptr))) return rc;
  k_force_final<<<(B + 127) / 128, 128, 0, st>>>(d_status, c->aux, B, max_span > 0 ? 1 : 0);
  GRID_CUDA(cudaGetLastError());
  return GRID_OK;
}

// ---------------------------------------------------------------------------
// Token-denominated reserve (GRID Sec. 5, Prop. 9, Termination; Sec. 6.1
// step 3): per row, the cheapest legal completion of the output plus EOS,
// counted in vocabulary tokens, so that a decoding loop whose remaining
// budget falls to that count plus a safety margin writes it instead of
// sampling.  The cost model is the paper's: every terminal of a completion
// is written as a fixed rendering (a blank and the terminal's lexeme, split
// greedily into vocabulary tokens), so a completion costs the sum of its
// terminals' rendering lengths; the pending lexeme is either ended as it
// stands (by the blank, or by the state's separator byte) or first extended,
// byte by byte, to the shortest lexeme of one terminal.  The cheapest
// terminal completion of a stack is found exactly over the LR(0) items:
// completing kernel item [A -> alpha . beta] of the top state costs beta's
// cheapest yield and leaves the stack with alpha popped and the goto on A
// pushed; every completion decomposes into such steps, and they only lower
// the stack (or keep its height, for |alpha| = 1), so one pass over the
// heights from the top down, with a fixpoint at each height, settles all
// costs.

namespace grid {
namespace {

constexpr uint32_t kInf = 0x3FFFFFFFu;
constexpr int kReserveEntries = 4096;  // search entries per row
constexpr int kMaxExt = 64;            // bytes of a pending-lexeme extension

struct REnt {
  int32_t level, state, cost, parent, item, next;
};

// The stack base[0:keep] ++ ovl[0:m].
struct VStack {
  const uint16_t* base;
  int keep;
  const uint16_t* ovl;
  int m;
  __device__ int at(int i) const { return i < keep ? base[i] : ovl[i - keep]; }
  __device__ int size() const { return keep + m; }
};

// The cheapest terminal completion of `vs` (in rendering tokens), or kInf;
// on success goal_e / goal_item name its last step.
__device__ uint32_t reserve_search(const Tables& t, const ReserveTables& rt, const VStack& vs, REnt* ent,
                                   int32_t* head, int& goal_e, int& goal_item, bool& overflow) {
  const int kmax = vs.size() - 1;
  goal_e = goal_item = -1;
  if (kmax >= t.D) {  // one level head per stack position: D of them
    overflow = true;
    return kInf;
  }
  for (int k = 0; k <= kmax; ++k) head[k] = -1;
  int cnt = 0;
  overflow = false;
  auto insert = [&](int level, int state, uint32_t cost, int parent, int item) -> bool {
    for (int e = head[level]; e >= 0; e = ent[e].next)
      if (ent[e].state == state) {
        if (cost >= (uint32_t)ent[e].cost) return false;
        ent[e].cost = (int32_t)cost;
        ent[e].parent = parent;
        ent[e].item = item;
        return true;
      }
    if (cnt >= rt.E) {
      overflow = true;
      return false;
    }
    ent[cnt] = REnt{level, state, (int32_t)cost, parent, item, head[level]};
    head[level] = cnt++;
    return true;
  };
  insert(kmax, vs.at(kmax), 0u, -1, -1);
  uint32_t best = kInf;
  goal_e = goal_item = -1;
  for (int k = kmax; k >= 0; --k) {
    // steps that keep the height (|alpha| = 1), to a fixpoint; the goal
    for (int round = 0; round <= t.S; ++round) {
      bool changed = false;
      for (int e = head[k]; e >= 0; e = ent[e].next) {
        const int s = ent[e].state;
        const uint32_t c0 = (uint32_t)ent[e].cost;
        for (int i = rt.item_off[s]; i < rt.item_off[s + 1]; ++i) {
          const uint32_t ic = rt.item_cost[i];
          if (ic >= kInf) continue;
          const int p = rt.item_p[i], d = rt.item_d[i];
          const uint32_t c = c0 + ic;
          if (p == 0) {  // S' -> . start at height 0, S' -> start . at height 1: the sentence is complete
            if (((d == 0 && k == 0) || (d == 1 && k == 1)) && c < best) {
              best = c;
              goal_e = e;
              goal_item = i;
            }
            continue;
          }
          if (d != 1 || k < 1) continue;
          const int g = t.go[vs.at(k - 1) * t.NNT + t.plhs[p]];
          if (g >= t.S) continue;
          if (insert(k, g, c, e, i)) changed = true;
        }
      }
      if (!changed) break;
    }
    // steps that lower the stack (|alpha| >= 2)
    for (int e = head[k]; e >= 0; e = ent[e].next) {
      const int s = ent[e].state;
      const uint32_t c0 = (uint32_t)ent[e].cost;
      for (int i = rt.item_off[s]; i < rt.item_off[s + 1]; ++i) {
        const int p = rt.item_p[i], d = rt.item_d[i];
        const uint32_t ic = rt.item_cost[i];
        if (p == 0 || d < 2 || d > k || ic >= kInf) continue;
        const int g = t.go[vs.at(k - d) * t.NNT + t.plhs[p]];
        if (g >= t.S) continue;
        insert(k - d + 1, g, c0 + ic, e, i);
      }
    }
  }
  return best;
}

// The tokens rendering terminal x (one warp lane writes).
__device__ void put_terminal(const ReserveTables& rt, int x, int32_t* out, int cap, int& n) {
  for (int j = rt.rend_off[x]; j < rt.rend_off[x + 1]; ++j) {
    if (n < cap) out[n] = rt.rend_tok[j];
    ++n;
  }
}

// One warp per row; lane 0 evaluates the ways to end the pending lexeme
// (option 0: as it stands; option 1 + tau: extended to tau's shortest
// lexeme) and keeps the cheapest, then writes its tokens.
__global__ void k_reserve(Tables t, ReserveTables rt, DevConfigs c, int32_t* __restrict__ scratch,
                          size_t scratch_ints, int32_t* __restrict__ d_cost, int32_t* __restrict__ d_tokens, int cap,
                          int32_t* __restrict__ d_status, const int32_t* __restrict__ d_budget, int safety,
                          int32_t* __restrict__ d_fire, int B) {
  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ Tables ts;
  stage_tables(t, ts, smem);
  const int b = blockIdx.x;
  if (b >= B || threadIdx.x != 0) return;
  REnt* ent = reinterpret_cast<REnt*>(scratch + (size_t)b * scratch_ints);
  int32_t* head = scratch + (size_t)b * scratch_ints + (size_t)rt.E * (sizeof(REnt) / 4);
  int32_t* out = d_tokens + (size_t)b * cap;
  const int depth = c.depth[b], q = c.q[b], lx = c.lx[b];
  const uint16_t* base = c.stack + (size_t)b * t.D;
  int status = GRID_ST_OK, n = 0;
  uint32_t total_best = kInf;
  if (c.flags[b] & 1) {
    status = GRID_ST_COMPLETE;
  } else {
    const int mc = max_chain_of(t);
    const uint32_t pc0 = lx >= 0 ? t.lx_pcats[lx] : 0u, wc0 = lx >= 0 ? t.lx_wcats[lx] : 0u;
    const Bits4 live0 = q == kStart ? Bits4::zero() : live_prime(ts, q, pc0);
    uint16_t lo[kMaxOvl], ls[kMaxOvl];
    uint8_t y[kMaxExt];
    int best_opt = -1;
    bool any_overflow = false;
    // builds option `opt` into (vs, y, ylen, sep); false when it does not apply
    auto build = [&](int opt, VStack& vs, int& ylen, int& sep) -> bool {
      ylen = 0;
      sep = ' ';
      if (q == kStart) {
        if (opt != 0) return false;
        vs = VStack{base, depth, lo, 0};
        return true;
      }
      int q2 = q, lx2 = lx;
      uint32_t pc = pc0, wc = wc0;
      if (opt > 0) {  // extend the lexeme to terminal tau's shortest lexeme
        const int tau = opt - 1;
        if (tau >= t.n_term || t.ign.has(tau) || !live0.has(tau)) return false;
        int cat = -1;
        for (int k = 0; k < t.n_cat; ++k)
          if (t.cat_term[k] == tau) cat = k;
        int len;
        if (cat >= 0) {
          if (lx < 0) return false;
          len = rt.lx_wdist[(size_t)lx * rt.NC + cat];
          if (len == 0xFFFF) return false;
        } else {
          len = rt.dfa_tdist[(size_t)q * t.T1 + tau];
          if (len == 0xFF) return false;
        }
        if (len == 0 || len > kMaxExt) return false;  // len 0: the lexeme as it stands (option 0)
        for (int i = 0; i < len; ++i) {
          const int by = cat >= 0 ? rt.lx_wbyte[(size_t)lx2 * rt.NC + cat] : rt.dfa_tbyte[(size_t)q2 * t.T1 + tau];
          const int nq = ts.next[q2 * ts.C + ts.byte_class[by]];
          if (nq == kDead) return false;
          q2 = nq;
          lx2 = lex_step(ts, lx2, by, pc, wc);
          if (cat >= 0 && lx2 < 0) return false;
          y[ylen++] = (uint8_t)by;
        }
      } else if (opt != 0) {
        return false;
      }
      sep = rt.sep_byte[q2];
      if (sep < 0) return false;
      Walker w;
      walker_init(w, LArr{lo, 1}, LArr{ls, 1}, kMaxOvl, base, depth, nullptr, 0, q2, lx2, pc, wc, nullptr, nullptr);
      if (emit(ts, w, mc) <= 0) return false;
      vs = VStack{base, w.keep, lo, w.m};
      return true;
    };
    auto total_of = [&](uint32_t C, int ylen, int sep) -> uint32_t {
      if (C >= kInf) return kInf;
      // the blank that ends the lexeme comes with the first rendering; another
      // separator is a token of its own, needed only before a rendering
      return (uint32_t)ylen + ((C > 0 && sep != ' ') ? 1u : 0u) + C + 1u;
    };
    for (int opt = 0; opt <= t.n_term; ++opt) {
      VStack vs;
      int ylen, sep;
      if (!build(opt, vs, ylen, sep)) continue;
      bool ok = true;
      for (int i = 0; i < ylen && ok; ++i) ok = rt.byte_tok[y[i]] >= 0;
      if (!ok) continue;
      int ge, gi;
      bool of;
      const uint32_t C = reserve_search(ts, rt, vs, ent, head, ge, gi, of);
      any_overflow |= of;
      if (C > 0 && C < kInf && sep != ' ' && rt.byte_tok[sep] < 0) continue;
      const uint32_t tot = total_of(C, ylen, sep);
      if (tot < total_best) {
        total_best = tot;
        best_opt = opt;
      }
    }
    if (best_opt < 0) {
      status = any_overflow ? GRID_ST_BOUND : GRID_ST_NONVIABLE;
    } else {
      // the chosen option again, and its tokens
      VStack vs;
      int ylen, sep, ge, gi;
      bool of;
      build(best_opt, vs, ylen, sep);
      const uint32_t C = reserve_search(ts, rt, vs, ent, head, ge, gi, of);
      for (int i = 0; i < ylen; ++i) {
        if (n < cap) out[n] = rt.byte_tok[y[i]];
        ++n;
      }
      if (C > 0 && sep != ' ') {
        if (n < cap) out[n] = rt.byte_tok[sep];
        ++n;
      }
      // the steps in order: reverse the parent chain from the goal entry
      int prev = -1, cur = ge;
      while (cur >= 0) {
        const int nx = ent[cur].parent;
        ent[cur].parent = prev;
        prev = cur;
        cur = nx;
      }
      auto put_item = [&](int i) {
        const int p = rt.item_p[i], d = rt.item_d[i];
        for (int j = rt.prod_off[p] + d; j < rt.prod_off[p + 1]; ++j) {
          const int X = rt.prod_rhs[j];
          if (X < t.T1) {
            put_terminal(rt, X, out, cap, n);
          } else {
            for (int k = rt.ny_off[X - t.T1]; k < rt.ny_off[X - t.T1 + 1]; ++k) put_terminal(rt, rt.ny[k], out, cap, n);
          }
        }
      };
      for (int e = prev; e >= 0; e = ent[e].parent)  // prev: the start entry, which has no step
        if (ent[e].item >= 0) put_item(ent[e].item);
      put_item(gi);
      if (n < cap) out[n] = t.eos;
      ++n;
      if (n > cap) status = GRID_ST_BOUND;
    }
  }
  for (int i = n; i < cap; ++i) out[i] = -1;
  d_cost[b] = status == GRID_ST_OK || (status == GRID_ST_BOUND && total_best < kInf) ? (int32_t)total_best : -1;
  if (status == GRID_ST_COMPLETE) d_cost[b] = 0;
  d_status[b] = status;
  if (d_fire) d_fire[b] = (status == GRID_ST_OK && d_budget && d_budget[b] <= (int)total_best + safety) ? 1 : 0;
}

}  // namespace

size_t reserve_scratch_bytes(const grid_spec* s) {
  return (size_t)kReserveEntries * sizeof(REnt) + (size_t)s->t.D * 4;
}

int build_reserve_tables(grid_spec* s) {
  const HostGrammar& h = s->g->h;
  const HostVocab& hv = s->v->h;
  ReserveTables& rt = s->rt;
  Arena& a = s->mem;
  const int T1 = h.T1, NNT = h.NNT, P = h.P, NS = hv.NS;
  auto is_ign = [&](int t) { return (h.ignored[t >> 5] >> (t & 31)) & 1u; };
  // the smallest id of every distinct spelling; exact lookup of a byte string
  std::vector<int32_t> id_of(std::max(1, NS), -1);
  for (int id = hv.V - 1; id >= 0; --id)
    if (hv.spell_of_id[id] >= 0) id_of[hv.spell_of_id[id]] = id;
  int maxlen = 1;
  for (int sp = 0; sp < NS; ++sp) maxlen = std::max(maxlen, hv.spell_off[sp + 1] - hv.spell_off[sp]);
  auto find = [&](const uint8_t* p, int n) {
    int lo = 0, hi = NS;
    while (lo < hi) {  // first spelling not below p[0:n] (bytes unsigned, shorter first)
      const int mid = (lo + hi) / 2;
      const int off = hv.spell_off[mid], len = hv.spell_off[mid + 1] - off;
      int cmp = std::memcmp(hv.spell_bytes.data() + off, p, (size_t)std::min(len, n));
      if (cmp == 0) cmp = len < n ? -1 : (len > n ? 1 : 0);
      if (cmp < 0)
        lo = mid + 1;
      else
        hi = mid;
    }
    if (lo < NS) {
      const int off = hv.spell_off[lo], len = hv.spell_off[lo + 1] - off;
      if (len == n && std::memcmp(hv.spell_bytes.data() + off, p, (size_t)n) == 0) return lo;
    }
    return -1;
  };
  std::vector<int32_t> byte_tok(256, -1);
  for (int b = 0; b < 256; ++b) {
    const uint8_t x = (uint8_t)b;
    const int sp = find(&x, 1);
    if (sp >= 0) byte_tok[b] = id_of[sp];
  }
  // renderings: " " + lexeme, split greedily (longest spelling first)
  std::vector<int32_t> rend_off(1, 0), rend_tok;
  std::vector<uint32_t> tcost(T1, kInf);
  for (int tau = 0; tau < T1; ++tau) {
    if (tau < h.n_term && !is_ign(tau) && !h.render_lex[tau].empty()) {
      const std::string str = " " + h.render_lex[tau];
      const uint8_t* p = reinterpret_cast<const uint8_t*>(str.data());
      const int n = (int)str.size();
      std::vector<int32_t> toks;
      bool ok = true;
      for (int i = 0; i < n && ok;) {
        ok = false;
        for (int L = std::min(maxlen, n - i); L >= 1; --L) {
          const int sp = find(p + i, L);
          if (sp >= 0) {
            toks.push_back(id_of[sp]);
            i += L;
            ok = true;
            break;
          }
        }
      }
      if (ok) {
        tcost[tau] = (uint32_t)toks.size();
        rend_tok.insert(rend_tok.end(), toks.begin(), toks.end());
      }
    }
    rend_off.push_back((int32_t)rend_tok.size());
  }
  // cheapest yield of every nonterminal, settled in order of cost (a
  // production is used only once all its nonterminals are settled, so every
  // yield is finite and well founded)
  std::vector<uint32_t> mcost(NNT, kInf);
  std::vector<int> bestp(NNT, -1), order;
  std::vector<char> settled(NNT, 0);
  for (;;) {
    uint32_t best = kInf;
    int bA = -1, bP = -1;
    for (int p = 0; p < P; ++p) {
      const int A = h.plhs[p];
      if (settled[A]) continue;
      uint32_t sum = 0;
      bool ok = true;
      for (int j = h.prod_off[p]; j < h.prod_off[p + 1] && ok; ++j) {
        const int X = h.prod_rhs[j];
        const uint32_t cx = X < T1 ? tcost[X] : (settled[X - T1] ? mcost[X - T1] : kInf);
        if (cx >= kInf) ok = false;
        sum = std::min<uint32_t>(kInf, sum + cx);
      }
      if (ok && sum < best) {
        best = sum;
        bA = A;
        bP = p;
      }
    }
    if (bA < 0) break;
    settled[bA] = 1;
    mcost[bA] = best;
    bestp[bA] = bP;
    order.push_back(bA);
  }
  std::vector<std::vector<int32_t>> yield(NNT);
  size_t ytotal = 0;
  for (int A : order) {
    const int p = bestp[A];
    for (int j = h.prod_off[p]; j < h.prod_off[p + 1]; ++j) {
      const int X = h.prod_rhs[j];
      if (X < T1)
        yield[A].push_back(X);
      else
        yield[A].insert(yield[A].end(), yield[X - T1].begin(), yield[X - T1].end());
    }
    ytotal += yield[A].size();
    if (ytotal > (1u << 24)) return set_error(GRID_E_TOO_LARGE, "grid_specialize: cheapest yields too long");
  }
  std::vector<int32_t> ny_off(1, 0), ny;
  for (int A = 0; A < NNT; ++A) {
    ny.insert(ny.end(), yield[A].begin(), yield[A].end());
    ny_off.push_back((int32_t)ny.size());
  }
  std::vector<uint32_t> item_cost(h.kitem_p.size(), kInf);
  for (size_t i = 0; i < h.kitem_p.size(); ++i) {
    const int p = h.kitem_p[i], d = h.kitem_d[i];
    uint32_t sum = 0;
    for (int j = h.prod_off[p] + d; j < h.prod_off[p + 1]; ++j) {
      const int X = h.prod_rhs[j];
      sum = std::min<uint32_t>(kInf, sum + (X < T1 ? tcost[X] : mcost[X - T1]));
    }
    item_cost[i] = sum;
  }
  int rc;
  if ((rc = a.upload(h.kitem_off, &rt.item_off)) || (rc = a.upload(h.kitem_p, &rt.item_p)) ||
      (rc = a.upload(h.kitem_d, &rt.item_d)) || (rc = a.upload(item_cost, &rt.item_cost)) ||
      (rc = a.upload(h.prod_off, &rt.prod_off)) || (rc = a.upload(h.prod_rhs, &rt.prod_rhs)) ||
      (rc = a.upload(ny_off, &rt.ny_off)) || (rc = a.upload(ny, &rt.ny)) || (rc = a.upload(rend_off, &rt.rend_off)) ||
      (rc = a.upload(rend_tok, &rt.rend_tok)) || (rc = a.upload(h.lx_wdist, &rt.lx_wdist)) ||
      (rc = a.upload(h.lx_wbyte, &rt.lx_wbyte)) || (rc = a.upload(h.dfa_tdist, &rt.dfa_tdist)) ||
      (rc = a.upload(h.dfa_tbyte, &rt.dfa_tbyte)) || (rc = a.upload(h.sep_byte, &rt.sep_byte)) ||
      (rc = a.upload(byte_tok, &rt.byte_tok)))
    return rc;
  rt.NC = std::max(1, h.n_cat);
  rt.E = kReserveEntries;
  rt.ok = 1;
  return GRID_OK;
}

}  // namespace grid

extern "C" int grid_reserve(const grid_spec* s, const grid_configs* c, int32_t* d_cost, int32_t* d_tokens, int32_t cap,
                            int32_t* d_status, const int32_t* d_budget, int32_t safety, int32_t* d_fire, void* stream) {
  if (!s || !c || !d_cost || !d_tokens || cap <= 0 || !d_status || (d_budget && !d_fire))
    return set_error(GRID_E_INVALID_ARG, "grid_reserve: bad arguments");
  if (!s->rt.ok) return set_error(GRID_E_INVALID_ARG, "grid_reserve: the spec has no reserve tables");
  const size_t ints = reserve_scratch_bytes(s) / 4;
  GRID_CUDA(cudaFuncSetAttribute(k_reserve, cudaFuncAttributeMaxDynamicSharedMemorySize, s->t.blob_bytes));
  k_reserve<<<c->B, 32, s->t.blob_bytes, (cudaStream_t)stream>>>(s->t, s->rt, c->c, c->rscratch, ints, d_cost,
                                                                d_tokens, cap, d_status, d_budget, safety, d_fire,
                                                                c->B);
  GRID_CUDA(cudaGetLastError());
  return GRID_OK;
}
