// Device-side data structures and per-lane routines of the mask path.
//
// A configuration kappa = (sigma, rho) (GRID Def. 1) is, on the device, the
// row's stack of LALR(1) states (uint16, bottom first) plus the scan state of
// the pending lexeme: the lexer DFA state q and the node lx of the identifier
// trie (-1 once the lexeme left every lexicon word).  While a token is tried,
// the row stack is never written: a lane works on the virtual stack
// base[0:keep] ++ ovl[0:m] (copy-on-write top of stack), and a simulated
// reduce chain additionally pushes into scr[0:ns].
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

#include "grid_internal.h"

namespace grid {

constexpr int kMaxOvl = 48;  // per-token overlay / scratch entries per lane

// CI class codes (Sec. 4.2).  Codes below kClsFirstCode are class ids
// ((kind * Q + q) << n_cat | cats): kind 0 = the verdict is "the live set of
// (q, cats) meets A u I" (token ends inside one lexeme), kind 1 = "the
// candidate set of (q, cats) meets A u I" (one boundary, then ignored bytes).
constexpr uint16_t kClsFirstCode = 0xFFFB;  // class ids are below this value
constexpr uint16_t kClsVC = 0xFFFB;   // context-dependent, decided by its verdict class (event record)
constexpr uint16_t kClsNA = 0xFFFC;   // spelling does not continue this lexer state
constexpr uint16_t kClsAcc = 0xFFFD;  // viable for every allowed set
constexpr uint16_t kClsRej = 0xFFFE;  // viable for no allowed set
constexpr uint16_t kClsCD = 0xFFFF;   // context-dependent, too many events: walked byte by byte

// Event record of a context-dependent spelling (GRID Sec. 4.2, verdict-
// equivalence grouping): rec[0] = number of stack-dependent emissions n,
// rec[1] = the final test (a live class id, or kClsAcc when the trailing
// lexeme is live for an ignored terminal), rec[2 .. 2+n) = the candidate
// classes of the emissions in order.  Spellings with equal records have equal
// verdicts at every stack; each distinct record is a verdict class.
constexpr int kRecLen = 16;
constexpr int kMaxEv = kRecLen - 2;

// A set of at most 128 terminals held in four registers.  Word access goes
// through selects, never through a runtime-indexed array (which would live
// in local memory).
struct Bits4 {
  uint32_t x, y, z, w;
  __host__ __device__ __forceinline__ static Bits4 zero() { return Bits4{0u, 0u, 0u, 0u}; }
  __device__ __forceinline__ static Bits4 load(const uint32_t* p) { return Bits4{p[0], p[1], p[2], p[3]}; }
  __device__ __forceinline__ uint32_t word(int i) const { return i == 0 ? x : (i == 1 ? y : (i == 2 ? z : w)); }
  __device__ __forceinline__ bool has(int t) const { return (word(t >> 5) >> (t & 31)) & 1u; }
  __device__ __forceinline__ void set(int t) {
    const uint32_t b = 1u << (t & 31);
    const int i = t >> 5;
    x |= i == 0 ? b : 0u;
    y |= i == 1 ? b : 0u;
    z |= i == 2 ? b : 0u;
    w |= i == 3 ? b : 0u;
  }
  __device__ __forceinline__ bool any() const { return (x | y | z | w) != 0u; }
  __device__ __forceinline__ int count() const { return __popc(x) + __popc(y) + __popc(z) + __popc(w); }
  __device__ __forceinline__ Bits4 operator&(const Bits4& o) const { return Bits4{x & o.x, y & o.y, z & o.z, w & o.w}; }
  __device__ __forceinline__ Bits4 operator|(const Bits4& o) const { return Bits4{x | o.x, y | o.y, z | o.z, w | o.w}; }
  __device__ __forceinline__ Bits4 andnot(const Bits4& o) const {
    return Bits4{x & ~o.x, y & ~o.y, z & ~o.z, w & ~o.w};
  }
  __device__ __forceinline__ int lowest() const {
    return x ? __ffs(x) - 1 : (y ? 31 + __ffs(y) : (z ? 63 + __ffs(z) : (w ? 95 + __ffs(w) : -1)));
  }
  __device__ __forceinline__ void clear_lowest() {
    if (x)
      x &= x - 1u;
    else if (y)
      y &= y - 1u;
    else if (z)
      z &= z - 1u;
    else
      w &= w - 1u;
  }
};

struct Tables {
  int n_term, T1, S, NNT, P, Q, C, n_cat, LN;
  int NS, V, eos, W, D;
  int Vp;     // V rounded up to a multiple of 32: the row length of the id-indexed tables
  Bits4 ign;  // ignored terminals (the set I)
  Bits4 cm;   // category terminals
  int cat_term[32];
  // staged block: these eight arrays live contiguously in `blob`
  const uint8_t* blob;
  int blob_bytes;  // 0 = too large to stage in shared memory
  const uint8_t* byte_class;
  const uint16_t* next;
  const uint32_t* acc;
  const uint32_t* live;
  const int16_t* action;
  const uint16_t* go;
  const uint8_t* plen;
  const uint16_t* plhs;
  const uint32_t* shift_mask;  // S * 4: terminals whose action is SHIFT
  const uint32_t* red_off;     // S + 1: reduce groups of state s are red_off[s] .. red_off[s+1]
  const uint16_t* red_p;       // each reduce group's production as plen << 10 | lhs
  const uint32_t* red_mask;    // 4 per reduce group: its lookahead terminals
  // identifier trie
  const int32_t* lx_cstart;
  const uint8_t* lx_cbyte;
  const int32_t* lx_cnode;
  const uint32_t* lx_pcats;
  const uint32_t* lx_wcats;
  // open-addressing hash of the identifier-trie edges: key = node * 256 + byte,
  // entry = {key, child, child's prefix categories, child's word categories}
  const uint4* lx_hash;
  uint32_t lx_hmask;
  int lx_hshift;
  uint32_t root_pc, root_wc;
  // vocabulary trie
  const int32_t* spell_off;
  const uint8_t* spell_bytes;
  const uint4* spell16;  // first 16 bytes of each spelling, zero padded (one load per walk)
  const int32_t* spell_of_id;
  const int32_t* id_of_spell;  // NS: the smallest id with each spelling
  const int32_t* next_alias;   // Vp: the next larger id with the same spelling, -1 after the last
  const int32_t* first_of_byte;
  const uint8_t* first_byte_by_id;
  const uint32_t* id_valid;    // W words: bit set for the ids with a spelling (not EOS, special or padding)
  const uint32_t* killw;       // Q * W: bit j of word (q, wi): id 32 wi + j's first byte ends a lexeme at q
  // CI tables (one per lexer state in the precomputed set; table 0 = start state)
  int ci_on;
  int n_tbl;
  int ncls;
  int nselw;
  const int16_t* tbl_of_q;
  const int32_t* tbl_q;
  const uint16_t* cls_by_id;  // n_tbl * V
  const int32_t* cd_off;      // n_tbl + 1
  const int32_t* cd_list;     // ascending spelling indices per table
  const uint16_t* cd_key;     // per cd_list entry: class of its first stack-dependent emission
  // verdict classes: table k owns records vc_off[k] .. vc_off[k+1] of vc_rec
  const int32_t* vc_off;
  const uint16_t* vc_rec;     // kRecLen per verdict class
  const uint16_t* vc_first;   // class id of each verdict class's first event
  const uint32_t* vc_by_id;   // n_tbl * V: verdict class (within its table) of kClsVC spellings, or NULL
                              // when the class codes carry it (vc_inline)
  int vc_inline;              // 1: a verdict-class id's code is ncls + kPackCodes + its class index
  const uint32_t* cls_sets;   // ncls * 4: terminal set of every class id
  const uint32_t* cls_mask;   // T1 * nselw: bit c of row tau = tau is in class c's set
  const uint32_t* acc_sym;    // S: the symbol entering each state (audit node hash)
};

// Work counters of a walk, kept in the lane's registers when the walk is
// measured and absent (a null pointer the compiler sees) otherwise:
// [0] lexer steps (trie node visits), [1] ACTION lookups (one per reduce
// chain step, for a terminal or a set of terminals), [2] GOTO lookups,
// [3] verdict-class events evaluated.
__device__ __forceinline__ void count_work(uint32_t* ctr, int k) {
  if (ctr) ++ctr[k];
}

// Membership test in a 4-word set stored in memory.
__device__ __forceinline__ bool bit4(const uint32_t* m, int t) { return (m[t >> 5] >> (t & 31)) & 1u; }

// Copy the staged block into shared memory and publish one block-wide copy of
// the table descriptor, rebased onto it, in shared memory (`ts`).  Every thread
// of the block must call this.
// Copy the staged block into shared memory with one bulk asynchronous copy
// (the block is 16-byte aligned and a multiple of 16 bytes), completion
// tracked by an mbarrier.  The wait is bounded; if it gives up, the block is
// copied again with plain loads (same bytes), so the result never depends on
// the bulk copy finishing.
__device__ __forceinline__ void stage_tables(const Tables& t, Tables& ts, uint8_t* smem) {
  __shared__ __align__(8) uint64_t s_bar;
  __shared__ int s_late;
  if (t.blob_bytes) {
    const uint32_t bar = (uint32_t)__cvta_generic_to_shared(&s_bar);
    if (threadIdx.x == 0) {
      s_late = 0;
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(bar) : "memory");
      asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
      asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(t.blob_bytes)
                   : "memory");
      asm volatile(
          "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
              (uint32_t)__cvta_generic_to_shared(smem)),
          "l"(t.blob), "r"(t.blob_bytes), "r"(bar)
          : "memory");
    }
    __syncthreads();
    uint32_t done = 0;
    for (int it = 0; it < (1 << 20) && !done; ++it)
      asm volatile(
          "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0;\n selp.u32 %0, 1, 0, p;\n}"
          : "=r"(done)
          : "r"(bar)
          : "memory");
    if (!done) s_late = 1;
    __syncthreads();
    if (s_late) {
      const uint4* src = reinterpret_cast<const uint4*>(t.blob);
      uint4* dst = reinterpret_cast<uint4*>(smem);
      for (int i = threadIdx.x; i < (t.blob_bytes >> 4); i += blockDim.x) dst[i] = src[i];
    }
  }
  if (threadIdx.x == 0) {
    ts = t;
    if (t.blob_bytes) {
      auto rebase = [&](const void* p) { return smem + ((const uint8_t*)p - t.blob); };
      ts.byte_class = rebase(t.byte_class);
      ts.next = reinterpret_cast<const uint16_t*>(rebase(t.next));
      ts.acc = reinterpret_cast<const uint32_t*>(rebase(t.acc));
      ts.live = reinterpret_cast<const uint32_t*>(rebase(t.live));
      ts.action = reinterpret_cast<const int16_t*>(rebase(t.action));
      ts.go = reinterpret_cast<const uint16_t*>(rebase(t.go));
      ts.plen = rebase(t.plen);
      ts.plhs = reinterpret_cast<const uint16_t*>(rebase(t.plhs));
      ts.shift_mask = reinterpret_cast<const uint32_t*>(rebase(t.shift_mask));
      ts.red_off = reinterpret_cast<const uint32_t*>(rebase(t.red_off));
      ts.red_p = reinterpret_cast<const uint16_t*>(rebase(t.red_p));
      ts.red_mask = reinterpret_cast<const uint32_t*>(rebase(t.red_mask));
    }
  }
  __syncthreads();
}

// Programmatic dependent launch: the step's kernels are launched so that each
// may start while its predecessor in the stream finishes; everything a kernel
// does before this wait touches only the spec's read-only tables.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

constexpr uint32_t kHashEmpty = 0xFFFFFFFFu;

// Child of identifier-trie node lx on byte b (-1 if none), with the child's
// prefix / word category bits (0 when there is no child).  One 16-byte load
// per probe; the table is at most half full, so probing ends at an empty slot.
__device__ __forceinline__ int lex_step(const Tables& t, int lx, int b, uint32_t& pc, uint32_t& wc) {
  pc = 0u;
  wc = 0u;
  if (lx < 0) return -1;
  const uint32_t key = (uint32_t)lx * 256u + (uint32_t)b;
  uint32_t h = (key * 0x9E3779B1u) >> t.lx_hshift;
  for (uint32_t i = 0; i <= t.lx_hmask; ++i) {
    const uint4 e = __ldg(&t.lx_hash[h]);
    if (e.x == key) {
      pc = e.z;
      wc = e.w;
      return (int)e.y;
    }
    if (e.x == kHashEmpty) return -1;
    h = (h + 1u) & t.lx_hmask;
  }
  return -1;
}

// Terminal set of DFA state q filtered by the lexicon: non-category terminals
// pass, category terminal c passes iff bit c of `cats` is set.
__device__ __forceinline__ Bits4 lex_filter(const Tables& t, const uint32_t* src, int q, uint32_t cats) {
  const Bits4 v = Bits4::load(src + q * 4);
  Bits4 out = v.andnot(t.cm);
  while (cats) {
    const int c = __ffs(cats) - 1;
    cats &= cats - 1;
    const int term = t.cat_term[c];
    if (v.has(term)) out.set(term);
  }
  return out;
}

// live'(q, r): terminals live at q, category terminals only while r is a
// prefix of one of their words (pc = prefix category bits of r's trie node).
__device__ __forceinline__ Bits4 live_prime(const Tables& t, int q, uint32_t pc) { return lex_filter(t, t.live, q, pc); }

// Emission candidates of r: terminals accepting at q, category terminals only
// if r is one of their words (wc = word category bits of r's trie node).
__device__ __forceinline__ Bits4 cands(const Tables& t, int q, uint32_t wc) { return lex_filter(t, t.acc, q, wc); }

__device__ __forceinline__ int max_chain_of(const Tables& t) { return 2 * t.D + 256; }

// A lane's small array: element i lives at p[i * s].  Walk lanes keep their
// overlays in shared memory interleaved across the warp (s = 32, no bank
// conflicts); single-thread users keep them in local arrays (s = 1).
struct LArr {
  uint16_t* p;
  int s;
  __device__ __forceinline__ uint16_t& operator[](int i) const { return p[i * s]; }
};

// Reduce chain of terminal tau on the virtual stack base[0:keep] ++ ovl[0:m]
// (Sec. 3.2, "allowed terminals by simulation").  Returns the ACTION code that
// ends it (> 0: shift to code-1, or kAccept), 0 on error, -1 on a bound.  On
// shift/accept, (keep_o, m_o, scr[0:ns]) is the stack under the pushed state.
template <typename OV>
__device__ __forceinline__ int simulate(const Tables& t, const uint16_t* base, int keep, OV ovl, int m, int tau,
                                        LArr scr, int cap, int& keep_o, int& m_o, int& ns, int max_chain,
                                        uint32_t* ctr = nullptr) {
  int k = keep, mm = m;
  ns = 0;
  int top = mm ? ovl[mm - 1] : base[k - 1];
  for (int it = 0; it < max_chain; ++it) {
    if (top >= t.S) return 0;
    count_work(ctr, 1);
    const int a = t.action[top * t.T1 + tau];
    if (a == 0) return 0;
    if (a > 0) {
      keep_o = k;
      m_o = mm;
      return a;
    }
    const int code = -a - 1;  // plen << 10 | lhs
    int n = code >> 10;
    int x = min(n, ns);
    ns -= x;
    n -= x;
    x = min(n, mm);
    mm -= x;
    n -= x;
    k -= n;
    if (k < 1) return 0;
    const int top2 = ns ? scr[ns - 1] : (mm ? ovl[mm - 1] : base[k - 1]);
    if (top2 >= t.S) return 0;
    if (ns >= cap) return -1;
    count_work(ctr, 2);
    top = t.go[top2 * t.NNT + (code & 1023)];
    scr[ns++] = (uint16_t)top;
  }
  return -1;
}

// The terminals of G whose reduce chains on the virtual stack reach SHIFT:
// simulate() for a set of terminals at once.  Terminals travel together while
// they take the same action; where the remaining ones reduce by different
// productions, the group of the first production listed for the state goes
// on and the others are simulated again from the start in a later round
// (they follow the same path up to that state).  After kSetRounds rounds the
// rest is simulated one terminal at a time.  `bound` is set on a bound.
constexpr int kSetRounds = 8;

template <typename OV>
__device__ __forceinline__ Bits4 simulate_set(const Tables& t, const uint16_t* base, int keep, OV ovl, int m, Bits4 G,
                                              LArr scr, int cap, int max_chain, bool& bound,
                                              uint32_t* ctr = nullptr) {
  Bits4 res = Bits4::zero();
  Bits4 todo = G;
  for (int round = 0; round < kSetRounds && todo.any(); ++round) {
    Bits4 g = todo;
    todo = Bits4::zero();
    int k = keep, mm = m, ns = 0;
    int it = 0;
    int top = mm ? ovl[mm - 1] : base[k - 1];
    for (; it < max_chain && g.any(); ++it) {
      if (top >= t.S) break;
      count_work(ctr, 1);
      const Bits4 sh = Bits4::load(t.shift_mask + top * 4);
      res = res | (g & sh);
      g = g.andnot(sh);
      if (!g.any()) break;
      int p = -1;
      Bits4 gp = Bits4::zero();
      for (uint32_t e = t.red_off[top]; e < t.red_off[top + 1]; ++e) {
        const Bits4 x = g & Bits4::load(t.red_mask + e * 4);
        if (!x.any()) continue;
        if (p < 0) {
          p = t.red_p[e];
          gp = x;
        } else {
          todo = todo | x;
        }
      }
      if (p < 0) break;  // the rest is an error here
      g = gp;
      int n = p >> 10;  // p: plen << 10 | lhs
      int x = min(n, ns);
      ns -= x;
      n -= x;
      x = min(n, mm);
      mm -= x;
      n -= x;
      k -= n;
      if (k < 1) break;
      const int top2 = ns ? scr[ns - 1] : (mm ? ovl[mm - 1] : base[k - 1]);
      if (top2 >= t.S) break;
      if (ns >= cap) {
        bound = true;
        return res;
      }
      count_work(ctr, 2);
      top = t.go[top2 * t.NNT + (p & 1023)];
      scr[ns++] = (uint16_t)top;
    }
    if (it == max_chain && g.any()) {
      bound = true;
      return res;
    }
  }
  while (todo.any()) {
    const int tau = todo.lowest();
    todo.clear_lowest();
    int keep_o, m_o, ns;
    const int a = simulate(t, base, keep, ovl, m, tau, scr, cap, keep_o, m_o, ns, max_chain, ctr);
    if (a < 0) {
      bound = true;
      return res;
    }
    if (a > 0 && a != kAccept) res.set(tau);
  }
  return res;
}

// Per-lane walk state.  Acur is the allowed-terminal set of the current
// virtual stack when it is known without simulation: the context's set before
// any shift, and after the first shift of terminal tau the precomputed set
// A2[tau] (if the caller has it); after a second shift it is NULL and the
// reduce chains are simulated.
struct Walker {
  const uint16_t* base;
  int keep, m;
  int q, lx;
  uint32_t pc, wc;  // category bits of trie node lx (0 if lx < 0)
  int nshift;
  bool shifted;
  int pend;  // a first shift not yet applied to the overlay (-1: none)
  const uint32_t* Acur;
  const uint32_t* A2;
  LArr ovl, scr;  // overlay and simulation scratch, `cap` entries each
  int cap;
  uint32_t* ctr;  // work counters (measured walks), or NULL
};

__device__ __forceinline__ void walker_init(Walker& w, LArr ovl_store, LArr scr_store, int cap, const uint16_t* base,
                                            int keep, const uint16_t* ovl, int m, int q, int lx, uint32_t pc,
                                            uint32_t wc, const uint32_t* A, const uint32_t* A2,
                                            uint32_t* ctr = nullptr) {
  w.ctr = ctr;
  w.ovl = ovl_store;
  w.scr = scr_store;
  w.cap = cap;
  w.base = base;
  w.keep = keep;
  w.m = min(m, cap);  // callers pass m <= cap; a larger m would only be a caller bug
  for (int k = 0; k < w.m; ++k) w.ovl[k] = ovl[k];
  w.q = q;
  w.lx = lx;
  w.pc = pc;
  w.wc = wc;
  w.nshift = 0;
  w.shifted = false;
  w.pend = -1;
  w.Acur = A;
  w.A2 = A2;
}

__device__ __forceinline__ bool commit(Walker& w, int keep_o, int m_o, int ns, int target) {
  if (m_o + ns + 1 > w.cap) return false;
  w.keep = keep_o;
  w.m = m_o;
  for (int i = 0; i < ns; ++i) w.ovl[w.m++] = w.scr[i];
  w.ovl[w.m++] = (uint16_t)target;
  return true;
}

// Apply a deferred first shift to the overlay.  The terminal is in the
// allowed set of the stack it was deferred at, so it reaches SHIFT.
__device__ __forceinline__ bool materialize(const Tables& t, Walker& w, int max_chain) {
  int keep_o, m_o, ns;
  const int a = simulate(t, w.base, w.keep, w.ovl, w.m, w.pend, w.scr, w.cap, keep_o, m_o, ns, max_chain, w.ctr);
  w.pend = -1;
  if (a <= 0 || a == kAccept) return false;
  return commit(w, keep_o, m_o, ns, a - 1);
}

// Emission of the pending lexeme (Sec. 2, contextual resolution): the first
// candidate in priority order that is ignored or reaches SHIFT wins and is
// shifted.  While the walker knows the allowed set of its stack (Acur) the
// pick is a set test; a first shift whose successor allowed set is known (A2)
// is only recorded, and applied to the overlay when a later step needs the
// stack itself.  Returns 1 ok, 0 reject, -1 bound.
__device__ __forceinline__ int emit_set(const Tables& t, Walker& w, Bits4 K, int max_chain) {
  while (K.any()) {
    const int tau = K.lowest();
    K.clear_lowest();
    if (t.ign.has(tau)) return 1;
    if (w.Acur && !bit4(w.Acur, tau)) continue;
    if (w.Acur && w.nshift == 0 && w.A2) {
      w.pend = tau;
      w.shifted = true;
      w.Acur = w.A2 + tau * 4;
      w.nshift = 1;
      return 1;
    }
    if (w.pend >= 0 && !materialize(t, w, max_chain)) return -1;
    if (!w.Acur && K.count() > 0) {
      // several candidates left: find the first that reaches SHIFT (or is
      // ignored) with one set simulation, then simulate that one to shift it
      bool bound = false;
      Bits4 rest = K;
      rest.set(tau);
      const Bits4 ok =
          simulate_set(t, w.base, w.keep, w.ovl, w.m, rest.andnot(t.ign), w.scr, w.cap, max_chain, bound, w.ctr);
      if (bound) return -1;
      const int pick = (ok | (rest & t.ign)).lowest();
      if (pick < 0) return 0;
      if (t.ign.has(pick)) return 1;
      K = Bits4::zero();
      int keep_o, m_o, ns;
      const int a = simulate(t, w.base, w.keep, w.ovl, w.m, pick, w.scr, w.cap, keep_o, m_o, ns, max_chain, w.ctr);
      if (a <= 0 || a == kAccept || !commit(w, keep_o, m_o, ns, a - 1)) return -1;
      w.shifted = true;
      w.Acur = (w.nshift == 0 && w.A2) ? w.A2 + pick * 4 : nullptr;
      ++w.nshift;
      return 1;
    }
    int keep_o, m_o, ns;
    int a = simulate(t, w.base, w.keep, w.ovl, w.m, tau, w.scr, w.cap, keep_o, m_o, ns, max_chain, w.ctr);
    if (a < 0) return -1;
    if (a > 0 && a != kAccept) {
      if (!commit(w, keep_o, m_o, ns, a - 1)) return -1;
      w.shifted = true;
      w.Acur = (w.nshift == 0 && w.A2) ? w.A2 + tau * 4 : nullptr;
      ++w.nshift;
      return 1;
    }
  }
  return 0;
}

__device__ __forceinline__ int emit(const Tables& t, Walker& w, int max_chain) {
  return emit_set(t, w, cands(t, w.q, w.wc), max_chain);
}

// Def. 2 trailing liveness for live set L.  1 / 0 / -1.
__device__ __forceinline__ int trailing_set(const Tables& t, Walker& w, Bits4 L, int max_chain) {
  if ((L & t.ign).any()) return 1;
  if (const uint32_t* A = w.Acur) return (L & Bits4::load(A)).any() ? 1 : 0;
  if (w.pend >= 0 && !materialize(t, w, max_chain)) return -1;
  if (L.count() == 1) {
    int keep_o, m_o, ns;
    const int a =
        simulate(t, w.base, w.keep, w.ovl, w.m, L.lowest(), w.scr, w.cap, keep_o, m_o, ns, max_chain, w.ctr);
    if (a < 0) return -1;
    return a > 0 && a != kAccept ? 1 : 0;
  }
  bool bound = false;
  const Bits4 ok = simulate_set(t, w.base, w.keep, w.ovl, w.m, L, w.scr, w.cap, max_chain, bound, w.ctr);
  if (bound) return -1;
  return ok.any() ? 1 : 0;
}

__device__ __forceinline__ int trailing_live(const Tables& t, Walker& w, int max_chain) {
  return trailing_set(t, w, live_prime(t, w.q, w.pc), max_chain);
}

// A spelling's bytes: the first 16 come from one 16-byte load into registers,
// longer spellings read the rest from the byte array.
struct Spell {
  uint4 head;
  const uint8_t* all;
  int len;
  __device__ __forceinline__ int at(int i) const {
    if (i < 16) {
      const uint32_t w = i < 8 ? (i < 4 ? head.x : head.y) : (i < 12 ? head.z : head.w);
      return (int)((w >> ((i & 3) * 8)) & 0xFFu);
    }
    return all[i];
  }
};

__device__ __forceinline__ Spell load_spell(const Tables& t, int s) {
  Spell sp;
  const int off = t.spell_off[s];
  sp.len = t.spell_off[s + 1] - off;
  sp.head = __ldg(&t.spell16[s]);
  sp.all = t.spell_bytes + off;
  return sp;
}

// Walk one token's bytes (Sec. 4.1).  1 = the output stays a viable prefix,
// 0 = rejected, -1 = bound.
__device__ __forceinline__ int walk_bytes(const Tables& t, Walker& w, const Spell& sp, int max_chain) {
  const int len = sp.len;
  for (int i = 0; i < len; ++i) {
    count_work(w.ctr, 0);
    const int b = sp.at(i);
    const int c = t.byte_class[b];
    int nq = t.next[w.q * t.C + c];
    if (nq == kDead) {
      if (w.q == kStart) return 0;
      const int e = emit(t, w, max_chain);
      if (e <= 0) return e;
      w.q = kStart;
      w.lx = 0;
      w.pc = t.root_pc;
      w.wc = t.root_wc;
      nq = t.next[kStart * t.C + c];
      if (nq == kDead) return 0;
    }
    w.q = nq;
    w.lx = lex_step(t, w.lx, b, w.pc, w.wc);
    const Bits4 L = live_prime(t, w.q, w.pc);
    const bool any = w.Acur ? (L & (Bits4::load(w.Acur) | t.ign)).any() : L.any();
    if (!any) return 0;
  }
  return trailing_live(t, w, max_chain);
}

// EOS gate (Sec. 3.2).  1 / 0 / -1.
__device__ __forceinline__ int eos_gate(const Tables& t, Walker& w, int max_chain) {
  if (w.q != kStart) {
    int e = emit(t, w, max_chain);
    if (e <= 0) return e;
  }
  if (w.pend >= 0 && !materialize(t, w, max_chain)) return -1;
  int keep_o, m_o, ns;
  int a = simulate(t, w.base, w.keep, w.ovl, w.m, t.n_term, w.scr, w.cap, keep_o, m_o, ns, max_chain, w.ctr);
  if (a < 0) return -1;
  return a == kAccept ? 1 : 0;
}

__device__ __forceinline__ int class_id(const Tables& t, int kind, int q, uint32_t cats) {
  return ((kind * t.Q + q) << t.n_cat) | (int)(cats & ((1u << t.n_cat) - 1u));
}

// Terminal set of a class id, computed from the lexer tables.
__device__ __forceinline__ Bits4 class_terms(const Tables& t, int cls) {
  const int hi = cls >> t.n_cat;
  const uint32_t cats = (uint32_t)cls & ((1u << t.n_cat) - 1u);
  const int kind = hi / t.Q, q = hi - kind * t.Q;
  return lex_filter(t, kind ? t.acc : t.live, q, cats);
}

// The same, from the table of all class ids' sets built at specialization.
__device__ __forceinline__ Bits4 class_set(const Tables& t, int cls) { return Bits4::load(t.cls_sets + cls * 4); }

// Sec. 4.2 CI/CD classification of one spelling from lexer state (q, lx),
// with the stack abstracted away.  Emissions whose first candidate is ignored
// leave the stack alone and are dropped; every other emission, and the final
// liveness test, is a stack-dependent event.
//   no event but the final test      -> CI live class / kClsAcc / kClsRej
//   one emission, then ignored bytes -> CI candidate class (or kClsAcc)
//   otherwise                        -> kClsVC with its event record `rec`
//                                       (kClsCD when it has more than kMaxEv
//                                       emissions; then `first_key` is the
//                                       class of the first one, 0xFFFF if that
//                                       emission always succeeds)
__device__ __forceinline__ uint16_t classify(const Tables& t, int q, int lx, const uint8_t* bytes, int len,
                                             uint16_t& first_key, uint16_t* rec) {
  first_key = 0xFFFF;
  uint32_t pc = lx == 0 ? t.root_pc : 0u, wc = lx == 0 ? t.root_wc : 0u;
  int n = 0;
  bool first_ign = false, overflow = false;
  for (int i = 0; i < len; ++i) {
    const int b = bytes[i];
    const int c = t.byte_class[b];
    int nq = t.next[q * t.C + c];
    if (nq == kDead) {
      if (q == kStart) return kClsRej;
      const Bits4 K = cands(t, q, wc);
      const int first = K.lowest();
      if (first < 0) return kClsRej;
      if (!t.ign.has(first)) {
        if (n == 0) first_ign = (K & t.ign).any();
        if (n < kMaxEv)
          rec[2 + n] = (uint16_t)class_id(t, 1, q, wc);
        else
          overflow = true;
        ++n;
      }
      q = kStart;
      lx = 0;
      pc = t.root_pc;
      wc = t.root_wc;
      nq = t.next[kStart * t.C + c];
      if (nq == kDead) return kClsRej;
    }
    q = nq;
    lx = lex_step(t, lx, b, pc, wc);
  }
  const Bits4 L = live_prime(t, q, pc);
  const bool lign = (L & t.ign).any();
  if (!L.any()) return kClsRej;
  if (n == 0) return lign ? kClsAcc : (uint16_t)class_id(t, 0, q, pc);
  if (n == 1 && lign) return first_ign ? kClsAcc : rec[2];
  if (overflow) {
    first_key = first_ign ? 0xFFFF : rec[2];
    return kClsCD;
  }
  rec[0] = (uint16_t)n;
  rec[1] = lign ? kClsAcc : (uint16_t)class_id(t, 0, q, pc);
  return kClsVC;
}

// Verdict of an event record at the walker's stack: each event is an emission
// with the recorded candidate set, then the final liveness test.  1 / 0 / -1.
__device__ __forceinline__ int eval_record(const Tables& t, Walker& w, const uint16_t* rec, int max_chain) {
  const int n = rec[0];
  for (int i = 0; i < n; ++i) {
    count_work(w.ctr, 3);
    const int e = emit_set(t, w, class_set(t, rec[2 + i]), max_chain);
    if (e <= 0) return e;
  }
  const uint16_t f = rec[1];
  if (f == kClsAcc) return 1;
  return trailing_set(t, w, class_set(t, f), max_chain);
}

}  // namespace grid
