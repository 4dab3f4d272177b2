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
constexpr uint16_t kClsCD2 = 0xFFFB;  // two stack-dependent events: resolved by (key1, key2) lookups
constexpr uint16_t kClsNA = 0xFFFC;   // spelling does not continue this lexer state
constexpr uint16_t kClsAcc = 0xFFFD;  // viable for every allowed set
constexpr uint16_t kClsRej = 0xFFFE;  // viable for no allowed set
constexpr uint16_t kClsCD = 0xFFFF;   // context-dependent: walked against the live stack

struct Tables {
  int n_term, T1, S, NNT, P, Q, C, n_cat, LN;
  int NS, V, eos, W, D;
  uint32_t ignored[4];
  uint32_t catmask[4];
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
  const int32_t* skip;
  const int32_t* spell_of_id;
  const int32_t* first_of_byte;
  const uint8_t* first_byte_by_id;
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
  const uint32_t* pair_by_id; // n_tbl * V: (key1 << 16 | key2) of kClsCD2 spellings
};

__device__ __forceinline__ bool bit4(const uint32_t* m, int t) { return (m[t >> 5] >> (t & 31)) & 1u; }

__device__ __forceinline__ int lowest4(const uint32_t m[4]) {
#pragma unroll
  for (int w = 0; w < 4; ++w)
    if (m[w]) return w * 32 + __ffs(m[w]) - 1;
  return -1;
}

// Copy the staged block into shared memory and publish one block-wide copy of
// the table descriptor, rebased onto it, in shared memory (`ts`).  Every thread
// of the block must call this.
__device__ __forceinline__ void stage_tables(const Tables& t, Tables& ts, uint8_t* smem) {
  if (t.blob_bytes) {
    const uint4* src = reinterpret_cast<const uint4*>(t.blob);
    uint4* dst = reinterpret_cast<uint4*>(smem);
    for (int i = threadIdx.x; i < (t.blob_bytes >> 4); i += blockDim.x) dst[i] = src[i];
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
    }
  }
  __syncthreads();
}

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
__device__ __forceinline__ void lex_filter(const Tables& t, const uint32_t* src, int q, uint32_t cats,
                                           uint32_t out[4]) {
#pragma unroll
  for (int w = 0; w < 4; ++w) out[w] = src[q * 4 + w] & ~t.catmask[w];
  while (cats) {
    int c = __ffs(cats) - 1;
    cats &= cats - 1;
    int term = t.cat_term[c];
    out[term >> 5] |= src[q * 4 + (term >> 5)] & (1u << (term & 31));
  }
}

// live'(q, r): terminals live at q, category terminals only while r is a
// prefix of one of their words (pc = prefix category bits of r's trie node).
__device__ __forceinline__ void live_prime(const Tables& t, int q, uint32_t pc, uint32_t out[4]) {
  lex_filter(t, t.live, q, pc, out);
}

// Emission candidates of r: terminals accepting at q, category terminals only
// if r is one of their words (wc = word category bits of r's trie node).
__device__ __forceinline__ void cands(const Tables& t, int q, uint32_t wc, uint32_t out[4]) {
  lex_filter(t, t.acc, q, wc, out);
}

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
                                        LArr scr, int cap, int& keep_o, int& m_o, int& ns, int max_chain) {
  int k = keep, mm = m;
  ns = 0;
  for (int it = 0; it < max_chain; ++it) {
    int top = ns ? scr[ns - 1] : (mm ? ovl[mm - 1] : base[k - 1]);
    if (top >= t.S) return 0;
    int a = t.action[top * t.T1 + tau];
    if (a == 0) return 0;
    if (a > 0) {
      keep_o = k;
      m_o = mm;
      return a;
    }
    int p = -a - 1;
    int n = t.plen[p];
    int x = min(n, ns);
    ns -= x;
    n -= x;
    x = min(n, mm);
    mm -= x;
    n -= x;
    k -= n;
    if (k < 1) return 0;
    int top2 = ns ? scr[ns - 1] : (mm ? ovl[mm - 1] : base[k - 1]);
    if (top2 >= t.S) return 0;
    if (ns >= cap) return -1;
    scr[ns++] = t.go[top2 * t.NNT + t.plhs[p]];
  }
  return -1;
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
  const uint32_t* Acur;
  const uint32_t* A2;
  LArr ovl, scr;  // overlay and simulation scratch, `cap` entries each
  int cap;
};

__device__ __forceinline__ void walker_init(Walker& w, LArr ovl_store, LArr scr_store, int cap, const uint16_t* base,
                                            int keep, const uint16_t* ovl, int m, int q, int lx, uint32_t pc,
                                            uint32_t wc, const uint32_t* A, const uint32_t* A2) {
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

// Emission of the pending lexeme (Sec. 2, contextual resolution): the first
// candidate in priority order that is ignored or reaches SHIFT wins and is
// shifted.  `A` (may be NULL) = allowed set of the walker's starting stack,
// valid while nothing has been shifted.  Returns 1 ok, 0 reject, -1 bound.
__device__ __forceinline__ int emit(const Tables& t, Walker& w, int max_chain) {
  uint32_t K[4];
  cands(t, w.q, w.wc, K);
  for (int wd = 0; wd < 4; ++wd) {
    uint32_t bits = K[wd];
    while (bits) {
      int tau = wd * 32 + __ffs(bits) - 1;
      bits &= bits - 1;
      if (bit4(t.ignored, tau)) return 1;
      if (w.Acur && !bit4(w.Acur, tau)) continue;
      int keep_o, m_o, ns;
      int a = simulate(t, w.base, w.keep, w.ovl, w.m, tau, w.scr, w.cap, keep_o, m_o, ns, max_chain);
      if (a < 0) return -1;
      if (a > 0 && a != kAccept) {
        if (!commit(w, keep_o, m_o, ns, a - 1)) return -1;
        w.shifted = true;
        w.Acur = (w.nshift == 0 && w.A2) ? w.A2 + tau * 4 : nullptr;
        ++w.nshift;
        return 1;
      }
    }
  }
  return 0;
}

// Def. 2 trailing liveness.  1 / 0 / -1.
__device__ __forceinline__ int trailing_live(const Tables& t, Walker& w, int max_chain) {
  uint32_t L[4];
  live_prime(t, w.q, w.pc, L);
  if ((L[0] & t.ignored[0]) | (L[1] & t.ignored[1]) | (L[2] & t.ignored[2]) | (L[3] & t.ignored[3])) return 1;
  if (const uint32_t* A = w.Acur) return ((L[0] & A[0]) | (L[1] & A[1]) | (L[2] & A[2]) | (L[3] & A[3])) ? 1 : 0;
  for (int wd = 0; wd < 4; ++wd) {
    uint32_t bits = L[wd];
    while (bits) {
      int tau = wd * 32 + __ffs(bits) - 1;
      bits &= bits - 1;
      int keep_o, m_o, ns;
      int a = simulate(t, w.base, w.keep, w.ovl, w.m, tau, w.scr, w.cap, keep_o, m_o, ns, max_chain);
      if (a < 0) return -1;
      if (a > 0 && a != kAccept) return 1;
    }
  }
  return 0;
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
// 0 = rejected (every spelling sharing bytes[0..rej] is rejected too:
// rejection is monotone under extension), -1 = bound.
__device__ __forceinline__ int walk_bytes(const Tables& t, Walker& w, const Spell& sp, int max_chain, int& rej) {
  const int len = sp.len;
  for (int i = 0; i < len; ++i) {
    const int b = sp.at(i);
    const int c = t.byte_class[b];
    int nq = t.next[w.q * t.C + c];
    if (nq == kDead) {
      if (w.q == kStart) {
        rej = i;
        return 0;
      }
      int e = emit(t, w, max_chain);
      if (e <= 0) {
        rej = i;
        return e;
      }
      w.q = kStart;
      w.lx = 0;
      w.pc = t.root_pc;
      w.wc = t.root_wc;
      nq = t.next[kStart * t.C + c];
      if (nq == kDead) {
        rej = i;
        return 0;
      }
    }
    w.q = nq;
    w.lx = lex_step(t, w.lx, b, w.pc, w.wc);
    uint32_t L[4];
    live_prime(t, w.q, w.pc, L);
    bool any;
    if (const uint32_t* A = w.Acur)
      any = (L[0] & (A[0] | t.ignored[0])) | (L[1] & (A[1] | t.ignored[1])) | (L[2] & (A[2] | t.ignored[2])) |
            (L[3] & (A[3] | t.ignored[3]));
    else
      any = L[0] | L[1] | L[2] | L[3];
    if (!any) {
      rej = i;
      return 0;
    }
  }
  int r = trailing_live(t, w, max_chain);
  if (r == 0) rej = len - 1;
  return r;
}

// EOS gate (Sec. 3.2).  1 / 0 / -1.
__device__ __forceinline__ int eos_gate(const Tables& t, Walker& w, int max_chain) {
  if (w.q != kStart) {
    int e = emit(t, w, max_chain);
    if (e <= 0) return e;
  }
  int keep_o, m_o, ns;
  int a = simulate(t, w.base, w.keep, w.ovl, w.m, t.n_term, w.scr, w.cap, keep_o, m_o, ns, max_chain);
  if (a < 0) return -1;
  return a == kAccept ? 1 : 0;
}

__device__ __forceinline__ int class_id(const Tables& t, int kind, int q, uint32_t cats) {
  return ((kind * t.Q + q) << t.n_cat) | (int)(cats & ((1u << t.n_cat) - 1u));
}

// Terminal set of a class id (for the per-row class selection).
__device__ __forceinline__ void class_set(const Tables& t, int cls, uint32_t out[4]) {
  const int hi = cls >> t.n_cat;
  const uint32_t cats = (uint32_t)cls & ((1u << t.n_cat) - 1u);
  const int kind = hi / t.Q, q = hi - kind * t.Q;
  lex_filter(t, kind ? t.acc : t.live, q, cats, out);
}

// Sec. 4.2 CI/CD classification of one spelling from lexer state (q, lx),
// with the stack abstracted to its allowed set A.  Emissions whose first
// candidate is ignored leave the stack alone; an emission whose first candidate
// is a parser terminal, or the final liveness test, is a stack-dependent event.
//   one event  -> CI class (verdict = class set meets A u I)
//   two events -> kClsCD2 with pair = key1 << 16 | key2: the first event picks
//                 tau1 = lowest(set(key1) & A) and the second is decided by the
//                 allowed set after shifting tau1 (verdict-equivalent spellings
//                 share the pair; GRID Sec. 4.2 "verdict-equivalence grouping")
//   more       -> kClsCD, walked against the live stack.
// For kClsCD, `first_key` is the class of the first event (0xFFFF if that
// event always succeeds): the walk is skipped when that class is not selected.
__device__ __forceinline__ uint16_t classify(const Tables& t, int q, int lx, const uint8_t* bytes, int len,
                                             uint16_t& first_key, uint32_t& pair) {
  first_key = 0xFFFF;
  pair = 0u;
  uint32_t pc = lx == 0 ? t.root_pc : 0u, wc = lx == 0 ? t.root_wc : 0u;
  int key1 = -1, key2 = -1;
  bool ign1 = false, ign2 = false;
  for (int i = 0; i < len; ++i) {
    const int b = bytes[i];
    const int c = t.byte_class[b];
    int nq = t.next[q * t.C + c];
    if (nq == kDead) {
      if (q == kStart) return kClsRej;
      uint32_t K[4];
      cands(t, q, wc, K);
      const int first = lowest4(K);
      if (first < 0) return kClsRej;
      if (!bit4(t.ignored, first)) {
        const bool kign = (K[0] & t.ignored[0]) | (K[1] & t.ignored[1]) | (K[2] & t.ignored[2]) | (K[3] & t.ignored[3]);
        if (key1 < 0) {
          key1 = class_id(t, 1, q, wc);
          ign1 = kign;
        } else if (key2 < 0 && !ign1) {
          key2 = class_id(t, 1, q, wc);
          ign2 = kign;
        } else {
          first_key = ign1 ? 0xFFFF : (uint16_t)key1;
          return kClsCD;
        }
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
  uint32_t L[4];
  live_prime(t, q, pc, L);
  const bool lign = (L[0] & t.ignored[0]) | (L[1] & t.ignored[1]) | (L[2] & t.ignored[2]) | (L[3] & t.ignored[3]);
  const bool lany = L[0] | L[1] | L[2] | L[3];
  if (key1 < 0) {
    if (lign) return kClsAcc;
    if (!lany) return kClsRej;
    return (uint16_t)class_id(t, 0, q, pc);
  }
  if (key2 < 0) {
    if (lign) return ign1 ? kClsAcc : (uint16_t)key1;
    if (!lany) return kClsRej;
    if (ign1) {
      first_key = 0xFFFF;
      return kClsCD;
    }
    pair = ((uint32_t)key1 << 16) | (uint32_t)class_id(t, 0, q, pc);
    return kClsCD2;
  }
  if (lign) {
    if (ign2) return (uint16_t)key1;
    pair = ((uint32_t)key1 << 16) | (uint32_t)key2;
    return kClsCD2;
  }
  if (!lany) return kClsRej;
  first_key = (uint16_t)key1;
  return kClsCD;
}

}  // namespace grid
