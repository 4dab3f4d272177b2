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

// CI class codes (Sec. 4.2).  Codes below kClsNA are class ids
// ((kind * Q + q) << n_cat | cats): kind 0 = the verdict is "the live set of
// (q, cats) meets A u I" (token ends inside one lexeme), kind 1 = "the
// candidate set of (q, cats) meets A u I" (one boundary, then ignored bytes).
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
  // vocabulary trie
  const int32_t* spell_off;
  const uint8_t* spell_bytes;
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

__device__ __forceinline__ int lex_step(const Tables& t, int lx, int b) {
  if (lx < 0) return -1;
  int lo = t.lx_cstart[lx], hi = t.lx_cstart[lx + 1];
  const int end = hi;
  while (lo < hi) {
    int mid = (lo + hi) >> 1;
    if ((int)t.lx_cbyte[mid] < b)
      lo = mid + 1;
    else
      hi = mid;
  }
  return (lo < end && (int)t.lx_cbyte[lo] == b) ? t.lx_cnode[lo] : -1;
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

__device__ __forceinline__ void live_prime(const Tables& t, int q, int lx, uint32_t out[4]) {
  lex_filter(t, t.live, q, lx >= 0 ? t.lx_pcats[lx] : 0u, out);
}

__device__ __forceinline__ void cands(const Tables& t, int q, int lx, uint32_t out[4]) {
  lex_filter(t, t.acc, q, lx >= 0 ? t.lx_wcats[lx] : 0u, out);
}

__device__ __forceinline__ int max_chain_of(const Tables& t) { return 2 * t.D + 256; }

// Reduce chain of terminal tau on the virtual stack base[0:keep] ++ ovl[0:m]
// (Sec. 3.2, "allowed terminals by simulation").  Returns the ACTION code that
// ends it (> 0: shift to code-1, or kAccept), 0 on error, -1 on a bound.  On
// shift/accept, (keep_o, m_o, scr[0:ns]) is the stack under the pushed state.
__device__ __forceinline__ int simulate(const Tables& t, const uint16_t* base, int keep, const uint16_t* ovl,
                                        int m, int tau, uint16_t* scr, int& keep_o, int& m_o, int& ns,
                                        int max_chain) {
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
    if (ns >= kMaxOvl) return -1;
    scr[ns++] = t.go[top2 * t.NNT + t.plhs[p]];
  }
  return -1;
}

struct Walker {
  const uint16_t* base;
  int keep, m;
  int q, lx;
  bool shifted;
  uint16_t ovl[kMaxOvl];
  uint16_t scr[kMaxOvl];
};

__device__ __forceinline__ bool commit(Walker& w, int keep_o, int m_o, int ns, int target) {
  if (m_o + ns + 1 > kMaxOvl) return false;
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
__device__ __forceinline__ int emit(const Tables& t, Walker& w, const uint32_t* A, int max_chain) {
  uint32_t K[4];
  cands(t, w.q, w.lx, K);
  for (int wd = 0; wd < 4; ++wd) {
    uint32_t bits = K[wd];
    while (bits) {
      int tau = wd * 32 + __ffs(bits) - 1;
      bits &= bits - 1;
      if (bit4(t.ignored, tau)) return 1;
      if (A && !w.shifted && !bit4(A, tau)) continue;
      int keep_o, m_o, ns;
      int a = simulate(t, w.base, w.keep, w.ovl, w.m, tau, w.scr, keep_o, m_o, ns, max_chain);
      if (a < 0) return -1;
      if (a > 0 && a != kAccept) {
        if (!commit(w, keep_o, m_o, ns, a - 1)) return -1;
        w.shifted = true;
        return 1;
      }
    }
  }
  return 0;
}

// Def. 2 trailing liveness.  1 / 0 / -1.
__device__ __forceinline__ int trailing_live(const Tables& t, Walker& w, const uint32_t* A, int max_chain) {
  uint32_t L[4];
  live_prime(t, w.q, w.lx, L);
  if ((L[0] & t.ignored[0]) | (L[1] & t.ignored[1]) | (L[2] & t.ignored[2]) | (L[3] & t.ignored[3])) return 1;
  if (A && !w.shifted) return ((L[0] & A[0]) | (L[1] & A[1]) | (L[2] & A[2]) | (L[3] & A[3])) ? 1 : 0;
  for (int wd = 0; wd < 4; ++wd) {
    uint32_t bits = L[wd];
    while (bits) {
      int tau = wd * 32 + __ffs(bits) - 1;
      bits &= bits - 1;
      int keep_o, m_o, ns;
      int a = simulate(t, w.base, w.keep, w.ovl, w.m, tau, w.scr, keep_o, m_o, ns, max_chain);
      if (a < 0) return -1;
      if (a > 0 && a != kAccept) return 1;
    }
  }
  return 0;
}

// Walk one token's bytes (Sec. 4.1).  1 = the output stays a viable prefix,
// 0 = rejected (every spelling sharing bytes[0..rej] is rejected too:
// rejection is monotone under extension), -1 = bound.
__device__ __forceinline__ int walk_bytes(const Tables& t, Walker& w, const uint8_t* bytes, int len,
                                          const uint32_t* A, int max_chain, int& rej) {
  uint32_t AI[4] = {0, 0, 0, 0};
  if (A) {
#pragma unroll
    for (int k = 0; k < 4; ++k) AI[k] = A[k] | t.ignored[k];
  }
  for (int i = 0; i < len; ++i) {
    const int b = bytes[i];
    const int c = t.byte_class[b];
    int nq = t.next[w.q * t.C + c];
    if (nq == kDead) {
      if (w.q == kStart) {
        rej = i;
        return 0;
      }
      int e = emit(t, w, A, max_chain);
      if (e <= 0) {
        rej = i;
        return e;
      }
      w.q = kStart;
      w.lx = 0;
      nq = t.next[kStart * t.C + c];
      if (nq == kDead) {
        rej = i;
        return 0;
      }
    }
    w.q = nq;
    w.lx = lex_step(t, w.lx, b);
    uint32_t L[4];
    live_prime(t, w.q, w.lx, L);
    bool any;
    if (A && !w.shifted)
      any = (L[0] & AI[0]) | (L[1] & AI[1]) | (L[2] & AI[2]) | (L[3] & AI[3]);
    else
      any = L[0] | L[1] | L[2] | L[3];
    if (!any) {
      rej = i;
      return 0;
    }
  }
  int r = trailing_live(t, w, A, max_chain);
  if (r == 0) rej = len - 1;
  return r;
}

// EOS gate (Sec. 3.2).  1 / 0 / -1.
__device__ __forceinline__ int eos_gate(const Tables& t, Walker& w, const uint32_t* A, int max_chain) {
  if (w.q != kStart) {
    int e = emit(t, w, A, max_chain);
    if (e <= 0) return e;
  }
  int keep_o, m_o, ns;
  int a = simulate(t, w.base, w.keep, w.ovl, w.m, t.n_term, w.scr, keep_o, m_o, ns, max_chain);
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
// candidate is ignored leave the stack alone; the first emission whose first
// candidate is a parser terminal makes the verdict depend on A; anything that
// then still depends on the stack makes the spelling CD.
__device__ __forceinline__ uint16_t classify(const Tables& t, int q, int lx, const uint8_t* bytes, int len) {
  int key = -1;
  bool key_ign = false;
  for (int i = 0; i < len; ++i) {
    const int b = bytes[i];
    const int c = t.byte_class[b];
    int nq = t.next[q * t.C + c];
    if (nq == kDead) {
      if (q == kStart) return kClsRej;
      uint32_t K[4];
      cands(t, q, lx, K);
      const int first = lowest4(K);
      if (first < 0) return kClsRej;
      if (!bit4(t.ignored, first)) {
        if (key >= 0) return kClsCD;
        key = class_id(t, 1, q, lx >= 0 ? t.lx_wcats[lx] : 0u);
        key_ign = (K[0] & t.ignored[0]) | (K[1] & t.ignored[1]) | (K[2] & t.ignored[2]) | (K[3] & t.ignored[3]);
      }
      q = kStart;
      lx = 0;
      nq = t.next[kStart * t.C + c];
      if (nq == kDead) return kClsRej;
    }
    q = nq;
    lx = lex_step(t, lx, b);
  }
  uint32_t L[4];
  live_prime(t, q, lx, L);
  const bool lign = (L[0] & t.ignored[0]) | (L[1] & t.ignored[1]) | (L[2] & t.ignored[2]) | (L[3] & t.ignored[3]);
  const bool lany = L[0] | L[1] | L[2] | L[3];
  if (key < 0) {
    if (lign) return kClsAcc;
    if (!lany) return kClsRej;
    return (uint16_t)class_id(t, 0, q, lx >= 0 ? t.lx_pcats[lx] : 0u);
  }
  if (lign) return key_ign ? kClsAcc : (uint16_t)key;
  if (!lany) return kClsRej;
  return kClsCD;
}

}  // namespace grid
