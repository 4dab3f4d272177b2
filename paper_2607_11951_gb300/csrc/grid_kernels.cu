// libgrid device side for sm_103a: table upload, configurations, and the
// kernels of the cold full-vocabulary mask.
//
//   k_reset    configurations <- start configuration (Def. 1)
//   k_prep     per row: allowed terminals A(sigma) by reduce-chain simulation,
//              the EOS gate (Sec. 3.2), and clearing of the row's scratch
//   k_walk     per (row, spelling range): walk every token's bytes through the
//              lexer DFA and the identifier trie; each emission picks the
//              highest-priority parser-viable candidate and is shifted on a
//              per-lane copy-on-write overlay over the row's read-only stack;
//              rejected prefixes skip their whole trie subtree (Sec. 4.1)
//   k_pack     spelling-order verdict bits -> id-order mask words with alias
//              expansion, EOS bit, special tokens zero, empty-mask status
//   k_advance  per row: feed sampled tokens, commit shifts/reduces (Sec. 6.1)
//   k_apply    logits <- -inf where the mask bit is 0 (Sec. 2)
//
// Every loop is bounded; a bound that is hit writes GRID_ST_BOUND and the
// token is counted as rejected.  No kernel traps.

#include <cuda_runtime.h>

#include <cstring>
#include <string>
#include <vector>

#include "grid_internal.h"

namespace grid {
namespace {

constexpr int kMaxOvl = 64;       // per-token overlay / scratch entries per lane
constexpr int kWalkWarps = 4;     // warps per k_walk block
constexpr int kWalkSpan = 128;    // spellings per warp task

#define GRID_CUDA(call)                                                                  \
  do {                                                                                   \
    cudaError_t e_ = (call);                                                             \
    if (e_ != cudaSuccess)                                                               \
      return set_error(GRID_E_CUDA, std::string(#call) + ": " + cudaGetErrorString(e_)); \
  } while (0)

// All device tables of one (grammar, vocabulary) pair; passed by value.
struct Tables {
  int n_term, T1, S, NNT, P, Q, C, n_cat, LN;
  int NS, V, eos, W, D;
  uint32_t ignored[4];
  uint32_t catmask[4];
  int cat_term[32];
  const uint8_t* byte_class;
  const uint16_t* next;
  const uint32_t* acc;
  const uint32_t* live;
  const int16_t* action;
  const uint16_t* go;
  const uint8_t* plen;
  const uint16_t* plhs;
  const int32_t* lx_cstart;
  const uint8_t* lx_cbyte;
  const int32_t* lx_cnode;
  const uint32_t* lx_pcats;
  const uint32_t* lx_wcats;
  const int32_t* spell_off;
  const uint8_t* spell_bytes;
  const int32_t* skip;
  const int32_t* spell_of_id;
};

// Per-row scratch written by k_prep and read by k_walk / k_pack.
struct RowCtx {
  uint32_t A[4];      // allowed terminals at the row's stack
  int32_t eos_ok;
  int32_t status;
  uint32_t nonempty;
  uint32_t done_blocks;
};

struct DevConfigs {
  uint16_t* stack;  // B*D
  int32_t* depth;
  int32_t* q;
  int32_t* lx;
  int32_t* flags;   // bit 0 = complete
};

__device__ __forceinline__ bool bit4(const uint32_t* m, int t) { return (m[t >> 5] >> (t & 31)) & 1u; }

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

// Terminal set of state q filtered by the lexicon: non-category terminals pass,
// category terminal c passes iff bit c of `cats` is set.
__device__ __forceinline__ void lex_filter(const Tables& t, const uint32_t* __restrict__ src, int q,
                                           uint32_t cats, uint32_t out[4]) {
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

// Virtual stack = base[0:keep] ++ ovl[0:m] ++ scr[0:ns].  Runs the reduce
// chain of terminal tau without modifying base or ovl.  Returns the ACTION
// code that ends the chain (>0 shift target+1, kAccept) or 0 (error) or -1
// (bound).  On a shift/accept, (keep_o, m_o, scr[0:ns]) is the stack below
// the pushed state.
__device__ int simulate(const Tables& t, const uint16_t* __restrict__ base, int keep,
                        const uint16_t* ovl, int m, int tau, uint16_t* scr, int& keep_o, int& m_o,
                        int& ns, int max_chain) {
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

// Per-token walk state over a row.
struct Walker {
  const uint16_t* base;
  int keep, m;
  int q, lx;
  bool shifted;
  uint16_t ovl[kMaxOvl];
  uint16_t scr[kMaxOvl];
};

// Commit the result of a successful simulate(tau) + push of the shift target.
__device__ __forceinline__ bool commit(Walker& w, int keep_o, int m_o, int ns, int target) {
  if (m_o + ns + 1 > kMaxOvl) return false;
  w.keep = keep_o;
  w.m = m_o;
  for (int i = 0; i < ns; ++i) w.ovl[w.m++] = w.scr[i];
  w.ovl[w.m++] = (uint16_t)target;
  return true;
}

// Emit the pending lexeme of (w.q, w.lx): pick the first candidate in priority
// order that is ignored or reaches SHIFT; shift it.  `A` (may be NULL) is the
// allowed set of the unmodified row stack, usable while nothing was shifted.
// Returns 1 ok, 0 reject, -1 bound.
__device__ int emit(const Tables& t, Walker& w, const uint32_t* A, int max_chain) {
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

// Trailing liveness (Def. 2): some terminal live at (q, lx) is ignored or
// allowed at the current virtual stack.  1 / 0 / -1 (bound).
__device__ int trailing_live(const Tables& t, Walker& w, const uint32_t* A, int max_chain) {
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

// Walk the bytes of one token from the walker's state (Sec. 4.1).  Returns 1 if
// the output stays a viable prefix, 0 if rejected (rej = index of the byte
// from which on every extension is rejected), -1 on a bound.
__device__ int walk_bytes(const Tables& t, Walker& w, const uint8_t* __restrict__ bytes, int len,
                          const uint32_t* A, int max_chain, int& rej) {
  uint32_t AI[4];
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

// EOS gate (Sec. 3.2): the pending lexeme finalizes (same pick) and the reduce
// chain of $end reaches ACCEPT on the resulting scratch stack.
__device__ int eos_gate(const Tables& t, Walker& w, const uint32_t* A, int max_chain) {
  if (w.q != kStart) {
    int e = emit(t, w, A, max_chain);
    if (e <= 0) return e;
  }
  int keep_o, m_o, ns;
  int a = simulate(t, w.base, w.keep, w.ovl, w.m, t.n_term, w.scr, keep_o, m_o, ns, max_chain);
  if (a < 0) return -1;
  return a == kAccept ? 1 : 0;
}

__device__ __forceinline__ int max_chain_of(const Tables& t) { return 2 * t.D + 256; }

// ---------------------------------------------------------------------------
__global__ void k_reset(DevConfigs c, int B, int D) {
  int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  c.stack[(size_t)b * D] = 0;
  c.depth[b] = 1;
  c.q[b] = kStart;
  c.lx[b] = 0;
  c.flags[b] = 0;
}

// One warp per row: A(sigma) (lanes over terminals), EOS gate, scratch clear.
__global__ void k_prep(Tables t, DevConfigs c, RowCtx* __restrict__ ctx, uint32_t* __restrict__ verd,
                       int B, int words_ns) {
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (b >= B) return;
  RowCtx& r = ctx[b];
  uint32_t* vb = verd + (size_t)b * words_ns;
  for (int i = lane; i < words_ns; i += 32) vb[i] = 0u;
  const int complete = c.flags[b] & 1;
  const uint16_t* base = c.stack + (size_t)b * t.D;
  const int depth = c.depth[b];
  const int mc = max_chain_of(t);
  int status = complete ? GRID_ST_COMPLETE : GRID_ST_OK;
  uint32_t A[4] = {0, 0, 0, 0};
  if (!complete) {
    for (int wd = 0; wd < 4; ++wd) {
      int tau = wd * 32 + lane;
      bool ok = false;
      if (tau < t.n_term && !bit4(t.ignored, tau)) {
        uint16_t scr[kMaxOvl];
        int keep_o, m_o, ns;
        int a = simulate(t, base, depth, nullptr, 0, tau, scr, keep_o, m_o, ns, mc);
        ok = a > 0 && a != kAccept;
        if (a < 0) status = GRID_ST_BOUND;
      }
      A[wd] = __ballot_sync(0xffffffffu, ok);
    }
    status = __reduce_max_sync(0xffffffffu, status);
  }
  if (lane == 0) {
    int eos = 0;
    if (!complete) {
      Walker w;
      w.base = base;
      w.keep = depth;
      w.m = 0;
      w.q = c.q[b];
      w.lx = c.lx[b];
      w.shifted = false;
      int e = eos_gate(t, w, A, mc);
      if (e < 0) status = GRID_ST_BOUND;
      eos = e > 0;
    }
    for (int k = 0; k < 4; ++k) r.A[k] = A[k];
    r.eos_ok = eos;
    r.status = status;
    r.nonempty = 0;
    r.done_blocks = 0;
  }
}

// grid = (chunks, B); each warp walks kWalkSpan consecutive spellings.
__global__ void __launch_bounds__(kWalkWarps * 32) k_walk(Tables t, DevConfigs c, RowCtx* __restrict__ ctx,
                                                          uint32_t* __restrict__ verd, int words_ns) {
  const int b = blockIdx.y;
  if (c.flags[b] & 1) return;
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int lo = (blockIdx.x * kWalkWarps + warp) * kWalkSpan;
  __shared__ uint32_t sA[4];
  if (threadIdx.x < 4) sA[threadIdx.x] = ctx[b].A[threadIdx.x];
  __syncthreads();
  if (lo >= t.NS) return;
  const int hi = min(lo + kWalkSpan, t.NS);
  uint32_t A[4] = {sA[0], sA[1], sA[2], sA[3]};
  const uint16_t* base = c.stack + (size_t)b * t.D;
  const int depth = c.depth[b], q0 = c.q[b], lx0 = c.lx[b];
  const int mc = max_chain_of(t);
  uint32_t* vb = verd + (size_t)b * words_ns;
  int bound = 0;
  Walker w;
  for (int cursor = lo; cursor < hi;) {
    const int s = cursor + lane;
    int ok = 0, rej = -1;
    if (s < hi) {
      const int off = t.spell_off[s];
      const int len = t.spell_off[s + 1] - off;
      w.base = base;
      w.keep = depth;
      w.m = 0;
      w.q = q0;
      w.lx = lx0;
      w.shifted = false;
      int r = walk_bytes(t, w, t.spell_bytes + off, len, A, mc, rej);
      if (r < 0) {
        bound = 1;
        rej = -1;
      }
      ok = r > 0;
    }
    const uint32_t m = __ballot_sync(0xffffffffu, ok);
    if (lane == 0 && m) {
      const int sh = cursor & 31;
      atomicOr(&vb[cursor >> 5], m << sh);
      if (sh && (m >> (32 - sh))) atomicOr(&vb[(cursor >> 5) + 1], m >> (32 - sh));
    }
    // skip the rejected subtree of the last lane's spelling
    int nxt = cursor + 32;
    const int last = min(31, hi - 1 - cursor);
    const int lrej = __shfl_sync(0xffffffffu, rej, last);
    if (lrej >= 0) {
      const int sl = cursor + last;
      const int sk = t.skip[t.spell_off[sl] + lrej];
      nxt = max(nxt, sk);
    }
    cursor = nxt;
  }
  if (__any_sync(0xffffffffu, bound) && lane == 0) atomicCAS(&ctx[b].status, GRID_ST_OK, GRID_ST_BOUND);
}

// grid = (ceil(W/8), B), 256 threads: one thread per token id.
__global__ void k_pack(Tables t, RowCtx* __restrict__ ctx, const uint32_t* __restrict__ verd, int words_ns,
                       uint32_t* __restrict__ mask, int32_t* __restrict__ d_status) {
  const int b = blockIdx.y;
  const int id = blockIdx.x * blockDim.x + threadIdx.x;
  const int lane = threadIdx.x & 31;
  RowCtx& r = ctx[b];
  const bool complete = r.status == GRID_ST_COMPLETE;
  bool bit = false;
  if (id < t.V && !complete) {
    if (id == t.eos) {
      bit = r.eos_ok != 0;
    } else {
      int s = t.spell_of_id[id];
      if (s >= 0) bit = (verd[(size_t)b * words_ns + (s >> 5)] >> (s & 31)) & 1u;
    }
  }
  const uint32_t word = __ballot_sync(0xffffffffu, bit);
  const int wi = id >> 5;
  if (lane == 0 && wi < t.W) {
    mask[(size_t)b * t.W + wi] = word;
    if (word) atomicOr(&r.nonempty, 1u);
    __threadfence();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    unsigned prev = atomicAdd(&r.done_blocks, 1u);
    if (prev == gridDim.x - 1) {
      __threadfence();
      int st = atomicAdd(&r.status, 0);
      if (st == GRID_ST_OK && atomicAdd(&r.nonempty, 0u) == 0u) st = GRID_ST_EMPTY_MASK;
      d_status[b] = st;
    }
  }
}

// One warp per row; lane 0 feeds the tokens, all lanes copy for out-of-place.
__global__ void k_advance(Tables t, DevConfigs cin, DevConfigs cout, const int32_t* __restrict__ tokens,
                          int n_steps, int32_t* __restrict__ d_status, int B, int copy) {
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (b >= B) return;
  if (copy) {
    const int d = cin.depth[b];
    for (int i = lane; i < d; i += 32) cout.stack[(size_t)b * t.D + i] = cin.stack[(size_t)b * t.D + i];
    if (lane == 0) {
      cout.depth[b] = d;
      cout.q[b] = cin.q[b];
      cout.lx[b] = cin.lx[b];
      cout.flags[b] = cin.flags[b];
    }
    __syncwarp();
  }
  if (lane != 0) return;
  uint16_t* stack = cout.stack + (size_t)b * t.D;
  int depth = cout.depth[b], q = cout.q[b], lx = cout.lx[b], flags = cout.flags[b];
  int status = GRID_ST_OK;
  const int mc = max_chain_of(t);
  Walker w;
  for (int k = 0; k < n_steps; ++k) {
    const int tok = tokens[(size_t)b * n_steps + k];
    if (tok < 0) continue;
    if (flags & 1) {
      status = GRID_ST_COMPLETE;
      break;
    }
    if (tok >= t.V) {
      status = GRID_ST_TOKEN_NOT_ALLOWED;
      break;
    }
    w.base = stack;
    w.keep = depth;
    w.m = 0;
    w.q = q;
    w.lx = lx;
    w.shifted = false;
    if (tok == t.eos) {
      int e = eos_gate(t, w, nullptr, mc);
      if (e < 0) {
        status = GRID_ST_BOUND;
        break;
      }
      if (e == 0) {
        status = GRID_ST_TOKEN_NOT_ALLOWED;
        break;
      }
      flags |= 1;
      continue;
    }
    const int s = t.spell_of_id[tok];
    if (s < 0) {
      status = GRID_ST_TOKEN_NOT_ALLOWED;
      break;
    }
    const int off = t.spell_off[s];
    int rej;
    int r = walk_bytes(t, w, t.spell_bytes + off, t.spell_off[s + 1] - off, nullptr, mc, rej);
    if (r < 0) {
      status = GRID_ST_BOUND;
      break;
    }
    if (r == 0) {
      status = GRID_ST_TOKEN_NOT_ALLOWED;
      break;
    }
    if (w.keep + w.m > t.D) {
      status = GRID_ST_STACK_OVERFLOW;
      break;
    }
    for (int i = 0; i < w.m; ++i) stack[w.keep + i] = w.ovl[i];
    depth = w.keep + w.m;
    q = w.q;
    lx = w.lx;
  }
  cout.depth[b] = depth;
  cout.q[b] = q;
  cout.lx[b] = lx;
  cout.flags[b] = flags;
  d_status[b] = status;
}

// In-place -inf fill: one thread per 32-byte sector of logits.
template <typename T>
__global__ void k_apply(const uint32_t* __restrict__ mask, T* __restrict__ logits, int B, int V, int W,
                        long long stride, int vec_ok) {
  constexpr int E = 32 / sizeof(T);  // elements per sector: 8 fp32 or 16 bf16
  const long long per_row = (V + E - 1) / E;
  const long long total = per_row * B;
  for (long long g = (long long)blockIdx.x * blockDim.x + threadIdx.x; g < total;
       g += (long long)gridDim.x * blockDim.x) {
    const int b = (int)(g / per_row);
    const int e0 = (int)(g - (long long)b * per_row) * E;
    const uint32_t word = mask[(size_t)b * W + (e0 >> 5)];
    const uint32_t bits = (word >> (e0 & 31)) & ((E == 32) ? 0xffffffffu : ((1u << E) - 1u));
    T* p = logits + (size_t)b * stride + e0;
    const int n = min(E, V - e0);
    if (vec_ok && n == E) {
      uint4* p4 = reinterpret_cast<uint4*>(p);
      if (bits == 0u) {
        uint4 v;
        if (sizeof(T) == 4)
          v = make_uint4(0xFF800000u, 0xFF800000u, 0xFF800000u, 0xFF800000u);
        else
          v = make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u);
        p4[0] = v;
        p4[1] = v;
      } else if (bits != ((1u << E) - 1u)) {
        uint4 v[2] = {p4[0], p4[1]};
        if (sizeof(T) == 4) {
          uint32_t* u = reinterpret_cast<uint32_t*>(v);
#pragma unroll
          for (int k = 0; k < 8; ++k)
            if (!((bits >> k) & 1u)) u[k] = 0xFF800000u;
        } else {
          uint16_t* u = reinterpret_cast<uint16_t*>(v);
#pragma unroll
          for (int k = 0; k < 16; ++k)
            if (!((bits >> k) & 1u)) u[k] = 0xFF80u;
        }
        p4[0] = v[0];
        p4[1] = v[1];
      }
    } else {
      for (int k = 0; k < n; ++k) {
        if (!((bits >> k) & 1u)) {
          if (sizeof(T) == 4)
            reinterpret_cast<uint32_t*>(p)[k] = 0xFF800000u;
          else
            reinterpret_cast<uint16_t*>(p)[k] = 0xFF80u;
        }
      }
    }
  }
}

template <typename T>
int upload(std::vector<void*>& owned, const std::vector<T>& v, const T** out) {
  void* p = nullptr;
  size_t n = std::max<size_t>(v.size(), 1) * sizeof(T);
  GRID_CUDA(cudaMalloc(&p, n));
  owned.push_back(p);
  if (!v.empty()) GRID_CUDA(cudaMemcpy(p, v.data(), v.size() * sizeof(T), cudaMemcpyHostToDevice));
  *out = static_cast<const T*>(p);
  return GRID_OK;
}

}  // namespace
}  // namespace grid

using namespace grid;

struct grid_spec {
  const grid_grammar* g = nullptr;
  const grid_vocab* v = nullptr;
  Tables t;
  std::vector<void*> owned;
  int device = 0;
};

struct grid_configs {
  int B = 0, D = 0, words_ns = 0;
  DevConfigs c;
  RowCtx* ctx = nullptr;
  uint32_t* verd = nullptr;
  std::vector<void*> owned;
};

extern "C" int grid_specialize(const grid_grammar* g, const grid_vocab* v, void* stream, grid_spec** out) {
  if (!g || !v || !out) return set_error(GRID_E_INVALID_ARG, "grid_specialize: bad arguments");
  *out = nullptr;
  const HostGrammar& h = g->h;
  const HostVocab& hv = v->h;
  auto* s = new grid_spec();
  s->g = g;
  s->v = v;
  Tables& t = s->t;
  std::memset(&t, 0, sizeof(t));
  t.n_term = h.n_term;
  t.T1 = h.T1;
  t.S = h.S;
  t.NNT = h.NNT;
  t.P = h.P;
  t.Q = h.Q;
  t.C = h.C;
  t.n_cat = h.n_cat;
  t.LN = h.LN;
  t.NS = hv.NS;
  t.V = hv.V;
  t.eos = hv.eos;
  t.W = (hv.V + 31) / 32;
  t.D = h.max_depth;
  for (int k = 0; k < 4; ++k) {
    t.ignored[k] = h.ignored[k];
    t.catmask[k] = h.catmask[k];
  }
  for (int c = 0; c < h.n_cat; ++c) t.cat_term[c] = h.cat_term[c];
  std::vector<uint8_t> bc(h.byte_class, h.byte_class + 256);
  int rc = GRID_OK;
  auto& o = s->owned;
  if ((rc = upload(o, bc, &t.byte_class)) || (rc = upload(o, h.next, &t.next)) ||
      (rc = upload(o, h.acc, &t.acc)) || (rc = upload(o, h.live, &t.live)) ||
      (rc = upload(o, h.action, &t.action)) || (rc = upload(o, h.go, &t.go)) ||
      (rc = upload(o, h.plen, &t.plen)) || (rc = upload(o, h.plhs, &t.plhs)) ||
      (rc = upload(o, h.lx_cstart, &t.lx_cstart)) || (rc = upload(o, h.lx_cbyte, &t.lx_cbyte)) ||
      (rc = upload(o, h.lx_cnode, &t.lx_cnode)) || (rc = upload(o, h.lx_pcats, &t.lx_pcats)) ||
      (rc = upload(o, h.lx_wcats, &t.lx_wcats)) || (rc = upload(o, hv.spell_off, &t.spell_off)) ||
      (rc = upload(o, hv.spell_bytes, &t.spell_bytes)) || (rc = upload(o, hv.skip, &t.skip)) ||
      (rc = upload(o, hv.spell_of_id, &t.spell_of_id))) {
    grid_spec_free(s);
    return rc;
  }
  cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
  if (e != cudaSuccess) {
    grid_spec_free(s);
    return set_error(GRID_E_CUDA, std::string("grid_specialize: ") + cudaGetErrorString(e));
  }
  cudaGetDevice(&s->device);
  *out = s;
  return GRID_OK;
}

extern "C" void grid_spec_free(grid_spec* s) {
  if (!s) return;
  for (void* p : s->owned) cudaFree(p);
  delete s;
}

extern "C" int grid_configs_create(const grid_spec* s, int32_t B, grid_configs** out) {
  if (!s || !out || B <= 0) return set_error(GRID_E_INVALID_ARG, "grid_configs_create: bad arguments");
  *out = nullptr;
  auto* c = new grid_configs();
  c->B = B;
  c->D = s->t.D;
  c->words_ns = (s->t.NS + 31) / 32 + 1;
  auto alloc = [&](void** p, size_t n) -> int {
    GRID_CUDA(cudaMalloc(p, n));
    c->owned.push_back(*p);
    return GRID_OK;
  };
  int rc;
  if ((rc = alloc((void**)&c->c.stack, (size_t)B * c->D * sizeof(uint16_t))) ||
      (rc = alloc((void**)&c->c.depth, B * sizeof(int32_t))) || (rc = alloc((void**)&c->c.q, B * sizeof(int32_t))) ||
      (rc = alloc((void**)&c->c.lx, B * sizeof(int32_t))) ||
      (rc = alloc((void**)&c->c.flags, B * sizeof(int32_t))) ||
      (rc = alloc((void**)&c->ctx, B * sizeof(RowCtx))) ||
      (rc = alloc((void**)&c->verd, (size_t)B * c->words_ns * sizeof(uint32_t)))) {
    grid_configs_free(c);
    return rc;
  }
  k_reset<<<(B + 127) / 128, 128>>>(c->c, B, c->D);
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    grid_configs_free(c);
    return set_error(GRID_E_CUDA, std::string("grid_configs_create: ") + cudaGetErrorString(e));
  }
  *out = c;
  return GRID_OK;
}

extern "C" void grid_configs_free(grid_configs* c) {
  if (!c) return;
  for (void* p : c->owned) cudaFree(p);
  delete c;
}

extern "C" int grid_configs_reset(const grid_spec* s, grid_configs* c, void* stream) {
  if (!s || !c) return set_error(GRID_E_INVALID_ARG, "grid_configs_reset: bad arguments");
  k_reset<<<(c->B + 127) / 128, 128, 0, (cudaStream_t)stream>>>(c->c, c->B, c->D);
  GRID_CUDA(cudaGetLastError());
  return GRID_OK;
}

extern "C" int grid_advance(const grid_spec* s, const grid_configs* in, grid_configs* out,
                            const int32_t* d_tokens, int32_t n_steps, int32_t* d_status, void* stream) {
  if (!s || !in || !out || !d_tokens || !d_status || n_steps < 0 || in->B != out->B || in->D != out->D)
    return set_error(GRID_E_INVALID_ARG, "grid_advance: bad arguments");
  const int B = in->B;
  k_advance<<<(B + 3) / 4, 128, 0, (cudaStream_t)stream>>>(s->t, in->c, out->c, d_tokens, n_steps, d_status, B,
                                                          in != out ? 1 : 0);
  GRID_CUDA(cudaGetLastError());
  return GRID_OK;
}

extern "C" int grid_masks(const grid_spec* s, const grid_configs* c, uint32_t* d_mask, int32_t* d_status,
                          void* stream) {
  if (!s || !c || !d_mask || !d_status) return set_error(GRID_E_INVALID_ARG, "grid_masks: bad arguments");
  cudaStream_t st = (cudaStream_t)stream;
  const Tables& t = s->t;
  const int B = c->B;
  k_prep<<<(B + 3) / 4, 128, 0, st>>>(t, c->c, c->ctx, c->verd, B, c->words_ns);
  const int per_block = kWalkWarps * kWalkSpan;
  dim3 gw((t.NS + per_block - 1) / per_block, B);
  if (t.NS > 0) k_walk<<<gw, kWalkWarps * 32, 0, st>>>(t, c->c, c->ctx, c->verd, c->words_ns);
  dim3 gp((t.W + 7) / 8, B);
  k_pack<<<gp, 256, 0, st>>>(t, c->ctx, c->verd, c->words_ns, d_mask, d_status);
  GRID_CUDA(cudaGetLastError());
  return GRID_OK;
}

extern "C" int grid_apply_mask(const uint32_t* d_mask, void* d_logits, int32_t dtype, int32_t B, int32_t V,
                               int64_t row_stride, void* stream) {
  if (!d_mask || !d_logits || B <= 0 || V <= 0 || row_stride < V ||
      (dtype != GRID_DTYPE_F32 && dtype != GRID_DTYPE_BF16))
    return set_error(GRID_E_INVALID_ARG, "grid_apply_mask: bad arguments");
  cudaStream_t st = (cudaStream_t)stream;
  const int W = (V + 31) / 32;
  const int esz = dtype == GRID_DTYPE_F32 ? 4 : 2;
  const int vec_ok = ((uintptr_t)d_logits % 16 == 0) && ((row_stride * esz) % 16 == 0);
  const long long sectors = (long long)B * ((V * esz + 31) / 32);
  int dev = 0, sms = 152;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  long long blocks = (sectors + 255) / 256;
  blocks = std::min<long long>(blocks, (long long)sms * 8);
  if (dtype == GRID_DTYPE_F32)
    k_apply<float><<<(int)blocks, 256, 0, st>>>(d_mask, (float*)d_logits, B, V, W, row_stride, vec_ok);
  else
    k_apply<uint16_t><<<(int)blocks, 256, 0, st>>>(d_mask, (uint16_t*)d_logits, B, V, W, row_stride, vec_ok);
  GRID_CUDA(cudaGetLastError());
  return GRID_OK;
}

extern "C" int grid_configs_export(const grid_configs* c, int32_t row, int32_t* stack, int32_t cap,
                                   int32_t* depth, int32_t* dfa_state, int32_t* lex_node, int32_t* flags) {
  if (!c || row < 0 || row >= c->B || !depth || !dfa_state || !lex_node || !flags || cap < 0 || (cap && !stack))
    return set_error(GRID_E_INVALID_ARG, "grid_configs_export: bad arguments");
  GRID_CUDA(cudaMemcpy(depth, c->c.depth + row, 4, cudaMemcpyDeviceToHost));
  GRID_CUDA(cudaMemcpy(dfa_state, c->c.q + row, 4, cudaMemcpyDeviceToHost));
  GRID_CUDA(cudaMemcpy(lex_node, c->c.lx + row, 4, cudaMemcpyDeviceToHost));
  GRID_CUDA(cudaMemcpy(flags, c->c.flags + row, 4, cudaMemcpyDeviceToHost));
  int n = std::min(*depth, cap);
  if (n > 0) {
    std::vector<uint16_t> tmp(n);
    GRID_CUDA(cudaMemcpy(tmp.data(), c->c.stack + (size_t)row * c->D, n * 2, cudaMemcpyDeviceToHost));
    for (int i = 0; i < n; ++i) stack[i] = tmp[i];
  }
  return GRID_OK;
}
