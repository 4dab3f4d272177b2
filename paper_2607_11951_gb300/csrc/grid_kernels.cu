// libgrid device side for sm_103a: table upload, CI precompute, configurations
// and the kernels of the cold full-vocabulary mask.
//
// Specialization (grid_specialize, Sec. 4.2 / cold-schema specialization), for
// every precomputed lexer state (the start state and each state where no
// lexicon category is live) and every distinct spelling:
//   k_classify    the spelling's class: a CI class id (its verdict is a
//                 function of the allowed set alone), always / never viable,
//                 a verdict class (its stack-dependent events fit one record),
//                 or byte-walked CD (more events than a record holds)
//   k_events      the event records of the verdict-class spellings; the host
//                 merges equal records (after rewriting class ids with equal
//                 terminal sets to one id) into the table's verdict classes
//   k_compact     per lexer state: the ascending list of its byte-walked spellings
//   k_scatter_vc, k_permute   class codes and verdict-class indices re-indexed
//                 by token id (coalesced in k_pack)
//
// Mask step (grid_masks, Def. 4):
//   k_row    one block per row: the forced emission of the pending lexeme
//            (what every token whose first byte ends the lexeme must go
//            through) -> sigma', and the EOS gate (Sec. 3.2); the first bytes
//            that end the lexeme; one lane per terminal tau and context runs
//            tau's reduce chain (A0 = A(sigma), A1 = A(sigma') are the ballots)
//            and, for allowed tau, the allowed set after shifting tau (walks
//            simulate nothing before their second shift); then, for rows
//            without a table, the live first-byte ranges that continue the
//            lexeme, and the class selections
//   k_filter per row and context: the byte-walked spellings and the verdict
//            classes whose first stack-dependent emission can succeed
//   k_walk   persistent; per row: each surviving verdict class evaluated once
//            against the row's stack, and the byte walks: lanes walk token
//            bytes through the DFA and the identifier trie, emissions pick the
//            highest-priority parser-viable candidate on a copy-on-write
//            overlay (Sec. 4.1); first-byte subtrees of the trie in which no
//            spelling can survive are never entered; a walked spelling's
//            verdict is set for each of its ids (alias ids share a spelling
//            and so a verdict) in an id-indexed bitmap with the mask's layout
//   k_pack   per token id: CI class selection | verdict class | walked verdict
//            | EOS gate, packed into the id-order mask; with logits
//            (grid_masks_apply) the -inf fill of the word's sectors as well;
//            with a mask cache, the context-independent bits of a hit read
//            from the cache entry (or stored into the entry the row claimed)
// Decoding step (grid_advance_masks): the same kernels, k_row feeding each
// row's tokens on warp 0 of its block before it prepares the row.
// Parser step (grid_advance):  k_advance.   Masked logits:  k_apply.
//
// Every loop is bounded; hitting a bound writes GRID_ST_BOUND.  No kernel traps.

#include <cuda_runtime.h>

#include <algorithm>
#include <array>
#include <cstring>
#include <mutex>
#include <string>
#include <type_traits>
#include <unordered_map>
#include <utility>
#include <vector>

#include "grid_state.cuh"

namespace grid {
namespace {

constexpr int kWalkWarps = 8;    // warps per k_walk block
constexpr int kSpan = 32;        // CD list entries per walk item (one warp batch)
constexpr int kAdvWarps = 4;     // rows per k_advance block
constexpr int kStackWin = 1024;  // stacks up to this depth are copied to shared memory in k_row/k_advance
constexpr int kFilterPer = 4;    // records per k_filter thread
constexpr int kRangeSpan = 32;   // continuing first-byte ranges are walked in items of (up to) this many spellings
constexpr int kWalkWin = 512;    // k_walk mirrors row stacks up to this depth per warp
constexpr int kRowWarps = 6;     // k_row: warps per row block
constexpr int kRowJobWarps = 4;  // k_row: warps 2 .. 5 compute the allowed sets after one shift
// Class codes as k_pack reads them: CI class ids 0..ncls-1, then these five
// (so that one bit test of the row's class selection covers CI, always and
// never, and only verdict-class and walked tokens need a second lookup).
constexpr int kPackCodes = 5;  // ncls + 0 always, +1 never, +2 n/a, +3 verdict class, +4 walked;
                               // with vc_inline, ncls + 5 + v: verdict class v of the code's table
constexpr int kWalkRowsCached = 256;  // rows whose queue bounds k_walk keeps in shared memory
constexpr int kLaneOvl = 32;     // overlay / scratch entries per walk lane (shared memory)
constexpr int kMaxStage = 96 * 1024;
constexpr int kMaxRows = 65535;  // rows of one configurations object (a grid dimension of the mask kernels)

// ---------------------------------------------------------------------------
__global__ void k_reset(DevConfigs c, int B, int D) {
  int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  c.stack[(size_t)b * D] = 0;
  if (c.hs) c.hs[(size_t)b * D] = 0;  // H(root) = 0
  c.depth[b] = 1;
  c.q[b] = kStart;
  c.lx[b] = 0;
  c.flags[b] = 0;
}

// ---------------- specialization ----------------
__global__ void k_classify(Tables t, uint16_t* __restrict__ cls_sp, uint16_t* __restrict__ key_sp,
                           int32_t* __restrict__ counts) {
  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ Tables ts;
  stage_tables(t, ts, smem);
  const int tbl = blockIdx.y;
  const int q0 = t.tbl_q[tbl];
  const int lx0 = q0 == kStart ? 0 : -1;
  int ncd = 0, nvc = 0;
  uint16_t rec[kRecLen];
  for (int s = blockIdx.x * blockDim.x + threadIdx.x; s < t.NS; s += gridDim.x * blockDim.x) {
    const int off = t.spell_off[s];
    const int len = t.spell_off[s + 1] - off;
    const uint8_t* by = t.spell_bytes + off;
    uint16_t code, key = 0xFFFF;
    if (!t.ci_on)
      code = kClsCD;
    else if (q0 != kStart && ts.next[q0 * ts.C + ts.byte_class[by[0]]] == kDead)
      code = kClsNA;
    else
      code = classify(ts, q0, lx0, by, len, key, rec);
    cls_sp[(size_t)tbl * t.NS + s] = code;
    key_sp[(size_t)tbl * t.NS + s] = key;
    ncd += code == kClsCD;
    nvc += code == kClsVC;
  }
  ncd = __reduce_add_sync(0xffffffffu, ncd);
  nvc = __reduce_add_sync(0xffffffffu, nvc);
  if ((threadIdx.x & 31) == 0) {
    if (ncd) atomicAdd(&counts[2 * tbl], ncd);
    if (nvc) atomicAdd(&counts[2 * tbl + 1], nvc);
  }
}

// Event records of the kClsVC spellings, appended per table in any order:
// slot -> (table, spelling, record).
__global__ void k_events(Tables t, const uint16_t* __restrict__ cls_sp, const int32_t* __restrict__ vc_base,
                         int32_t* __restrict__ fill, int32_t* __restrict__ slot_tbl, int32_t* __restrict__ slot_sp,
                         uint16_t* __restrict__ slot_rec) {
  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ Tables ts;
  stage_tables(t, ts, smem);
  const int tbl = blockIdx.y;
  const int q0 = t.tbl_q[tbl];
  const int lx0 = q0 == kStart ? 0 : -1;
  uint16_t rec[kRecLen];
  for (int s = blockIdx.x * blockDim.x + threadIdx.x; s < t.NS; s += gridDim.x * blockDim.x) {
    if (cls_sp[(size_t)tbl * t.NS + s] != kClsVC) continue;
    const int off = t.spell_off[s];
    uint16_t key;
    for (int k = 0; k < kRecLen; ++k) rec[k] = 0;
    classify(ts, q0, lx0, t.spell_bytes + off, t.spell_off[s + 1] - off, key, rec);
    const int slot = vc_base[tbl] + atomicAdd(&fill[tbl], 1);
    slot_tbl[slot] = tbl;
    slot_sp[slot] = s;
    for (int k = 0; k < kRecLen; ++k) slot_rec[(size_t)slot * kRecLen + k] = rec[k];
  }
}

// Per lexer state q and mask word wi, the ids whose first byte ends a pending
// lexeme in state q (every id at the start state): the split of a row's ids
// between sigma' and sigma that k_pack applies one word at a time.
__global__ void k_killw(Tables t, uint32_t* __restrict__ out) {
  const int wi = blockIdx.x * blockDim.x + threadIdx.x;
  const int q = blockIdx.y;
  if (wi >= t.W) return;
  uint32_t w = 0u;
  for (int j = 0; j < 32; ++j) {
    const int id = 32 * wi + j;
    const int by = id < t.Vp ? t.first_byte_by_id[id] : 0;
    if (q == kStart || q == kDead || t.next[q * t.C + t.byte_class[by]] == kDead) w |= 1u << j;
  }
  out[(size_t)q * t.W + wi] = w;
}

// Terminal set of every class id (events and final tests of the verdict
// classes use nothing else of a class).
__global__ void k_class_sets(Tables t, uint4* __restrict__ out) {
  const int cls = blockIdx.x * blockDim.x + threadIdx.x;
  if (cls >= t.ncls) return;
  const Bits4 v = class_terms(t, cls);
  out[cls] = make_uint4(v.x, v.y, v.z, v.w);
}

__global__ void k_scatter_vc(const int32_t* __restrict__ slot_tbl, const int32_t* __restrict__ slot_sp,
                             const int32_t* __restrict__ slot_vc, int nslot, int NS, uint32_t* __restrict__ vc_sp) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < nslot) vc_sp[(size_t)slot_tbl[i] * NS + slot_sp[i]] = (uint32_t)slot_vc[i];
}

// One block per table: ordered stream compaction of the CD spellings.
__global__ void k_compact(const uint16_t* __restrict__ cls_sp, const uint16_t* __restrict__ key_sp, int NS,
                          const int32_t* __restrict__ cd_off, int32_t* __restrict__ cd_list,
                          uint16_t* __restrict__ cd_key) {
  __shared__ int32_t warp_tot[32];
  __shared__ int32_t base;
  const int tbl = blockIdx.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  if (threadIdx.x == 0) base = cd_off[tbl];
  __syncthreads();
  for (int s0 = 0; s0 < NS; s0 += blockDim.x) {
    const int s = s0 + threadIdx.x;
    const bool f = s < NS && cls_sp[(size_t)tbl * NS + s] == kClsCD;
    const uint32_t bal = __ballot_sync(0xffffffffu, f);
    if (lane == 0) warp_tot[warp] = __popc(bal);
    __syncthreads();
    int before = 0;
    for (int k = 0; k < warp; ++k) before += warp_tot[k];
    if (f) {
      const int at = base + before + __popc(bal & ((1u << lane) - 1u));
      cd_list[at] = s;
      cd_key[at] = key_sp[(size_t)tbl * NS + s];
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int tot = 0;
      for (int k = 0; k < nw; ++k) tot += warp_tot[k];
      base += tot;
    }
    __syncthreads();
  }
}

__global__ void k_permute(Tables t, const uint16_t* __restrict__ cls_sp, const uint32_t* __restrict__ vc_sp,
                          uint16_t* __restrict__ cls_by_id, uint32_t* __restrict__ vc_by_id,
                          uint8_t* __restrict__ fb_by_id) {
  const int id = blockIdx.x * blockDim.x + threadIdx.x;
  if (id >= t.Vp) return;
  const int s = t.spell_of_id[id];  // -1 for EOS, specials and the padding ids
  fb_by_id[id] = s >= 0 ? t.spell_bytes[t.spell_off[s]] : 0;
  for (int k = 0; k < t.n_tbl; ++k) {
    const uint16_t c = s >= 0 ? cls_sp[(size_t)k * t.NS + s] : kClsNA;
    uint16_t code = c;  // the k_pack code of c
    if (c >= kClsFirstCode)
      code = (uint16_t)(t.ncls + (c == kClsAcc ? 0 : c == kClsRej ? 1 : c == kClsNA ? 2 : c == kClsVC ? 3 : 4));
    if (c == kClsVC && t.vc_inline) code = (uint16_t)(t.ncls + kPackCodes + vc_sp[(size_t)k * t.NS + s]);
    cls_by_id[(size_t)k * t.Vp + id] = code;
    if (vc_by_id) vc_by_id[(size_t)k * t.Vp + id] = c == kClsVC ? vc_sp[(size_t)k * t.NS + s] : 0xFFFFFFFFu;
  }
}

// ---------------- mask step ----------------
// Class selection for allowed set A, word w0: bit c = set(c) meets A u I,
// the OR of the class masks of the terminals in A u I.  The terminals' words
// are loaded kSelBatch at a time, so that a word costs |A u I| / kSelBatch
// memory round trips instead of |A u I|.
constexpr int kSelBatch = 16;
__device__ __forceinline__ uint32_t select_word(const Tables& t, const Bits4 AI, int w0) {
  uint32_t acc = 0u;
  Bits4 r = AI;
  while (r.any()) {
    uint32_t v[kSelBatch];
#pragma unroll
    for (int k = 0; k < kSelBatch; ++k) {
      const int tau = r.lowest();
      v[k] = 0u;
      if (tau >= 0) {
        r.clear_lowest();
        v[k] = __ldg(&t.cls_mask[(size_t)tau * t.nselw + w0]);
      }
    }
#pragma unroll
    for (int k = 0; k < kSelBatch; ++k) acc |= v[k];
  }
  if (w0 == (t.ncls >> 5)) acc |= 1u << (t.ncls & 31);  // the code "always"
  return acc;
}

// The configuration one warp leaves after feeding its row's tokens (lane 0's
// values; `win`: the warp's shared-memory window holds the row's stack).
struct AdvOut {
  int depth, q, lx, flags, status;
  uint32_t pc, wc;
  bool win;
};

// Advance of row b by one warp (Sec. 3.1 parser step, Sec. 4.1 byte walk).
// The lanes copy the row's stack for an out-of-place advance and mirror it in
// `win` (kStackWin entries, 16-byte accesses when the row stride allows them);
// lane 0 then feeds the tokens, with its overlay and simulation scratch in
// `lo` / `ls`, and writes the configuration it leaves (and the row's status
// when d_status is given).  The loads that start a row are issued as two
// independent chains: the configuration and then its stack (the first 256
// entries are read before the depth is known), and the first token with its
// spelling.  Returns in lane 0 only; the other lanes return once the copy is
// done.
constexpr int kAdvSpec = 32;  // 16-byte stack accesses issued per lane before the depth is known
__device__ __forceinline__ bool advance_warp(const Tables& t, const Tables& ts, const DevConfigs& cin,
                                             const DevConfigs& cout, const int32_t* __restrict__ tokens,
                                             int n_steps, int32_t* __restrict__ d_status, int b, int copy,
                                             int lane, uint16_t* win, LArr lo, LArr ls, AdvOut& out) {
  // chain 1: the row's configuration (lanes 0-3), the speculative stack read
  const uint16_t* src = (copy ? cin.stack : cout.stack) + (size_t)b * t.D;
  uint16_t* stack = cout.stack + (size_t)b * t.D;
  int cf = 0;
  if (lane < 4) {
    const int32_t* f = lane == 0 ? (copy ? cin.depth : cout.depth)
                     : lane == 1 ? (copy ? cin.q : cout.q)
                     : lane == 2 ? (copy ? cin.lx : cout.lx)
                                 : (copy ? cin.flags : cout.flags);
    cf = f[b];
  }
  uint32_t cpc = 0u, cwc = 0u;  // category bits of the pending lexeme's trie node (lane 2)
  if (lane == 2 && cf >= 0) {
    cpc = t.lx_pcats[cf];
    cwc = t.lx_wcats[cf];
  }
  const bool vec = t.D % 8 == 0;  // rows start on 16-byte boundaries: 8 entries per access
  const uint4* s4 = reinterpret_cast<const uint4*>(src);
  uint4 sv = make_uint4(0u, 0u, 0u, 0u);
  if (vec && lane < kAdvSpec && lane * 8 < t.D) sv = s4[lane];
  // chain 2: the first token and its spelling (lane 0)
  int tok0 = -1, sp0 = -1;
  Spell spl0;
  spl0.len = 0;
  if (lane == 0 && n_steps > 0) {
    tok0 = tokens[(size_t)b * n_steps];
    if (tok0 >= 0 && tok0 < t.V && tok0 != t.eos) {
      sp0 = t.spell_of_id[tok0];
      if (sp0 >= 0) spl0 = load_spell(t, sp0);
    }
  }
  const int depth0 = __shfl_sync(0xffffffffu, cf, 0);
  bool use_win = depth0 <= kStackWin;
  if (vec) {
    const int n8 = (depth0 + 7) >> 3;  // (n8 * 8 <= D: the last access stays inside the row)
    uint4* d4 = reinterpret_cast<uint4*>(stack);
    uint4* w4 = reinterpret_cast<uint4*>(win);
    if (lane < n8) {
      if (copy) d4[lane] = sv;
      if (use_win) w4[lane] = sv;
    }
    for (int i = lane + kAdvSpec; i < n8; i += 32) {
      const uint4 v = s4[i];
      if (copy) d4[i] = v;
      if (use_win) w4[i] = v;
    }
  } else {
    for (int i = lane; i < depth0; i += 32) {
      const uint16_t v = src[i];
      if (copy) stack[i] = v;
      if (use_win) win[i] = v;
    }
  }
  if (copy && cout.hs) {  // the node hashes travel with the stack
    const uint64_t* hsrc = cin.hs + (size_t)b * t.D;
    uint64_t* hdst = cout.hs + (size_t)b * t.D;
    for (int i = lane; i < depth0; i += 32) hdst[i] = hsrc[i];
  }
  const int q0 = __shfl_sync(0xffffffffu, cf, 1);
  const int lx0 = __shfl_sync(0xffffffffu, cf, 2);
  const int flags0 = __shfl_sync(0xffffffffu, cf, 3);
  const uint32_t pc0 = __shfl_sync(0xffffffffu, cpc, 2), wc0 = __shfl_sync(0xffffffffu, cwc, 2);
  __syncwarp();
  if (lane != 0) return false;
  int depth = depth0, q = q0, lx = lx0, flags = flags0;
  uint32_t pc = pc0, wcat = wc0;
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
    walker_init(w, lo, ls, kMaxOvl, use_win ? win : stack, depth, nullptr, 0, q, lx, pc, wcat, nullptr, nullptr);
    if (tok == t.eos) {
      const int e = eos_gate(ts, w, mc);
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
    const int s = k == 0 ? sp0 : t.spell_of_id[tok];
    if (s < 0) {
      status = GRID_ST_TOKEN_NOT_ALLOWED;
      break;
    }
    const int r = walk_bytes(ts, w, k == 0 ? spl0 : load_spell(t, s), mc);
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
    if (cout.hs) {  // rolling hash of every pushed node: O(1) per push
      uint64_t* hrow = cout.hs + (size_t)b * t.D;
      uint64_t hp = hrow[w.keep - 1];
      for (int i = 0; i < w.m; ++i) {
        hp = node_hash(hp, t.acc_sym[w.ovl[i]]);
        hrow[w.keep + i] = hp;
      }
    }
    if (use_win && w.keep + w.m <= kStackWin) {
      for (int i = 0; i < w.m; ++i) win[w.keep + i] = w.ovl[i];
    } else {
      use_win = false;
    }
    depth = w.keep + w.m;
    q = w.q;
    lx = w.lx;
    pc = w.pc;
    wcat = w.wc;
  }
  cout.depth[b] = depth;
  cout.q[b] = q;
  cout.lx[b] = lx;
  cout.flags[b] = flags;
  if (d_status) d_status[b] = status;
  out.depth = depth;
  out.q = q;
  out.lx = lx;
  out.flags = flags;
  out.status = status;
  out.pc = pc;
  out.wc = wcat;
  out.win = use_win;
  return true;
}

// One block per row (kRowWarps warps), plus clearing blocks after the rows.
// Phase 1, every warp at once: warp 0 finds the first bytes that end the
// pending lexeme; warp 1 makes the forced emission of the pending lexeme
// (sigma -> sigma', what every token whose first byte ends the lexeme must go
// through) and the EOS gate (Sec. 3.2) on the stack it leaves; lanes of the
// job warps take one terminal tau each, in sigma (first half) or sigma'
// (second half, each lane making the same forced emission itself): tau is
// allowed iff its reduce chain reaches SHIFT (A0 and A1 are the warps'
// ballots), and then the allowed set after that shift is A2 (walks and verdict
// classes simulate nothing before their second shift).  Phase 2: warp 0 lays
// out the live first-byte ranges that continue the lexeme (rows without a CI
// table; they need A0), warps 1 .. 5 select the contexts' CI classes.  Then
// thread 0 writes the row's context for the later kernels and, with a mask
// cache, looks the row's key up (k_pack reads a ready entry) or claims an
// empty slot for it (k_pack fills it).
// Clearing blocks zero both verdict bitmaps and the verdict-class bits.
// With ADV the row's tokens are fed first (advance_warp on warp 0, from
// adv.cin into c), and the row is masked in the configuration that leaves:
// the advance of one row and the mask preparation of another overlap, and
// the stack window is taken from the advance.  The row's status is then the
// advance's error, if its token was refused, else the mask step's.
template <bool ADV>
__global__ void __launch_bounds__(kRowWarps * 32) k_row(Tables t, DevConfigs c, RowCtx* __restrict__ ctx,
                                                        RowRanges* __restrict__ rng, uint32_t* __restrict__ A2,
                                                        uint32_t* __restrict__ sel, uint32_t* __restrict__ verd0,
                                                        uint32_t* __restrict__ verd1, uint32_t* __restrict__ vcbits,
                                                        int n_vcbits, int B, int words_v, CacheDev cache,
                                                        AdvArgs adv) {
  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ Tables ts;
  __shared__ __align__(16) uint16_t s_stk[kStackWin];
  __shared__ uint16_t s_ovl1[kMaxOvl];
  __shared__ uint16_t s_ovl2[kRowJobWarps][kMaxOvl * 32];
  __shared__ uint16_t s_scr[kRowJobWarps][kMaxOvl * 32];
  __shared__ uint32_t s_A0[4], s_A1[4], s_keep[8], s_kill[8];
  __shared__ int s_row[8];  // complete, depth, q, lx, emit_ok, keep1, m1, eos_ok
  __shared__ uint32_t s_pc[2];
  __shared__ int s_status, s_total0, s_nrng, s_adv[2];
  if ((int)blockIdx.x >= B) {
    // clearing blocks: zero both verdict bitmaps and the verdict-class bits of every row
    pdl_wait();
    const size_t n = (size_t)B * words_v;
    const size_t n4 = n >> 2;
    const size_t stride = (size_t)(gridDim.x - B) * blockDim.x;
    const size_t first = (size_t)(blockIdx.x - B) * blockDim.x + threadIdx.x;
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    for (size_t i = first; i < n4; i += stride) {
      reinterpret_cast<uint4*>(verd0)[i] = z;
      reinterpret_cast<uint4*>(verd1)[i] = z;
    }
    for (size_t i = (n4 << 2) + first; i < n; i += stride) {
      verd0[i] = 0u;
      verd1[i] = 0u;
    }
    for (size_t i = first; i < (size_t)n_vcbits; i += stride) vcbits[i] = 0u;
    return;
  }
  stage_tables(t, ts, smem);
  pdl_wait();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int b = blockIdx.x;
  RowCtx& r = ctx[b];
  const uint16_t* base = c.stack + (size_t)b * t.D;
  const bool vec = !ADV && t.D % 8 == 0 && kStackWin / 8 <= kRowWarps * 32;
  uint4 sv = make_uint4(0u, 0u, 0u, 0u);
  if (ADV) {
    // the row's tokens, on warp 0 (overlay and scratch in job warp 0's area,
    // which phase 1 uses only after the barrier below)
    AdvOut o;
    if (warp == 0 && advance_warp(t, ts, adv.cin, c, adv.tokens, adv.n_steps, nullptr, b, adv.copy, lane, s_stk,
                                  LArr{s_scr[0], 1}, LArr{s_scr[0] + kMaxOvl, 1}, o)) {
      s_row[0] = o.flags & 1;
      s_row[1] = o.depth;
      s_row[2] = o.q;
      s_row[3] = o.lx;
      s_pc[0] = o.pc;
      s_pc[1] = o.wc;
      s_adv[0] = o.status;
      s_adv[1] = o.win ? 1 : 0;
      s_status = GRID_ST_OK;
      s_total0 = 0;
      s_nrng = 0;
    }
  } else {
    // the stack window is read before the depth is known (one 16-byte access
    // per thread), in parallel with the configuration
    if (vec && (int)threadIdx.x < kStackWin / 8 && (int)threadIdx.x * 8 < t.D)
      sv = reinterpret_cast<const uint4*>(base)[threadIdx.x];
    if (threadIdx.x == 0) {
      const int lx = c.lx[b];
      s_row[0] = c.flags[b] & 1;
      s_row[1] = c.depth[b];
      s_row[2] = c.q[b];
      s_row[3] = lx;
      s_pc[0] = lx >= 0 ? t.lx_pcats[lx] : 0u;
      s_pc[1] = lx >= 0 ? t.lx_wcats[lx] : 0u;
      s_adv[0] = GRID_ST_OK;
      s_adv[1] = 0;
      s_status = GRID_ST_OK;
      s_total0 = 0;
      s_nrng = 0;
    }
  }
  __syncthreads();
  const int complete = s_row[0], depth = s_row[1], q = s_row[2], lx = s_row[3];
  const uint32_t pc0 = s_pc[0], wc0 = s_pc[1];
  if (depth <= kStackWin) {  // the reduce chains below read the stack top repeatedly
    if (ADV && s_adv[1]) {
      // the advance left the row's stack in the window
    } else if (vec) {
      if ((int)threadIdx.x < ((depth + 7) >> 3)) reinterpret_cast<uint4*>(s_stk)[threadIdx.x] = sv;
    } else {
      for (int i = threadIdx.x; i < depth; i += blockDim.x) s_stk[i] = base[i];
    }
    base = s_stk;
  }
  __syncthreads();
  const int mc = max_chain_of(t);
  const int tbl0 = (q != kStart && t.ci_on) ? t.tbl_of_q[q] : -1;
  int status = GRID_ST_OK;
  // ---- phase 1: all at once
  if (threadIdx.x < 8) s_keep[threadIdx.x] = 0u;
  if (threadIdx.x < 4) {
    s_A0[threadIdx.x] = 0u;
    s_A1[threadIdx.x] = 0u;
  }
  __syncthreads();
  if (warp == 0) {
    // first bytes that end the pending lexeme (every byte when it is empty)
    for (int b0 = 0; b0 < 256; b0 += 32) {
      const int by = b0 + lane;
      const bool kill = q == kStart || ts.next[q * ts.C + ts.byte_class[by]] == kDead;
      const uint32_t word = __ballot_sync(0xffffffffu, kill);
      if (lane == 0) s_kill[b0 >> 5] = word;
    }
  } else if (warp == 1) {
    // the forced emission of the pending lexeme (sigma -> sigma'), and the
    // EOS gate (Sec. 3.2) on the stack it leaves
    int emit_ok = 0, keep1 = depth, m1 = 0, eos = 0;
    if (lane == 0 && !complete) {
      Walker w;
      uint16_t lo[kMaxOvl], ls[kMaxOvl];
      walker_init(w, LArr{lo, 1}, LArr{ls, 1}, kMaxOvl, base, depth, nullptr, 0, q, lx, pc0, wc0, nullptr, nullptr);
      if (q == kStart) {
        emit_ok = 1;
      } else {
        const int e = emit(ts, w, mc);
        if (e < 0) status = GRID_ST_BOUND;
        emit_ok = e > 0;
        keep1 = w.keep;
        m1 = w.m;
        for (int i = 0; i < m1; ++i) s_ovl1[i] = w.ovl[i];
      }
      if (emit_ok) {
        int keep_o, m_o, ns;
        const int a = simulate(ts, base, keep1, (const uint16_t*)s_ovl1, m1, t.n_term, LArr{ls, 1}, kMaxOvl, keep_o, m_o,
                               ns, mc);
        if (a < 0) status = GRID_ST_BOUND;
        eos = a == kAccept;
      }
      s_row[4] = emit_ok;
      s_row[5] = keep1;
      s_row[6] = m1;
      s_row[7] = eos;
    }
  } else if (!complete) {
    // job warps: lane l of job warp jw takes terminal tau = 32 jw + l (and
    // tau + 32 * half, ...) in one context: tau is allowed iff its reduce
    // chain reaches SHIFT (A0 / A1 are the ballots), and then the allowed set
    // after that shift (A2) comes from one set simulation.  sigma' lanes make
    // the forced emission themselves (the same pick as warp 1), so that both
    // contexts start at once.
    const int half = kRowJobWarps / 2;
    const int cx = warp - 2 >= half ? 1 : 0;
    const int jw = warp - 2 - cx * half;
    const LArr scr{s_scr[warp - 2] + lane, 32}, ovl{s_ovl2[warp - 2] + lane, 32};
    int keep = depth, m = 0;
    bool has_ctx = cx == 0 ? q != kStart : true;
    if (cx == 1 && q != kStart) {
      Walker w;
      walker_init(w, ovl, scr, kMaxOvl, base, depth, nullptr, 0, q, lx, pc0, wc0, nullptr, nullptr);
      const int e = emit(ts, w, mc);
      if (e < 0) status = GRID_ST_BOUND;
      has_ctx = e > 0;
      keep = w.keep;
      m = w.m;  // sigma' is base[0:keep] ++ ovl[0:m]
    }
    Bits4 G = Bits4::zero();
    for (int k = 0; k < t.n_term; ++k) G.set(k);
    G = G.andnot(ts.ign);
    for (int tau0 = jw * 32; has_ctx && tau0 < t.n_term; tau0 += 32 * half) {
      const int tau = tau0 + lane;
      bool allowed = false;
      Bits4 An = Bits4::zero();
      if (tau < t.n_term && !ts.ign.has(tau)) {
        int keep_o, m_o, ns;
        const int a = simulate(ts, base, keep, ovl, m, tau, scr, kMaxOvl, keep_o, m_o, ns, mc);
        if (a < 0) status = GRID_ST_BOUND;
        allowed = a > 0 && a != kAccept;
        if (allowed) {
          if (m_o + ns + 1 <= kMaxOvl) {
            // the stack after the shift, built in place: base[0:keep_o] ++
            // ovl[0:m_o] ++ scr[0:ns] ++ (a-1); sigma' itself is rebuilt for
            // the next terminal of this lane
            uint16_t saved[kMaxOvl];
            for (int i = 0; i < m; ++i) saved[i] = ovl[i];
            for (int i = 0; i < ns; ++i) ovl[m_o + i] = scr[i];
            ovl[m_o + ns] = (uint16_t)(a - 1);
            bool bound = false;
            An = simulate_set(ts, base, keep_o, ovl, m_o + ns + 1, G, scr, kMaxOvl, mc, bound);
            if (bound) status = GRID_ST_BOUND;
            for (int i = 0; i < m; ++i) ovl[i] = saved[i];
          } else {
            status = GRID_ST_BOUND;
          }
          uint32_t* out = A2 + (((size_t)b * 2 + cx) * t.T1 + tau) * 4;
          out[0] = An.x;
          out[1] = An.y;
          out[2] = An.z;
          out[3] = An.w;
        }
      }
      const uint32_t word = __ballot_sync(0xffffffffu, allowed);
      if (lane == 0 && word) atomicOr(cx ? &s_A1[tau0 >> 5] : &s_A0[tau0 >> 5], word);
    }
  }
  status = __reduce_max_sync(0xffffffffu, status);
  if (lane == 0 && status != GRID_ST_OK) atomicMax(&s_status, status);
  __syncthreads();
  const int emit_ok = complete ? 0 : s_row[4], keep1 = complete ? depth : s_row[5], m1 = complete ? 0 : s_row[6];
  const Bits4 A0 = Bits4::load(s_A0), A1 = Bits4::load(s_A1);
  // ---- phase 2: ranges (warp 0), class selections (warps 1, 2)
  if (!complete) {
    if (warp == 0 && q != kStart && tbl0 < 0) {
      // continuing first-byte ranges (rows without a CI table for q).  A first
      // byte whose lexeme has no live terminal in A0 u I (category terminals
      // counted only while the lexeme is a prefix of one of their words)
      // rejects every spelling it starts: liveness only shrinks along the
      // lexeme, and any later emission picks among its live terminals.
      int total0 = 0, nrng = 0;
      RowRanges& R = rng[b];
      const Bits4 AI = A0 | ts.ign;
      int lo_r[8], hi_r[8];
      uint32_t cw[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        lo_r[j] = t.first_of_byte[j * 32 + lane];
        hi_r[j] = t.first_of_byte[j * 32 + lane + 1];
      }
      int nc = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int by = j * 32 + lane;
        cw[j] = __ballot_sync(0xffffffffu, hi_r[j] > lo_r[j] && ts.next[q * ts.C + ts.byte_class[by]] != kDead);
        nc += __popc(cw[j]);
      }
      for (int i0 = 0; i0 < nc; i0 += 32) {  // the live test of the continuing bytes, one per lane
        int idx = i0 + lane, by = -1;
        if (idx < nc) {
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const int cnt = __popc(cw[j]);
            if (by < 0 && idx < cnt) by = j * 32 + (int)__fns(cw[j], 0u, idx + 1);
            if (by < 0) idx -= cnt;
          }
        }
        if (by >= 0) {
          uint32_t pc2 = 0u, wc2 = 0u;
          if (lx >= 0) lex_step(ts, lx, by, pc2, wc2);
          const int q2 = ts.next[q * ts.C + ts.byte_class[by]];
          if ((live_prime(ts, q2, pc2) & AI).any()) atomicOr(&s_keep[by >> 5], 1u << (by & 31));
        }
      }
      __syncwarp();
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const bool cont = (s_keep[j] >> lane) & 1u;
        const int chunks = cont ? (hi_r[j] - lo_r[j] + kRangeSpan - 1) / kRangeSpan : 0;
        const uint32_t bal = __ballot_sync(0xffffffffu, cont);
        int incl = chunks;
        for (int d = 1; d < 32; d <<= 1) {
          int v = __shfl_up_sync(0xffffffffu, incl, d);
          if (lane >= d) incl += v;
        }
        if (cont) {
          const int k = nrng + __popc(bal & ((1u << lane) - 1u));
          R.lo[k] = lo_r[j];
          R.hi[k] = hi_r[j];
          R.cpre[k] = total0 + incl - chunks;
        }
        total0 += __shfl_sync(0xffffffffu, incl, 31);
        nrng += __popc(bal);
      }
      if (lane == 0) {
        R.cpre[nrng] = total0;
        s_total0 = total0;
        s_nrng = nrng;
      }
    } else if (warp >= 1 && t.ci_on) {
      // both contexts' selection words, one per lane of warps 1 ..
      const Bits4 AI0 = A0 | ts.ign, AI1 = A1 | ts.ign;
      const int nw = t.nselw;
      for (int i = (warp - 1) * 32 + lane; i < 2 * nw; i += (kRowWarps - 1) * 32) {
        const int cx = i >= nw ? 1 : 0, w0 = i - cx * nw;
        if (cx ? !emit_ok : tbl0 < 0) continue;
        sel[((size_t)b * 2 + cx) * nw + w0] = select_word(ts, cx ? AI1 : AI0, w0);
      }
    }
  }
  __syncthreads();
  // ---- the row's context for the later kernels
  if (threadIdx.x == 0) {
    // configuration-keyed cache of the context-independent part (Sec. 4.3):
    // key = (kind, lexer state, emit_ok, A(sigma), A(sigma')); the CD residue
    // is never cached.  A ready entry with this key is read; an empty slot is
    // claimed and filled by k_pack; any other slot is left alone.
    int chit = -1, cfill = -1;
    if (cache.n && !complete) {
      uint32_t key[11];
      key[0] = (q != kStart && tbl0 < 0) ? 1u : 0u;
      key[1] = (uint32_t)q;
      key[2] = (uint32_t)emit_ok;
      for (int k = 0; k < 4; ++k) {
        key[3 + k] = s_A0[k];
        key[7 + k] = emit_ok ? s_A1[k] : 0u;
      }
      unsigned long long hsh = 1469598103934665603ull;  // FNV-1a over the key words
      for (int k = 0; k < 11; ++k) {
        hsh ^= key[k];
        hsh *= 1099511628211ull;
      }
      const int slot = (int)(hsh & (unsigned long long)(cache.n - 1));
      uint32_t* h = cache.hdr + (size_t)slot * 16;
      atomicAdd(&cache.stats[0], 1ull);
      const uint32_t state = *(volatile uint32_t*)h;
      if (state == 2u) {
        bool same = true;
        for (int k = 0; k < 11; ++k) same &= ((volatile uint32_t*)h)[1 + k] == key[k];
        if (same) {
          chit = slot;
          atomicAdd(&cache.stats[1], 1ull);
        }
      } else if (state == 0u && atomicCAS(h, 0u, 1u) == 0u) {
        for (int k = 0; k < 11; ++k) h[1 + k] = key[k];
        cfill = slot;
        atomicAdd(&cache.stats[2], 1ull);
      }
    }
    r.chit = chit;
    r.cfill = cfill;
    for (int k = 0; k < 4; ++k) {
      r.A0[k] = s_A0[k];
      r.A1[k] = emit_ok ? s_A1[k] : 0u;
    }
    for (int k = 0; k < 8; ++k) r.kill[k] = s_kill[k];
    r.q = q;
    r.lx = lx;
    r.pc0 = pc0;
    r.wc0 = wc0;
    r.depth = depth;
    r.tbl0 = tbl0;
    r.emit_ok = emit_ok;
    r.eos_ok = complete ? 0 : s_row[7];
    r.complete = complete;
    r.pack_done = 0ull;
    r.keep1 = keep1;
    r.m1 = m1;
    r.work0 = 0;
    r.nrange = s_total0;
    r.nsurv[0] = 0;
    r.nsurv[1] = 0;
    r.nvs[0] = 0;
    r.nvs[1] = 0;
    r.nrng = s_nrng;
  }
  for (int i = threadIdx.x; i < m1; i += blockDim.x) r.ovl1[i] = s_ovl1[i];
  if (threadIdx.x == 0) r.status = s_adv[0] != GRID_ST_OK ? s_adv[0] : (complete ? GRID_ST_COMPLETE : s_status);
}

// grid = (cd_blocks + vc_blocks, B, 2), 256 threads, kFilterPer records per
// thread (few blocks, all resident at once): compact, per row and context,
// what the walk has to evaluate.
//  - blocks x < cd_blocks: the byte-walked CD spellings that a walk could
//    admit: the class of the first stack-dependent emission must be selected
//    for the context's allowed set and, for sigma', the first byte must end
//    the pending lexeme; survivors go to surv[(b*2 + cx) * cap ...].
//  - the other blocks: the verdict classes whose first event's class is
//    selected (any other record fails at its first emission); survivors go to
//    vsurv[(b*2 + cx) * vcap ...].
// Both lists are in any order.
__global__ void __launch_bounds__(256) k_filter(Tables t, RowCtx* __restrict__ ctx, const uint32_t* __restrict__ sel,
                                                int32_t* __restrict__ surv, int cap, int32_t* __restrict__ vsurv,
                                                int vcap, int cd_blocks) {
  __shared__ int s_warp[8];
  __shared__ int s_base;
  pdl_wait();
  const int b = blockIdx.y, cx = blockIdx.z;
  RowCtx& r = ctx[b];
  const int q = r.q, tbl0 = r.tbl0;
  if (r.complete) return;
  if (cx == 1 && !r.emit_ok) return;
  if (cx == 0 && (q == kStart || tbl0 < 0)) return;
  const int tb = cx ? 0 : tbl0;
  const bool vc = (int)blockIdx.x >= cd_blocks;
  const int bx = vc ? (int)blockIdx.x - cd_blocks : (int)blockIdx.x;
  const int len = vc ? t.vc_off[tb + 1] - t.vc_off[tb] : t.cd_off[tb + 1] - t.cd_off[tb];
  const int i0 = bx * (int)blockDim.x * kFilterPer + threadIdx.x;  // records i0 + j * blockDim.x
  if (i0 - (int)threadIdx.x >= len) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t* csel = sel + ((size_t)b * 2 + cx) * t.nselw;
  bool pass[kFilterPer];
  int sv[kFilterPer];
#pragma unroll
  for (int j = 0; j < kFilterPer; ++j) {
    const int i = i0 + j * (int)blockDim.x;
    pass[j] = false;
    sv[j] = -1;
    if (i < len) {
      if (vc) {
        sv[j] = i;
        const uint16_t k = t.vc_first[t.vc_off[tb] + i];
        pass[j] = (csel[k >> 5] >> (k & 31)) & 1u;
      } else {
        const int s = t.cd_list[t.cd_off[tb] + i];
        sv[j] = s;
        const uint16_t k = t.cd_key[t.cd_off[tb] + i];
        pass[j] = k == 0xFFFF || ((csel[k >> 5] >> (k & 31)) & 1u);
        if (pass[j] && cx == 1 && q != kStart) {
          const int b0 = (int)(__ldg(&t.spell16[s]).x & 0xFFu);
          pass[j] = t.next[q * t.C + t.byte_class[b0]] == kDead;
        }
      }
    }
  }
  uint32_t bal[kFilterPer];
  int cnt = 0;
#pragma unroll
  for (int j = 0; j < kFilterPer; ++j) {
    bal[j] = __ballot_sync(0xffffffffu, pass[j]);
    cnt += __popc(bal[j]);
  }
  if (lane == 0) s_warp[warp] = cnt;
  __syncthreads();
  if (threadIdx.x == 0) {
    int tot = 0;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) {
      const int c = s_warp[k];
      s_warp[k] = tot;
      tot += c;
    }
    s_base = tot ? atomicAdd(vc ? &r.nvs[cx] : &r.nsurv[cx], tot) : 0;
  }
  __syncthreads();
  int at = s_base + s_warp[warp];
  int32_t* out = vc ? vsurv + ((size_t)b * 2 + cx) * vcap : surv + ((size_t)b * 2 + cx) * cap;
#pragma unroll
  for (int j = 0; j < kFilterPer; ++j) {
    if (pass[j]) out[at + __popc(bal[j] & ((1u << lane) - 1u))] = sv[j];
    at += __popc(bal[j]);
  }
}

// Ends of the first three queue segments of a row (x, y, z) and its length
// (w).  Segments: [sigma walked CD spellings, or ranges][sigma' verdict
// classes][sigma' walked CD spellings][sigma verdict classes].  The byte
// walks come first: their items are the longest, and starting them early
// keeps them off the end of the kernel.
__device__ __forceinline__ int4 row_queue(const Tables& t, const RowCtx& x) {
  if (x.complete) return make_int4(0, 0, 0, 0);
  const int ed = x.tbl0 >= 0 ? (x.nsurv[0] + kSpan - 1) / kSpan : x.nrange;
  const int ea = ed + ((x.nvs[1] + 31) >> 5);
  const int eb = ea + (x.nsurv[1] + kSpan - 1) / kSpan;
  return make_int4(ed, ea, eb, eb + ((x.nvs[0] + 31) >> 5));
}

// Persistent walk.  Every row owns one work queue of items, in four segments:
// the spellings that continue the pending lexeme under sigma (its table's
// byte-walked list, or its continuing first-byte ranges when the state has no
// table), the verdict classes of the start state's table under sigma' (the
// context of tokens whose first byte ends the pending lexeme), the start
// state's byte-walked spellings under sigma', and the verdict classes of the
// pending lexer state's table under sigma.  Warps start at different rows and drain a
// row's queue item by item; to find work a warp examines 32 rows at once (one
// per lane), from its current row on, and stops when no queue has items left.
// A warp keeps the current row's context (allowed sets, sigma' overlay, stack
// mirror) until it moves to another row.
//
// Verdict-class items: 32 of the records that k_filter kept for the row and
// context, one per lane, each evaluated once against the row's stack; an
// accepted record sets its bit in vcbits (cleared by k_row), which k_pack
// reads back per token id.
// List items (kSpan CD spellings): a spelling is walked only if the class of
// its first stack-dependent emission is selected for the context's allowed
// set (otherwise that emission, and so the spelling, fails) and, for sigma',
// if its first byte ends the pending lexeme; survivors are compacted onto the
// low lanes.  Range items (up to kRangeSpan spellings of one live first-byte
// range; k_row already dropped the first-byte subtrees in which no spelling
// can survive): the range's items interleave, lane j of item i walking
// spelling lo + i + j * (items of the range).  Both kinds share one call of
// walk_bytes, one spelling per lane.
// With COUNT, each lane also counts its work (lexer steps, ACTION and GOTO
// lookups, verdict-class events) in registers and adds the totals to
// work[0..3] when it is done (and the records and spellings it evaluated to
// work[4..5]); the plain instance has no counting code.
template <bool COUNT>
__global__ void __launch_bounds__(kWalkWarps * 32, 2) k_walk(Tables t, RowCtx* __restrict__ ctx,
                                                             const RowRanges* __restrict__ rng, const uint16_t* stacks,
                                                             const int32_t* __restrict__ surv, int cap,
                                                             const uint32_t* __restrict__ A2,
                                                             uint32_t* __restrict__ verd0,
                                                             uint32_t* __restrict__ verd1, uint32_t* __restrict__ vcbits,
                                                             int vcw, const int32_t* __restrict__ vsurv, int vcap,
                                                             int words_v, int B,
                                                             unsigned long long* __restrict__ work) {
  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ uint16_t s_ovl[kWalkWarps][kMaxOvl];
  __shared__ uint16_t s_win[kWalkWarps][kWalkWin];
  __shared__ uint16_t s_lane[kWalkWarps][2 * kLaneOvl * 32];
  __shared__ uint32_t s_A[kWalkWarps][2][4];  // the cached row's A0 and A1
  __shared__ int4 s_seg[kWalkRowsCached];
  __shared__ Tables ts;
  stage_tables(t, ts, smem);
  pdl_wait();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int gw = blockIdx.x * kWalkWarps + warp;
  const int mc = max_chain_of(t);
  const LArr lo{s_lane[warp] + lane, 32}, ls{s_lane[warp] + kLaneOvl * 32 + lane, 32};
  uint32_t cnt[6] = {0u, 0u, 0u, 0u, 0u, 0u};  // the walk's work units, then records and spellings evaluated
  uint32_t* const ctr = COUNT ? cnt : nullptr;
  // queue length and segment ends of every row
  const bool cached = B <= kWalkRowsCached;
  if (cached) {
    for (int i = threadIdx.x; i < B; i += blockDim.x) {
      const int4 e = row_queue(t, ctx[i]);
      s_seg[i] = e;
    }
  }
  __syncthreads();
  int row = gw % B;
  int bound_row = -1;  // first row whose walk hit a bound (its status becomes BOUND)
  int cur = -1;  // row whose context is cached below
  int tbl0 = -1, depth = 0, q = 0, lx = 0, keep1 = 0, m1 = 0, nrng = 0;
  uint32_t pc0 = 0, wc0 = 0;
  const uint16_t* base = stacks;
  for (;;) {
    // next item of the current row; once that queue is drained, of the first
    // row from there on with items left (32 rows examined at once, one per lane)
    int cidx = -1;
    int4 seg = make_int4(0, 0, 0, 0);
    {
      int got = 0;
      const int4 e = cached ? s_seg[row] : row_queue(t, ctx[row]);
      if (lane == 0 && e.w > 0) got = atomicAdd(&ctx[row].work0, 1);
      got = __shfl_sync(0xffffffffu, got, 0);
      if (e.w > 0 && got < e.w) {
        cidx = got;
        seg = e;
      }
    }
    for (int off = 0; off < B && cidx < 0; off += 32) {
      int rr = row + off + lane;
      rr = rr >= B ? rr - B : rr;
      int4 e = make_int4(0, 0, 0, 0);
      bool has = false;
      if (off + lane < B) {
        e = cached ? s_seg[rr] : row_queue(t, ctx[rr]);
        has = e.w > 0 && *((volatile const int32_t*)&ctx[rr].work0) < e.w;
      }
      uint32_t bal = __ballot_sync(0xffffffffu, has);
      while (bal) {  // warp-uniform
        const int l = __ffs(bal) - 1;
        bal &= bal - 1;
        const int rl = __shfl_sync(0xffffffffu, rr, l);
        const int tl = __shfl_sync(0xffffffffu, e.w, l);
        int got = 0;
        if (lane == 0) got = atomicAdd(&ctx[rl].work0, 1);
        got = __shfl_sync(0xffffffffu, got, 0);
        if (got < tl) {
          cidx = got;
          row = rl;
          seg = make_int4(__shfl_sync(0xffffffffu, e.x, l), __shfl_sync(0xffffffffu, e.y, l),
                          __shfl_sync(0xffffffffu, e.z, l), tl);
          break;
        }
      }
    }
    const int ed = seg.x, ea = seg.y, eb = seg.z;
    if (cidx < 0) break;
    RowCtx& r = ctx[row];
    if (cur != row) {
      cur = row;
      tbl0 = r.tbl0;
      depth = r.depth;
      q = r.q;
      lx = r.lx;
      pc0 = r.pc0;
      wc0 = r.wc0;
      keep1 = r.keep1;
      m1 = r.m1;
      nrng = r.nrng;
      __syncwarp();
      if (lane < 4) {
        s_A[warp][0][lane] = r.A0[lane];
        s_A[warp][1][lane] = r.A1[lane];
      }
      for (int i = lane; i < m1 && i < kMaxOvl; i += 32) s_ovl[warp][i] = r.ovl1[i];
      base = stacks + (size_t)row * t.D;
      if (depth <= kWalkWin) {  // mirror the row's stack: reduce chains read its top repeatedly
        for (int i = lane; i < depth; i += 32) s_win[warp][i] = base[i];
        base = s_win[warp];
      }
      __syncwarp();
    }
    // ---- the item: context and source
    const bool c1 = cidx >= ed && cidx < eb;
    const bool is_vc = (cidx >= ed && cidx < ea) || cidx >= eb;
    if (c1 && m1 > kLaneOvl) {  // sigma' overlay larger than a walk lane holds: flag the row
      bound_row = bound_row < 0 ? row : bound_row;
      continue;
    }
    const uint32_t* Ac = s_A[warp][c1 ? 1 : 0];
    const uint32_t* A2row = A2 + ((size_t)row * 2 + (c1 ? 1 : 0)) * t.T1 * 4;
    const int ckeep = c1 ? keep1 : depth, cm = c1 ? m1 : 0;
    const int cq = c1 ? kStart : q, clx = c1 ? 0 : lx;
    const uint32_t cpc = c1 ? t.root_pc : pc0, cwc = c1 ? t.root_wc : wc0;
    if (is_vc) {  // 32 surviving verdict classes of the context's table, one per lane
      const int tb = c1 ? 0 : tbl0;
      const int cxi = c1 ? 1 : 0;
      const int item = c1 ? cidx - ed : cidx - eb;
      const int k = item * 32 + lane;
      int res = 0, v = 0;
      if (k < r.nvs[cxi]) {
        if (COUNT) ++cnt[4];
        v = vsurv[((size_t)row * 2 + cxi) * vcap + k];
        Walker w;
        walker_init(w, lo, ls, kLaneOvl, base, ckeep, s_ovl[warp], cm, cq, clx, cpc, cwc, Ac, A2row, ctr);
        res = eval_record(ts, w, ts.vc_rec + (size_t)(t.vc_off[tb] + v) * kRecLen, mc);
        if (res < 0 && bound_row < 0) bound_row = row;
      }
      if (res > 0) atomicOr(&vcbits[((size_t)row * 2 + cxi) * vcw + (v >> 5)], 1u << (v & 31));
      continue;
    }
    uint32_t* vb = (c1 ? verd1 : verd0) + (size_t)row * words_v;
    const int32_t* list = nullptr;
    int p0, p1, step = 1;
    if (c1 || tbl0 >= 0) {  // survivors of k_filter
      const int n = c1 ? r.nsurv[1] : r.nsurv[0];
      list = surv + ((size_t)row * 2 + (c1 ? 1 : 0)) * cap;
      p0 = (c1 ? cidx - ea : cidx) * kSpan;
      p1 = min(n, p0 + kSpan);
    } else {
      const int c0 = cidx;
      const RowRanges& R = rng[row];
      int a = 0, z = nrng;  // range k with cpre[k] <= c0 < cpre[k+1]
      while (z - a > 1) {
        const int mid = (a + z) >> 1;
        if (R.cpre[mid] <= c0)
          a = mid;
        else
          z = mid;
      }
      // the range's items interleave: item i takes spellings lo + i,
      // lo + i + n, lo + i + 2n, ... (n items), so that runs of costly
      // neighbours (long multi-word continuations of one prefix) spread
      // over many warps instead of lengthening one
      step = R.cpre[a + 1] - R.cpre[a];
      p0 = R.lo[a] + (c0 - R.cpre[a]);
      p1 = R.hi[a];
    }
    // ---- one spelling per lane, one walk call site
    {
      int sp_i = -1;
      bool go = false;
      if (list) {
        const int i = p0 + lane;
        go = i < p1;
        if (go) sp_i = list[i];
      } else {
        sp_i = p0 + lane * step;
        go = sp_i < p1;
      }
      if (go) {
        if (COUNT) ++cnt[5];
        const Spell sp = load_spell(ts, sp_i);
        Walker w;
        walker_init(w, lo, ls, kLaneOvl, base, ckeep, s_ovl[warp], cm, cq, clx, cpc, cwc, Ac, A2row, ctr);
        const int res = walk_bytes(ts, w, sp, mc);
        if (res < 0 && bound_row < 0) bound_row = row;
        if (res > 0)  // the verdict of every id with this spelling, in the mask's layout
          for (int id = t.id_of_spell[sp_i]; id >= 0; id = t.next_alias[id]) atomicOr(&vb[id >> 5], 1u << (id & 31));
      }
    }
  }
  if (lane == 0 && bound_row >= 0) atomicCAS(&ctx[bound_row].status, GRID_ST_OK, GRID_ST_BOUND);
  if (COUNT)
    for (int k = 0; k < 6; ++k)
      if (cnt[k]) atomicAdd(&work[k], (unsigned long long)cnt[k]);
}

// grid = (ceil(W / kPackWords), B), kPackWords threads: thread (b, wi) makes
// mask word wi of row b, the 32 token ids 32 wi .. 32 wi + 31 (the id tables
// are padded to a multiple of 32 ids, so each thread reads its ids' first
// bytes and class codes with 16-byte loads).  Per id: the first byte decides
// the context (it ends the pending lexeme: sigma' and the start state's
// table; otherwise sigma and the pending state's table, or the walk when the
// state has none), the class code indexes that context's class selection (CI,
// always and never in one bit test), and only verdict-class and walked codes
// look further: the verdict-class bits of the row (staged in shared memory
// with its class selections) or the walks' verdict word.  The last block of a
// row writes its status (EMPTY_MASK for a viable row with no bit set).
//
// With APPLY (1 = fp32, 2 = bf16 logits) the thread also masks the logits of
// its 32 ids (Sec. 2 masked decoding, as grid_apply_mask): a 32-byte sector
// whose ids are all rejected is written with -inf without being read, a mixed
// sector is read, blended and written, an accepted sector is not touched.
constexpr int kPackWords = 256;
template <int APPLY, bool CACHE>
__global__ void __launch_bounds__(kPackWords) k_pack(Tables t, RowCtx* __restrict__ ctx, const uint32_t* __restrict__ sel,
                                                     const uint32_t* __restrict__ vcbits, int vcw,
                                                     const uint32_t* __restrict__ verd0,
                                                     const uint32_t* __restrict__ verd1, int words_v,
                                                     uint32_t* __restrict__ mask, int32_t* __restrict__ d_status,
                                                     void* __restrict__ logits, long long stride, int vec_ok,
                                                     CacheDev cache) {
  extern __shared__ __align__(16) uint32_t s_dyn[];  // class selections (2 nselw) | verdict-class bits (2 vcw)
  __shared__ int s_fl, s_tb, s_any, s_hit, s_fill, s_q;
  const int b = blockIdx.y;
  const int wi = blockIdx.x * kPackWords + threadIdx.x;
  const bool have = wi < t.W;
  const int nw = t.nselw;
  const int code_vc = t.ncls + 3, code_walk = t.ncls + 4, code_vc0 = t.ncls + kPackCodes;
  // spec tables only, read before the wait on the walks: which ids have a
  // spelling, the start state's class codes
  uint4 c04[4];
  uint32_t valid = 0u;
  if (have) {
    const uint4* c = reinterpret_cast<const uint4*>(t.cls_by_id) + 4 * wi;
#pragma unroll
    for (int k = 0; k < 4; ++k) c04[k] = c[k];
    valid = t.id_valid[wi];
  }
  pdl_wait();
  const RowCtx& rc = ctx[b];
  if (threadIdx.x == 0) {
    s_tb = rc.tbl0;
    s_fl = (rc.emit_ok ? 1 : 0) | (rc.eos_ok ? 2 : 0) | (rc.complete ? 4 : 0);
    s_any = 0;
    s_hit = CACHE ? rc.chit : -1;
    s_fill = CACHE ? rc.cfill : -1;
    s_q = rc.q;
  }
  // the row's class selections and verdict-class bits, staged alongside its
  // context (a selection k_row did not write is masked off at use)
  {
    for (int i = threadIdx.x; i < 2 * nw; i += kPackWords) s_dyn[i] = sel[(size_t)b * 2 * nw + i];
    const uint32_t* vb = vcbits + (size_t)b * 2 * vcw;
    for (int i = threadIdx.x; i < 2 * vcw; i += kPackWords) s_dyn[2 * nw + i] = vb[i];
  }
  __syncthreads();
  const int fl = s_fl, tb = s_tb, hit = CACHE ? s_hit : -1, fill = CACHE ? s_fill : -1;
  // a context that k_row did not select for (a completed row, sigma' without
  // a forced emission, sigma without a table) selects no class
  const uint32_t v0 = (t.ci_on && !(fl & 4) && tb >= 0) ? 1u : 0u, v1 = (t.ci_on && !(fl & 4) && (fl & 1)) ? 1u : 0u;
  const uint32_t* sel0 = s_dyn;
  const uint32_t* sel1 = s_dyn + nw;
  const uint32_t* vcb0 = s_dyn + 2 * nw;
  const uint32_t* vcb1 = s_dyn + 2 * nw + vcw;
  uint32_t m = 0u;
  if (have && !(fl & 4)) {
    const uint32_t wv0 = verd0[(size_t)b * words_v + wi];
    const uint32_t wv1 = (fl & 1) ? verd1[(size_t)b * words_v + wi] : 0u;
    // a cache hit gives the context-independent bits; only the residue ids
    // (verdict-class and walked) are decided here
    uint32_t todo = valid;
    // bit j: id 32 wi + j's first byte ends the pending lexeme (context sigma')
    const uint32_t killw = t.killw[(size_t)s_q * t.W + wi];
    if (CACHE && hit >= 0) {
      m = cache.ci[(size_t)hit * t.W + wi];
      todo = cache.sel[(size_t)hit * t.W + wi];
    }
    uint32_t ci_bits = 0u, sel_bits = 0u;  // what a filling row stores
    uint4 ct4[4];
    if (tb >= 0 && todo) {
      const uint4* c = reinterpret_cast<const uint4*>(t.cls_by_id + (size_t)tb * t.Vp) + 4 * wi;
#pragma unroll
      for (int k = 0; k < 4; ++k) ct4[k] = c[k];
    }
    const uint32_t c0w[16] = {c04[0].x, c04[0].y, c04[0].z, c04[0].w, c04[1].x, c04[1].y, c04[1].z, c04[1].w,
                              c04[2].x, c04[2].y, c04[2].z, c04[2].w, c04[3].x, c04[3].y, c04[3].z, c04[3].w};
    uint32_t ctw[16];
#pragma unroll
    for (int k = 0; k < 16; ++k) ctw[k] = code_walk | ((uint32_t)code_walk << 16);
    if (tb >= 0 && todo) {
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        ctw[4 * k] = ct4[k].x;
        ctw[4 * k + 1] = ct4[k].y;
        ctw[4 * k + 2] = ct4[k].z;
        ctw[4 * k + 3] = ct4[k].w;
      }
    }
    if (t.vc_inline) {
      // every id takes the same instructions (selects, no branches): its
      // class selection bit, its verdict-class bit and its walked bit are all
      // read (indices clamped into range) and the code picks one, so that the
      // warp's threads never split over the kinds of their ids
      const uint32_t ok1 = (fl & 1) ? 0xFFFFFFFFu : 0u;  // sigma' exists
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const uint32_t cx = (killw >> j) & 1u;
        const int code = (int)(((cx ? c0w[j >> 1] : ctw[j >> 1]) >> ((j & 1) * 16)) & 0xFFFFu);
        const int ci = min(code, code_vc - 1);
        const uint32_t cbit = ((cx ? sel1 : sel0)[ci >> 5] >> (ci & 31)) & (cx ? v1 : v0);
        const int v = max(code - code_vc0, 0);
        const uint32_t vbit = ((cx ? vcb1 : vcb0)[v >> 5] >> (v & 31)) & 1u;
        const uint32_t wbit = ((cx ? wv1 : wv0) >> j) & 1u;
        const bool dep = code >= code_vc;  // verdict class or walked: decided per row
        const bool live = !cx || ok1;      // a context k_row left out rejects its residue ids
        const uint32_t bit = dep ? (live ? (code == code_walk ? wbit : vbit) : 0u) : cbit;
        if (CACHE) {
          if (dep && live)
            sel_bits |= 1u << j;
          else
            ci_bits |= bit << j;
        }
        m |= (bit & (todo >> j)) << j;
      }
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        if (!((todo >> j) & 1u)) continue;
        const int cx = (killw >> j) & 1u;
        const int code = (int)(((cx ? c0w[j >> 1] : ctw[j >> 1]) >> ((j & 1) * 16)) & 0xFFFFu);
        uint32_t bit = 0u;  // codes of verdict classes and walks in a context k_row left out: rejected
        if (code < code_vc) bit = ((cx ? sel1 : sel0)[code >> 5] >> (code & 31)) & (cx ? v1 : v0);
        if (code >= code_vc && (!cx || (fl & 1))) {
          if (code == code_walk) {
            bit = ((cx ? wv1 : wv0) >> j) & 1u;
          } else {  // the verdict class, looked up
            const uint32_t v = t.vc_by_id[(size_t)(cx ? 0 : tb) * t.Vp + 32 * wi + j];
            bit = ((cx ? vcb1 : vcb0)[v >> 5] >> (v & 31)) & 1u;
          }
          if (CACHE) sel_bits |= 1u << j;
        } else if (CACHE) {
          ci_bits |= bit << j;
        }
        m |= bit << j;
      }
    }
    if (CACHE && fill >= 0) {
      cache.ci[(size_t)fill * t.W + wi] = ci_bits;
      cache.sel[(size_t)fill * t.W + wi] = sel_bits;
    }
    const int ej = t.eos - 32 * wi;
    if (ej >= 0 && ej < 32 && (fl & 2)) m |= 1u << ej;  // the EOS gate is stack-dependent: never cached
  }
  if (have) {
    mask[(size_t)b * t.W + wi] = m;
    if (m) s_any = 1;
  }
  if (APPLY && have) {
    using T = typename std::conditional<APPLY == 1, uint32_t, uint16_t>::type;
    constexpr int E = 32 / sizeof(T);  // elements per 32-byte sector
    constexpr int NS = 32 / E;         // sectors per mask word
    constexpr uint32_t sfull = E == 32 ? 0xFFFFFFFFu : (1u << E) - 1u;
    constexpr uint32_t fill = sizeof(T) == 4 ? 0xFF800000u : 0xFF80FF80u;
    T* row = reinterpret_cast<T*>(logits) + (size_t)b * stride;
    const int V = t.V;
    uint32_t v[NS][8];
#pragma unroll
    for (int u = 0; u < NS; ++u) {  // mixed whole sectors: read
      const int e0 = 32 * wi + u * E;
      const uint32_t sb = (m >> (u * E)) & sfull;
      if (vec_ok && e0 + E <= V && sb != 0u && sb != sfull)
        asm volatile("ld.global.v8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                     : "=r"(v[u][0]), "=r"(v[u][1]), "=r"(v[u][2]), "=r"(v[u][3]), "=r"(v[u][4]), "=r"(v[u][5]),
                       "=r"(v[u][6]), "=r"(v[u][7])
                     : "l"(row + e0)
                     : "memory");
    }
#pragma unroll
    for (int u = 0; u < NS; ++u) {  // blend and store
      const int e0 = 32 * wi + u * E;
      const uint32_t sb = (m >> (u * E)) & sfull;
      if (e0 >= V || sb == sfull) continue;
      T* p = row + e0;
      if (vec_ok && e0 + E <= V) {
        uint32_t w[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          if (sizeof(T) == 4) {
            w[k] = ((sb >> k) & 1u) ? v[u][k] : fill;
          } else {
            const uint32_t lo = (sb >> (2 * k)) & 1u, hi = (sb >> (2 * k + 1)) & 1u;
            w[k] = sb == 0u ? fill : (lo ? (v[u][k] & 0xFFFFu) : 0xFF80u) | (hi ? (v[u][k] & 0xFFFF0000u) : 0xFF800000u);
          }
        }
        asm volatile("st.global.v8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"l"(p), "r"(w[0]), "r"(w[1]), "r"(w[2]),
                     "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7])
                     : "memory");
      } else {
        for (int k = 0; k < E && e0 + k < V; ++k)
          if (!((sb >> k) & 1u)) p[k] = (T)fill;
      }
    }
  }
  if (CACHE && fill >= 0) __threadfence();  // the entry's words before its readiness
  __syncthreads();
  // one atomic per block counts the block for its row and carries whether it
  // set a bit; the row's last block writes the status (and marks a cache
  // entry the row filled ready: all blocks have written their words)
  if (threadIdx.x == 0) {
    const unsigned long long old = atomicAdd(&ctx[b].pack_done, 1ull + (s_any ? (1ull << 32) : 0ull));
    if ((uint32_t)old == gridDim.x - 1) {
      int st = atomicAdd(&ctx[b].status, 0);
      if (st == GRID_ST_OK && (old >> 32) == 0ull && !s_any) st = GRID_ST_EMPTY_MASK;
      d_status[b] = st;
      if (CACHE && fill >= 0) {
        __threadfence();
        atomicExch(cache.hdr + (size_t)fill * 16, 2u);
      }
    }
  }
}

// One warp per row (advance_warp).
__global__ void __launch_bounds__(kAdvWarps * 32) k_advance(Tables t, DevConfigs cin, DevConfigs cout,
                                                             const int32_t* __restrict__ tokens, int n_steps,
                                                             int32_t* __restrict__ d_status, int B, int copy) {
  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ Tables ts;
  __shared__ __align__(16) uint16_t s_stk[kAdvWarps][kStackWin];
  __shared__ uint16_t s_lo[kAdvWarps][kMaxOvl], s_ls[kAdvWarps][kMaxOvl];
  stage_tables(t, ts, smem);
  pdl_wait();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int b = blockIdx.x * kAdvWarps + warp;
  if (b >= B) return;
  AdvOut out;
  advance_warp(t, ts, cin, cout, tokens, n_steps, d_status, b, copy, lane, s_stk[warp], LArr{s_lo[warp], 1},
               LArr{s_ls[warp], 1}, out);
}

// In-place -inf fill, grid = (blocks per row, B): threads stride over a row's
// 32-byte sectors of logits (8 fp32 or 16 bf16), one 256-bit access per
// sector, so that every store writes a whole sector and a warp's store covers
// 1 KB of contiguous bytes (few, long-lived blocks: block scheduling, not
// memory, bounds a grid of one short block per 256 sectors).  A sector whose
// tokens are all rejected is written without being read; a mixed sector is
// read, blended and written; a fully accepted sector is not touched.  Each
// thread takes kApplyBatch sectors at a time: their mask words loaded
// together, then the rejected sectors stored (they wait on nothing), then the
// mixed sectors read together and stored, so that a thread waits on two
// rounds of loads per batch instead of two per sector.
// Rows whose sectors are not 32-byte aligned, and the ragged end of a row,
// are done element by element.
constexpr int kApplyBatch = 4;
template <typename T>
__global__ void __launch_bounds__(256) k_apply(const uint32_t* __restrict__ mask, T* __restrict__ logits, int B,
                                               int V, int W, long long stride, int vec_ok) {
  constexpr int E = 32 / sizeof(T);  // elements per sector
  constexpr uint32_t sfull = E == 32 ? 0xFFFFFFFFu : (1u << E) - 1u;
  constexpr uint32_t fill = sizeof(T) == 4 ? 0xFF800000u : 0xFF80FF80u;  // -inf in every element of a word
  pdl_wait();
  const int b = blockIdx.y;
  const int nsec = (V + E - 1) / E;
  const int step = gridDim.x * blockDim.x;
  T* row = logits + (size_t)b * stride;
  for (int s0 = blockIdx.x * blockDim.x + threadIdx.x; s0 < nsec; s0 += kApplyBatch * step) {
    uint32_t sb[kApplyBatch];
#pragma unroll
    for (int u = 0; u < kApplyBatch; ++u) {  // the sectors' accept bits
      const int e0 = (s0 + u * step) * E;
      sb[u] = s0 + u * step < nsec ? (mask[(size_t)b * W + (e0 >> 5)] >> (e0 & 31)) & sfull : sfull;
    }
#pragma unroll
    for (int u = 0; u < kApplyBatch; ++u) {  // rejected whole sectors first: written without a read
      const int e0 = (s0 + u * step) * E;
      if (vec_ok && s0 + u * step < nsec && e0 + E <= V && sb[u] == 0u)
        asm volatile("st.global.v8.b32 [%0], {%1,%1,%1,%1,%1,%1,%1,%1};" ::"l"(row + e0), "r"(fill) : "memory");
    }
    uint32_t v[kApplyBatch][8];
#pragma unroll
    for (int u = 0; u < kApplyBatch; ++u) {  // mixed whole sectors: read
      const int e0 = (s0 + u * step) * E;
      if (vec_ok && s0 + u * step < nsec && e0 + E <= V && sb[u] != 0u && sb[u] != sfull)
        asm volatile("ld.global.v8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                     : "=r"(v[u][0]), "=r"(v[u][1]), "=r"(v[u][2]), "=r"(v[u][3]), "=r"(v[u][4]), "=r"(v[u][5]),
                       "=r"(v[u][6]), "=r"(v[u][7])
                     : "l"(row + e0)
                     : "memory");
    }
#pragma unroll
    for (int u = 0; u < kApplyBatch; ++u) {  // mixed sectors: blend and store; partial sectors one by one
      const int e0 = (s0 + u * step) * E;
      if (s0 + u * step >= nsec || sb[u] == sfull) continue;
      T* p = row + e0;
      const int n = min(E, V - e0);
      if (vec_ok && n == E) {
        if (sb[u] == 0u) continue;  // written above
        uint32_t w[8];
        if (sizeof(T) == 4) {
#pragma unroll
          for (int k = 0; k < 8; ++k) w[k] = ((sb[u] >> k) & 1u) ? v[u][k] : fill;
        } else {
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint32_t lo = (sb[u] >> (2 * k)) & 1u, hi = (sb[u] >> (2 * k + 1)) & 1u;
            w[k] = (lo ? (v[u][k] & 0xFFFFu) : 0xFF80u) | (hi ? (v[u][k] & 0xFFFF0000u) : 0xFF800000u);
          }
        }
        asm volatile("st.global.v8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"l"(p), "r"(w[0]), "r"(w[1]), "r"(w[2]),
                     "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7])
                     : "memory");
      } else {
        for (int k = 0; k < n; ++k) {
          if (!((sb[u] >> k) & 1u)) {
            if (sizeof(T) == 4)
              reinterpret_cast<uint32_t*>(p)[k] = 0xFF800000u;
            else
              reinterpret_cast<uint16_t*>(p)[k] = 0xFF80u;
          }
        }
      }
    }
  }
}

// Launch with programmatic stream serialization: the kernel may begin (stage
// its tables) while the previous kernel in the stream drains; it waits for
// that kernel's results with griddepcontrol.wait (pdl_wait).
template <typename... KArgs, typename... Args>
static cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                              Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

size_t align16(size_t x) { return (x + 15) & ~size_t(15); }

}  // namespace
}  // namespace grid

using namespace grid;

int grid::g_sms = 152;  // SM count of the current device, set by grid_specialize

// The dynamic shared-memory cap is a per-function attribute shared by every
// spec in the process, so it is raised once to the largest staged block
// allowed instead of to this spec's size.
static int set_smem_limits() {
  const int dyn = kMaxStage;
  GRID_CUDA(cudaFuncSetAttribute(k_classify, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn));
  GRID_CUDA(cudaFuncSetAttribute(k_events, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn));
  // k_pack: one row's class selections and verdict-class bits, two contexts
  GRID_CUDA(cudaFuncSetAttribute(k_pack<0, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn));
  GRID_CUDA(cudaFuncSetAttribute(k_pack<1, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn));
  GRID_CUDA(cudaFuncSetAttribute(k_pack<2, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn));
  GRID_CUDA(cudaFuncSetAttribute(k_pack<0, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn));
  GRID_CUDA(cudaFuncSetAttribute(k_pack<1, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn));
  GRID_CUDA(cudaFuncSetAttribute(k_pack<2, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn));
  GRID_CUDA(cudaFuncSetAttribute(k_row<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn));
  GRID_CUDA(cudaFuncSetAttribute(k_row<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn));
  GRID_CUDA(cudaFuncSetAttribute(k_walk<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn));
  GRID_CUDA(cudaFuncSetAttribute(k_walk<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn));
  GRID_CUDA(cudaFuncSetAttribute(k_advance, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn));
  return GRID_OK;
}

extern "C" int grid_specialize(const grid_grammar* g, const grid_vocab* v, void* stream, grid_spec** out) {
  if (!g || !v || !out) return set_error(GRID_E_INVALID_ARG, "grid_specialize: bad arguments");
  *out = nullptr;
  const HostGrammar& h = g->h;
  const HostVocab& hv = v->h;
  cudaStream_t st = (cudaStream_t)stream;
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
  t.ign = Bits4{h.ignored[0], h.ignored[1], h.ignored[2], h.ignored[3]};
  t.cm = Bits4{h.catmask[0], h.catmask[1], h.catmask[2], h.catmask[3]};
  for (int c = 0; c < h.n_cat; ++c) t.cat_term[c] = h.cat_term[c];
  auto fail = [&](int rc) {
    s->mem.release();
    delete s;
    return rc;
  };
  // per LALR state: the terminals that shift, and the terminals grouped by
  // the production they reduce by (for simulating a set of terminals at once)
  std::vector<uint32_t> shift_mask((size_t)h.S * 4, 0u), red_mask;
  // reduce actions carry their production's length and left-hand side
  // (-(1 + (plen << 10 | lhs))), so that a reduce step needs no second lookup
  int max_plen = 0;
  for (int pr = 0; pr < h.P; ++pr) max_plen = std::max(max_plen, (int)h.plen[pr]);
  if (h.NNT >= 1024 || max_plen >= 32)
    return fail(set_error(GRID_E_TOO_LARGE, "grammar exceeds the packed reduce encoding (1024 nonterminals, "
                                            "right-hand sides of 31 symbols)"));
  std::vector<int16_t> action16(h.action.size());
  for (size_t i = 0; i < h.action.size(); ++i) {
    const int a = h.action[i];
    action16[i] = a >= 0 ? (int16_t)a : (int16_t)(-(1 + ((h.plen[-a - 1] << 10) | h.plhs[-a - 1])));
  }
  std::vector<uint32_t> red_off(h.S + 1, 0);
  std::vector<uint16_t> red_p;
  for (int st = 0; st < h.S; ++st) {
    std::vector<std::pair<int, std::array<uint32_t, 4>>> groups;
    for (int tau = 0; tau < h.T1; ++tau) {
      const int a = h.action[(size_t)st * h.T1 + tau];
      if (a > 0 && a != kAccept) {
        shift_mask[(size_t)st * 4 + (tau >> 5)] |= 1u << (tau & 31);
      } else if (a < 0) {
        const int pr = -a - 1;
        auto it = std::find_if(groups.begin(), groups.end(), [&](const auto& g) { return g.first == pr; });
        if (it == groups.end()) {
          groups.push_back({pr, {0u, 0u, 0u, 0u}});
          it = groups.end() - 1;
        }
        it->second[tau >> 5] |= 1u << (tau & 31);
      }
    }
    for (const auto& g : groups) {
      red_p.push_back((uint16_t)((h.plen[g.first] << 10) | h.plhs[g.first]));
      for (int w = 0; w < 4; ++w) red_mask.push_back(g.second[w]);
    }
    red_off[st + 1] = (uint32_t)red_p.size();
  }
  // staged block: byte classes, DFA, acc/live, ACTION, GOTO, production
  // tables, shift masks and reduce groups
  constexpr int kSec = 12;
  std::vector<size_t> off(kSec + 1, 0);
  const size_t sizes[kSec] = {256, h.next.size() * 2, h.acc.size() * 4, h.live.size() * 4, h.action.size() * 2,
                              h.go.size() * 2, h.plen.size(), h.plhs.size() * 2, shift_mask.size() * 4,
                              red_off.size() * 4, red_p.size() * 2, red_mask.size() * 4};
  const void* srcs[kSec] = {h.byte_class, h.next.data(), h.acc.data(), h.live.data(), action16.data(),
                            h.go.data(), h.plen.data(), h.plhs.data(), shift_mask.data(), red_off.data(),
                            red_p.data(), red_mask.data()};
  for (int k = 0; k < kSec; ++k) off[k + 1] = align16(off[k] + sizes[k]);
  std::vector<uint8_t> blob(off[kSec], 0);
  for (int k = 0; k < kSec; ++k)
    if (sizes[k]) std::memcpy(blob.data() + off[k], srcs[k], sizes[k]);
  const uint8_t* dblob = nullptr;
  int rc = s->mem.upload(blob, &dblob);
  if (rc) return fail(rc);
  t.blob = dblob;
  t.blob_bytes = off[kSec] <= (size_t)kMaxStage ? (int)off[kSec] : 0;
  t.byte_class = dblob + off[0];
  t.next = reinterpret_cast<const uint16_t*>(dblob + off[1]);
  t.acc = reinterpret_cast<const uint32_t*>(dblob + off[2]);
  t.live = reinterpret_cast<const uint32_t*>(dblob + off[3]);
  t.action = reinterpret_cast<const int16_t*>(dblob + off[4]);
  t.go = reinterpret_cast<const uint16_t*>(dblob + off[5]);
  t.plen = dblob + off[6];
  t.plhs = reinterpret_cast<const uint16_t*>(dblob + off[7]);
  t.shift_mask = reinterpret_cast<const uint32_t*>(dblob + off[8]);
  t.red_off = reinterpret_cast<const uint32_t*>(dblob + off[9]);
  t.red_p = reinterpret_cast<const uint16_t*>(dblob + off[10]);
  t.red_mask = reinterpret_cast<const uint32_t*>(dblob + off[11]);
  Arena& a = s->mem;
  {
    // identifier-trie edges -> open-addressing hash (load factor <= 1/2)
    const size_t edges = h.lx_cbyte.size();
    int bits = 4;
    while ((size_t(1) << bits) < 2 * edges + 2) ++bits;
    std::vector<uint32_t> hv4((size_t(4) << bits), 0u);
    for (size_t i = 0; i < (size_t(1) << bits); ++i) hv4[4 * i] = kHashEmpty;
    const uint32_t mask = (1u << bits) - 1u;
    for (int n = 0; n < h.LN; ++n)
      for (int e = h.lx_cstart[n]; e < h.lx_cstart[n + 1]; ++e) {
        const uint32_t key = (uint32_t)n * 256u + h.lx_cbyte[e];
        uint32_t hh = (key * 0x9E3779B1u) >> (32 - bits);
        while (hv4[4 * hh] != kHashEmpty) hh = (hh + 1u) & mask;
        const int child = h.lx_cnode[e];
        hv4[4 * hh] = key;
        hv4[4 * hh + 1] = (uint32_t)child;
        hv4[4 * hh + 2] = h.lx_pcats[child];
        hv4[4 * hh + 3] = h.lx_wcats[child];
      }
    const uint32_t* dh = nullptr;
    if ((rc = a.upload(hv4, &dh))) return fail(rc);
    t.lx_hash = reinterpret_cast<const uint4*>(dh);
    t.lx_hmask = mask;
    t.lx_hshift = 32 - bits;
    t.root_pc = h.LN > 0 ? h.lx_pcats[0] : 0u;
    t.root_wc = h.LN > 0 ? h.lx_wcats[0] : 0u;
  }
  // id-indexed tables are padded to Vp ids (a multiple of 32), so that the
  // ids of one mask word are read with 16-byte loads
  t.Vp = (hv.V + 31) & ~31;
  std::vector<int32_t> spell_of_id_p(hv.spell_of_id);
  spell_of_id_p.resize(t.Vp, -1);
  {
    std::vector<uint32_t> valid(t.W, 0u);  // ids with a spelling: not EOS, special or padding
    for (int id = 0; id < hv.V; ++id)
      if (spell_of_id_p[id] >= 0) valid[id >> 5] |= 1u << (id & 31);
    int rcv = s->mem.upload(valid, &t.id_valid);
    if (rcv) return fail(rcv);
  }
  // the ids of each spelling (aliases), for the walks' id-indexed verdicts
  std::vector<int32_t> id_of_spell(std::max(1, t.NS), -1), next_alias(t.Vp, -1);
  for (int id = t.Vp - 1; id >= 0; --id) {
    const int sp = spell_of_id_p[id];
    if (sp < 0) continue;
    next_alias[id] = id_of_spell[sp];
    id_of_spell[sp] = id;
  }
  if ((rc = a.upload(h.lx_cstart, &t.lx_cstart)) || (rc = a.upload(h.lx_cbyte, &t.lx_cbyte)) ||
      (rc = a.upload(h.lx_cnode, &t.lx_cnode)) || (rc = a.upload(h.lx_pcats, &t.lx_pcats)) ||
      (rc = a.upload(h.lx_wcats, &t.lx_wcats)) || (rc = a.upload(hv.spell_off, &t.spell_off)) ||
      (rc = a.upload(hv.spell_bytes, &t.spell_bytes)) ||
      (rc = a.upload(spell_of_id_p, &t.spell_of_id)) || (rc = a.upload(id_of_spell, &t.id_of_spell)) ||
      (rc = a.upload(next_alias, &t.next_alias)) || (rc = a.upload(hv.first_of_byte, &t.first_of_byte)))
    return fail(rc);
  {
    std::vector<uint32_t> s16((size_t)hv.NS * 4, 0u);
    for (int sp = 0; sp < hv.NS; ++sp) {
      const int off = hv.spell_off[sp], len = std::min(16, hv.spell_off[sp + 1] - off);
      std::memcpy(reinterpret_cast<uint8_t*>(s16.data() + (size_t)sp * 4), hv.spell_bytes.data() + off, len);
    }
    const uint32_t* d16 = nullptr;
    if ((rc = a.upload(s16, &d16))) return fail(rc);
    t.spell16 = reinterpret_cast<const uint4*>(d16);
  }
  // precomputed lexer states: the start state and every state at which no
  // lexicon category is live (there the lexicon node cannot matter)
  std::vector<int32_t> tq{kStart};
  std::vector<int16_t> tbl_of_q(h.Q, -1);
  tbl_of_q[kStart] = 0;
  const long ncls = (long)(2 * h.Q) << h.n_cat;
  t.ci_on = ncls < (long)kClsFirstCode ? 1 : 0;
  if (t.ci_on) {
    for (int q = 2; q < h.Q; ++q) {
      bool catlive = false;
      for (int w = 0; w < 4; ++w)
        if (h.live[q * 4 + w] & h.catmask[w]) catlive = true;
      if (!catlive && tq.size() < 4096) {
        tbl_of_q[q] = (int16_t)tq.size();
        tq.push_back(q);
      }
    }
  }
  t.n_tbl = (int)tq.size();
  t.ncls = t.ci_on ? (int)ncls : 0;
  t.nselw = (t.ncls + kPackCodes + 31) / 32;
  if ((rc = a.upload(tq, &t.tbl_q)) || (rc = a.upload(tbl_of_q, &t.tbl_of_q)) || (rc = a.upload(h.acc_sym, &t.acc_sym)))
    return fail(rc);
  {
    Blake2b fb;
    fb.init(16);
    fb.update("GRIDspec", 8);
    fb.update(h.fingerprint, 16);
    fb.update(hv.fingerprint, 16);
    fb.final(s->fingerprint);
  }
  if ((rc = set_smem_limits())) return fail(rc);
  int dev = 0;
  cudaGetDevice(&dev);
  s->device = dev;
  cudaDeviceGetAttribute(&s->sms, cudaDevAttrMultiProcessorCount, dev);
  g_sms = s->sms;
  // CI classification on the device (temporaries live in `tmp`)
  Arena tmp;
  auto fail_tmp = [&](int code) {
    tmp.release();
    return fail(code);
  };
  uint16_t* cls_sp = nullptr;
  uint16_t* key_sp = nullptr;
  int32_t* counts_d = nullptr;
  uint16_t* cls_by_id = nullptr;
  uint32_t* vc_by_id = nullptr;
  uint8_t* fb = nullptr;
  if ((rc = tmp.alloc((size_t)t.n_tbl * t.NS * 2, (void**)&cls_sp)) ||
      (rc = tmp.alloc((size_t)t.n_tbl * t.NS * 2, (void**)&key_sp)) ||
      (rc = tmp.alloc((size_t)t.n_tbl * 8, (void**)&counts_d)) ||
      (rc = a.alloc((size_t)t.n_tbl * t.Vp * 2, (void**)&cls_by_id)) || (rc = a.alloc((size_t)t.Vp, (void**)&fb)))
    return fail_tmp(rc);
  t.cls_by_id = cls_by_id;
  t.first_byte_by_id = fb;
  GRID_CUDA(cudaMemsetAsync(counts_d, 0, (size_t)t.n_tbl * 8, st));
  const dim3 cgrid(std::max(1, std::min((t.NS + 255) / 256, 4 * s->sms)), t.n_tbl);
  k_classify<<<cgrid, 256, t.blob_bytes, st>>>(t, cls_sp, key_sp, counts_d);
  std::vector<int32_t> counts2(2 * t.n_tbl);
  GRID_CUDA(cudaMemcpyAsync(counts2.data(), counts_d, t.n_tbl * 8, cudaMemcpyDeviceToHost, st));
  GRID_CUDA(cudaStreamSynchronize(st));
  std::vector<int32_t> counts(t.n_tbl), cdoff(t.n_tbl + 1, 0), vcbase(t.n_tbl + 1, 0);
  for (int k = 0; k < t.n_tbl; ++k) {
    counts[k] = counts2[2 * k];
    cdoff[k + 1] = cdoff[k] + counts2[2 * k];
    vcbase[k + 1] = vcbase[k] + counts2[2 * k + 1];
  }
  // CD spellings walked byte by byte (more than kMaxEv events)
  int32_t* cd_list = nullptr;
  uint16_t* cd_key = nullptr;
  if ((rc = a.upload(cdoff, &t.cd_off)) || (rc = a.alloc((size_t)cdoff.back() * 4, (void**)&cd_list)) ||
      (rc = a.alloc((size_t)cdoff.back() * 2, (void**)&cd_key)))
    return fail_tmp(rc);
  t.cd_list = cd_list;
  t.cd_key = cd_key;
  k_compact<<<t.n_tbl, 1024, 0, st>>>(cls_sp, key_sp, t.NS, t.cd_off, cd_list, cd_key);
  // event records of the verdict-class spellings -> distinct records per table
  const int nslot = vcbase.back();
  const int32_t* vcbase_d = nullptr;
  int32_t *fill = nullptr, *slot_tbl = nullptr, *slot_sp = nullptr;
  uint16_t* slot_rec = nullptr;
  uint32_t* vc_sp = nullptr;
  if ((rc = tmp.upload(vcbase, &vcbase_d)) || (rc = tmp.alloc((size_t)t.n_tbl * 4, (void**)&fill)) ||
      (rc = tmp.alloc((size_t)nslot * 4, (void**)&slot_tbl)) || (rc = tmp.alloc((size_t)nslot * 4, (void**)&slot_sp)) ||
      (rc = tmp.alloc((size_t)nslot * kRecLen * 2, (void**)&slot_rec)) ||
      (rc = tmp.alloc((size_t)t.n_tbl * t.NS * 4, (void**)&vc_sp)))
    return fail_tmp(rc);
  GRID_CUDA(cudaMemsetAsync(fill, 0, (size_t)t.n_tbl * 4, st));
  if (nslot > 0) k_events<<<cgrid, 256, t.blob_bytes, st>>>(t, cls_sp, vcbase_d, fill, slot_tbl, slot_sp, slot_rec);
  std::vector<int32_t> h_tbl(nslot);
  std::vector<uint16_t> h_rec((size_t)nslot * kRecLen);
  if (nslot > 0) {
    GRID_CUDA(cudaMemcpyAsync(h_tbl.data(), slot_tbl, (size_t)nslot * 4, cudaMemcpyDeviceToHost, st));
    GRID_CUDA(cudaMemcpyAsync(h_rec.data(), slot_rec, (size_t)nslot * kRecLen * 2, cudaMemcpyDeviceToHost, st));
  }
  GRID_CUDA(cudaStreamSynchronize(st));
  // class ids with equal terminal sets are interchangeable in a record:
  // rewrite each to the smallest such id before deduplication
  std::vector<uint16_t> canon(std::max(1, t.ncls));
  if (t.ncls > 0) {
    // terminal set of every class id, and per terminal the mask of the
    // classes whose set holds it (the class selection ORs these)
    uint4* sets_d = nullptr;
    if ((rc = a.alloc((size_t)t.ncls * 16, (void**)&sets_d))) return fail_tmp(rc);
    k_class_sets<<<(t.ncls + 255) / 256, 256, 0, st>>>(t, sets_d);
    std::vector<uint4> sets(t.ncls);
    GRID_CUDA(cudaMemcpyAsync(sets.data(), sets_d, (size_t)t.ncls * 16, cudaMemcpyDeviceToHost, st));
    GRID_CUDA(cudaStreamSynchronize(st));
    t.cls_sets = reinterpret_cast<const uint32_t*>(sets_d);
    std::vector<uint32_t> cmask((size_t)t.T1 * t.nselw, 0u);
    for (int c = 0; c < t.ncls; ++c) {
      const uint32_t wv[4] = {sets[c].x, sets[c].y, sets[c].z, sets[c].w};
      for (int tau = 0; tau < t.T1; ++tau)
        if ((wv[tau >> 5] >> (tau & 31)) & 1u) cmask[(size_t)tau * t.nselw + (c >> 5)] |= 1u << (c & 31);
    }
    if ((rc = a.upload(cmask, &t.cls_mask))) return fail_tmp(rc);
    std::unordered_map<std::string, uint16_t> first;
    for (int c = 0; c < t.ncls; ++c) {
      std::string key(reinterpret_cast<const char*>(&sets[c]), 16);
      canon[c] = first.emplace(key, (uint16_t)c).first->second;
    }
    for (int i = 0; i < nslot; ++i) {
      uint16_t* r = h_rec.data() + (size_t)i * kRecLen;
      if (r[1] < t.ncls) r[1] = canon[r[1]];
      for (int e = 0; e < r[0]; ++e)
        if (r[2 + e] < t.ncls) r[2 + e] = canon[r[2 + e]];
    }
  }
  std::vector<int32_t> vcoff(t.n_tbl + 1, 0), h_vc(nslot);
  std::vector<uint16_t> recs;
  {
    std::vector<std::unordered_map<std::string, int32_t>> seen(t.n_tbl);
    std::vector<std::vector<uint16_t>> per(t.n_tbl);
    for (int i = 0; i < nslot; ++i) {
      const int k = h_tbl[i];
      const uint16_t* r = h_rec.data() + (size_t)i * kRecLen;
      std::string key(reinterpret_cast<const char*>(r), kRecLen * 2);
      auto it = seen[k].find(key);
      if (it == seen[k].end()) {
        it = seen[k].emplace(key, (int32_t)(per[k].size() / kRecLen)).first;
        per[k].insert(per[k].end(), r, r + kRecLen);
      }
      h_vc[i] = it->second;
    }
    // order each table's records by their event sequences (then the event
    // count and the final class): a walk item evaluates 32 neighbouring
    // records on one row's stack, and records that share their first events
    // take the same path through them, so the warp's lanes stay together
    for (int k = 0; k < t.n_tbl; ++k) {
      const int n = (int)(per[k].size() / kRecLen);
      std::vector<int32_t> ord(n), pos(n);
      for (int i = 0; i < n; ++i) ord[i] = i;
      const uint16_t* R = per[k].data();
      std::sort(ord.begin(), ord.end(), [&](int x, int y) {
        const uint16_t* a = R + (size_t)x * kRecLen;
        const uint16_t* b = R + (size_t)y * kRecLen;
        const int m = std::min<int>(a[0], b[0]);
        for (int e = 0; e < m; ++e)
          if (a[2 + e] != b[2 + e]) return a[2 + e] < b[2 + e];
        if (a[0] != b[0]) return a[0] < b[0];
        if (a[1] != b[1]) return a[1] < b[1];
        return x < y;
      });
      std::vector<uint16_t> sorted(per[k].size());
      for (int i = 0; i < n; ++i) {
        pos[ord[i]] = i;
        std::copy(R + (size_t)ord[i] * kRecLen, R + (size_t)(ord[i] + 1) * kRecLen, sorted.begin() + (size_t)i * kRecLen);
      }
      per[k].swap(sorted);
      for (auto& kv : seen[k]) kv.second = pos[kv.second];
    }
    for (int i = 0; i < nslot; ++i) {
      const uint16_t* r = h_rec.data() + (size_t)i * kRecLen;
      h_vc[i] = seen[h_tbl[i]].at(std::string(reinterpret_cast<const char*>(r), kRecLen * 2));
    }
    for (int k = 0; k < t.n_tbl; ++k) {
      vcoff[k + 1] = vcoff[k] + (int32_t)(per[k].size() / kRecLen);
      recs.insert(recs.end(), per[k].begin(), per[k].end());
      s->vcw = std::max(s->vcw, (int)((per[k].size() / kRecLen + 31) / 32));
    }
  }
  std::vector<uint16_t> first(recs.size() / kRecLen);
  for (size_t i = 0; i < first.size(); ++i) first[i] = recs[i * kRecLen + 2];
  for (int k = 0; k < t.n_tbl; ++k) s->max_vc = std::max(s->max_vc, vcoff[k + 1] - vcoff[k]);
  const int32_t* slot_vc_c = nullptr;
  if ((rc = a.upload(vcoff, &t.vc_off)) || (rc = a.upload(recs, &t.vc_rec)) || (rc = a.upload(first, &t.vc_first)) ||
      (rc = tmp.upload(h_vc, &slot_vc_c)))
    return fail_tmp(rc);
  if (nslot > 0)
    k_scatter_vc<<<(nslot + 255) / 256, 256, 0, st>>>(slot_tbl, slot_sp, slot_vc_c, nslot, t.NS, vc_sp);
  // verdict-class indices ride in the 16-bit class codes when they fit;
  // otherwise k_pack looks them up per id
  t.vc_inline = t.ncls + kPackCodes + s->max_vc <= 0xFFFF ? 1 : 0;
  if (!t.vc_inline && (rc = a.alloc((size_t)t.n_tbl * t.Vp * 4, (void**)&vc_by_id))) return fail_tmp(rc);
  t.vc_by_id = vc_by_id;
  k_permute<<<(t.Vp + 255) / 256, 256, 0, st>>>(t, cls_sp, vc_sp, cls_by_id, vc_by_id, fb);
  {
    uint32_t* killw = nullptr;
    if ((rc = a.alloc((size_t)t.Q * t.W * 4, (void**)&killw))) return fail_tmp(rc);
    k_killw<<<dim3((t.W + 255) / 256, t.Q), 256, 0, st>>>(t, killw);
    t.killw = killw;
  }
  GRID_CUDA(cudaGetLastError());
  GRID_CUDA(cudaStreamSynchronize(st));
  tmp.release();
  s->n_vc = vcoff.back();
  if ((size_t)(2 * std::max(1, t.nselw) + 2 * std::max(1, s->vcw)) * 4 > (size_t)kMaxStage)
    return fail(set_error(GRID_E_TOO_LARGE, "grid_specialize: the class selections and verdict-class bits of one "
                                            "row exceed the packing kernel's shared memory"));
  s->n1 = (counts[0] + kSpan - 1) / kSpan;
  s->max_cd = *std::max_element(counts.begin(), counts.end());
  int per_sm = 0;
  GRID_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_walk<false>, kWalkWarps * 32, t.blob_bytes));
  s->walk_blocks = std::max(1, per_sm) * s->sms;
  if ((rc = build_reserve_tables(s))) return fail(rc);
  *out = s;
  return GRID_OK;
}

extern "C" int grid_spec_info(const grid_spec* s, int64_t out[8]) {
  if (!s || !out) return set_error(GRID_E_INVALID_ARG, "grid_spec_info: bad arguments");
  const Tables& t = s->t;
  std::vector<int32_t> off(t.n_tbl + 1);
  GRID_CUDA(cudaMemcpy(off.data(), t.cd_off, (t.n_tbl + 1) * 4, cudaMemcpyDeviceToHost));
  out[0] = t.n_tbl;
  out[1] = t.ncls;
  out[2] = off[1] - off[0];
  out[3] = off[t.n_tbl];
  out[4] = t.blob_bytes;
  out[5] = s->n_vc;
  out[6] = (t.ci_on ? 1 : 0) | (t.vc_inline ? 2 : 0);
  out[7] = t.NS;
  return GRID_OK;
}

extern "C" void grid_spec_free(grid_spec* s) {
  if (!s) return;
  s->mem.release();
  delete s;
}

extern "C" int grid_configs_create(const grid_spec* s, int32_t B, grid_configs** out) {
  if (!s || !out || B <= 0) return set_error(GRID_E_INVALID_ARG, "grid_configs_create: bad arguments");
  if (B > kMaxRows)
    return set_error(GRID_E_TOO_LARGE, "grid_configs_create: more than " + std::to_string(kMaxRows) + " rows");
  *out = nullptr;
  auto* c = new grid_configs();
  c->B = B;
  c->D = s->t.D;
  c->words_v = s->t.W;
  c->cap = std::max(1, s->max_cd);
  c->vcap = std::max(1, s->max_vc);
  Arena& a = c->mem;
  int rc;
  if ((rc = a.alloc((size_t)B * c->D * sizeof(uint16_t), (void**)&c->c.stack)) ||
      (rc = a.alloc(B * 4, (void**)&c->c.depth)) || (rc = a.alloc(B * 4, (void**)&c->c.q)) ||
      (rc = a.alloc(B * 4, (void**)&c->c.lx)) || (rc = a.alloc(B * 4, (void**)&c->c.flags)) ||
      (rc = a.alloc(B * sizeof(RowCtx), (void**)&c->ctx)) ||
      (rc = a.alloc(B * sizeof(RowRanges), (void**)&c->rng)) ||
      (rc = a.alloc((size_t)B * 2 * std::max(1, s->t.nselw) * 4, (void**)&c->sel)) ||
      (rc = a.alloc((size_t)B * c->words_v * 4, (void**)&c->verd0)) ||
      (rc = a.alloc((size_t)B * c->words_v * 4, (void**)&c->verd1)) ||
      (rc = a.alloc((size_t)B * 2 * s->t.T1 * 16, (void**)&c->A2)) ||
      (rc = a.alloc((size_t)B * 2 * std::max(1, s->vcw) * 4, (void**)&c->vcbits)) ||
      (rc = a.alloc((size_t)B * 2 * std::max(1, s->max_cd) * 4, (void**)&c->surv)) ||
      (rc = a.alloc((size_t)B * 2 * c->vcap * 4, (void**)&c->vsurv)) ||
      (rc = a.alloc((size_t)B * 4 * 4, (void**)&c->aux)) ||
      (rc = a.alloc((size_t)B * reserve_scratch_bytes(s), (void**)&c->rscratch))) {
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
  c->mem.release();
  delete c;
}

extern "C" int grid_configs_reset(const grid_spec* s, grid_configs* c, void* stream) {
  if (!s || !c) return set_error(GRID_E_INVALID_ARG, "grid_configs_reset: bad arguments");
  k_reset<<<(c->B + 127) / 128, 128, 0, (cudaStream_t)stream>>>(c->c, c->B, c->D);
  GRID_CUDA(cudaGetLastError());
  return audit_reset(s, c, (cudaStream_t)stream);  // a fresh chain for every row, when audit is on
}

int grid::launch_advance(const grid_spec* s, const DevConfigs& in, const DevConfigs& out, int B,
                         const int32_t* d_tokens, int32_t n_steps, int32_t* d_status, int copy, cudaStream_t st) {
  GRID_CUDA(launch_pdl(k_advance, dim3((B + kAdvWarps - 1) / kAdvWarps), dim3(kAdvWarps * 32), s->t.blob_bytes, st,
                       s->t, in, out, d_tokens, n_steps, d_status, B, copy));
  GRID_CUDA(cudaGetLastError());
  return GRID_OK;
}

extern "C" int grid_advance(const grid_spec* s, const grid_configs* in, grid_configs* out,
                            const int32_t* d_tokens, int32_t n_steps, int32_t* d_status, void* stream) {
  if (!s || !in || !out || !d_tokens || !d_status || n_steps < 0 || in->B != out->B || in->D != out->D)
    return set_error(GRID_E_INVALID_ARG, "grid_advance: bad arguments");
  if ((in->c.hs != nullptr) != (out->c.hs != nullptr))
    return set_error(GRID_E_INVALID_ARG, "grid_advance: audit must be enabled on both configurations or on neither");
  return launch_advance(s, in->c, out->c, in->B, d_tokens, n_steps, d_status, in != out ? 1 : 0,
                        (cudaStream_t)stream);
}

// The four kernels of one mask step on `st`; `ev` (5 events or NULL) is
// recorded before the first kernel and after each.
int grid::launch_masks(const grid_spec* s, const DevConfigs& c, const MaskScratch& m, int B, uint32_t* d_mask,
                       int32_t* d_status, cudaStream_t st, const cudaEvent_t* ev, const FusedLogits& lg,
                       const AdvArgs* adv) {
  const Tables& t = s->t;
  const int vcw = std::max(1, s->vcw);
  const int n_vcbits = B * 2 * vcw;
  const size_t zero_words = (size_t)B * m.words_v * 2 + n_vcbits;
  const int zero_blocks = std::min(128, (int)((zero_words / 8 + kRowWarps * 32 * 4 - 1) / (kRowWarps * 32 * 4)) + 1);
  if (ev) GRID_CUDA(cudaEventRecord(ev[0], st));
  if (adv)
    GRID_CUDA(launch_pdl(k_row<true>, dim3(B + zero_blocks), dim3(kRowWarps * 32), t.blob_bytes, st, t, c, m.ctx,
                         m.rng, m.A2, m.sel, m.verd0, m.verd1, m.vcbits, n_vcbits, B, m.words_v, m.cache, *adv));
  else
    GRID_CUDA(launch_pdl(k_row<false>, dim3(B + zero_blocks), dim3(kRowWarps * 32), t.blob_bytes, st, t, c, m.ctx,
                         m.rng, m.A2, m.sel, m.verd0, m.verd1, m.vcbits, n_vcbits, B, m.words_v, m.cache,
                         AdvArgs{}));
  if (ev) GRID_CUDA(cudaEventRecord(ev[1], st));
  const int cd_blocks = (s->max_cd + 256 * kFilterPer - 1) / (256 * kFilterPer);
  const int vc_blocks = (s->max_vc + 256 * kFilterPer - 1) / (256 * kFilterPer);
  GRID_CUDA(launch_pdl(k_filter, dim3(std::max(1, cd_blocks + vc_blocks), B, 2), dim3(256), 0, st, t, m.ctx,
                       (const uint32_t*)m.sel, m.surv, m.cap, m.vsurv, m.vcap, cd_blocks));
  if (ev) GRID_CUDA(cudaEventRecord(ev[2], st));
  if (s->walk_work)  // the measured instance, which counts its work
    GRID_CUDA(launch_pdl(k_walk<true>, dim3(s->walk_blocks), dim3(kWalkWarps * 32), t.blob_bytes, st, t, m.ctx,
                         (const RowRanges*)m.rng, (const uint16_t*)c.stack, (const int32_t*)m.surv, m.cap,
                         (const uint32_t*)m.A2, m.verd0, m.verd1, m.vcbits, vcw, (const int32_t*)m.vsurv, m.vcap,
                         m.words_v, B, s->walk_work));
  else
    GRID_CUDA(launch_pdl(k_walk<false>, dim3(s->walk_blocks), dim3(kWalkWarps * 32), t.blob_bytes, st, t, m.ctx,
                         (const RowRanges*)m.rng, (const uint16_t*)c.stack, (const int32_t*)m.surv, m.cap,
                         (const uint32_t*)m.A2, m.verd0, m.verd1, m.vcbits, vcw, (const int32_t*)m.vsurv, m.vcap,
                         m.words_v, B, (unsigned long long*)nullptr));
  if (ev) GRID_CUDA(cudaEventRecord(ev[3], st));
  const dim3 pgrid((t.W + kPackWords - 1) / kPackWords, B);
  const size_t psmem = (size_t)(2 * std::max(1, t.nselw) + 2 * vcw) * 4;
  const int esz = lg.dtype == GRID_DTYPE_F32 ? 4 : 2;
  const int vec_ok = lg.p && ((uintptr_t)lg.p % 32 == 0) && ((lg.stride * esz) % 32 == 0);  // 32-byte sectors
  auto pack = [&](auto kern) {
    return launch_pdl(kern, pgrid, dim3(kPackWords), psmem, st, t, m.ctx, (const uint32_t*)m.sel,
                      (const uint32_t*)m.vcbits, vcw, (const uint32_t*)m.verd0, (const uint32_t*)m.verd1, m.words_v,
                      d_mask, d_status, lg.p, (long long)lg.stride, lg.p ? vec_ok : 0, m.cache);
  };
  const bool cached = m.cache.n > 0;
  const int mode = !lg.p ? 0 : (lg.dtype == GRID_DTYPE_F32 ? 1 : 2);
  cudaError_t pe;
  if (mode == 0)
    pe = cached ? pack(k_pack<0, true>) : pack(k_pack<0, false>);
  else if (mode == 1)
    pe = cached ? pack(k_pack<1, true>) : pack(k_pack<1, false>);
  else
    pe = cached ? pack(k_pack<2, true>) : pack(k_pack<2, false>);
  GRID_CUDA(pe);
  if (ev) GRID_CUDA(cudaEventRecord(ev[4], st));
  GRID_CUDA(cudaGetLastError());
  return GRID_OK;
}

extern "C" int grid_masks(const grid_spec* s, const grid_configs* c, uint32_t* d_mask, int32_t* d_status,
                          void* stream) {
  if (!s || !c || !d_mask || !d_status) return set_error(GRID_E_INVALID_ARG, "grid_masks: bad arguments");
  const MaskScratch m{c->ctx, c->rng, c->sel, c->verd0, c->verd1, c->A2, c->vcbits,
                      c->surv, c->vsurv, c->cap, c->vcap, c->words_v};
  return launch_masks(s, c->c, m, c->B, d_mask, d_status, (cudaStream_t)stream, c->ev[0] ? c->ev : nullptr);
}

extern "C" int grid_masks_apply(const grid_spec* s, const grid_configs* c, uint32_t* d_mask, int32_t* d_status,
                                void* d_logits, int32_t dtype, int64_t row_stride, void* stream) {
  if (!s || !c || !d_mask || !d_status || !d_logits || row_stride < s->t.V ||
      (dtype != GRID_DTYPE_F32 && dtype != GRID_DTYPE_BF16))
    return set_error(GRID_E_INVALID_ARG, "grid_masks_apply: bad arguments");
  const MaskScratch m{c->ctx, c->rng, c->sel, c->verd0, c->verd1, c->A2, c->vcbits,
                      c->surv, c->vsurv, c->cap, c->vcap, c->words_v};
  FusedLogits lg;
  lg.p = d_logits;
  lg.dtype = dtype;
  lg.stride = row_stride;
  return launch_masks(s, c->c, m, c->B, d_mask, d_status, (cudaStream_t)stream, c->ev[0] ? c->ev : nullptr, lg);
}

// ---------------------------------------------------------------------------
// Configuration-keyed mask cache (Sec. 4.3, Def. T1 key, Prop. OBL-KEY1).
struct grid_cache {
  const grid_spec* s = nullptr;
  CacheDev d;
  Arena mem;
};

extern "C" int grid_cache_create(const grid_spec* s, int32_t n_entries, grid_cache** out) {
  if (!s || !out || n_entries <= 0 || (n_entries & (n_entries - 1)) || n_entries > (1 << 20))
    return set_error(GRID_E_INVALID_ARG, "grid_cache_create: n_entries must be a power of two in 1 .. 2^20");
  *out = nullptr;
  auto* c = new grid_cache();
  c->s = s;
  c->d.n = n_entries;
  const size_t W = s->t.W;
  int rc;
  if ((rc = c->mem.alloc((size_t)n_entries * 16 * 4, (void**)&c->d.hdr)) ||
      (rc = c->mem.alloc((size_t)n_entries * W * 4, (void**)&c->d.ci)) ||
      (rc = c->mem.alloc((size_t)n_entries * W * 4, (void**)&c->d.sel)) ||
      (rc = c->mem.alloc(4 * 8, (void**)&c->d.stats))) {
    c->mem.release();
    delete c;
    return rc;
  }
  cudaError_t e = cudaMemset(c->d.hdr, 0, (size_t)n_entries * 16 * 4);
  if (e == cudaSuccess) e = cudaMemset(c->d.stats, 0, 4 * 8);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    c->mem.release();
    delete c;
    return set_error(GRID_E_CUDA, std::string("grid_cache_create: ") + cudaGetErrorString(e));
  }
  *out = c;
  return GRID_OK;
}

extern "C" void grid_cache_free(grid_cache* c) {
  if (!c) return;
  c->mem.release();
  delete c;
}

extern "C" int grid_cache_clear(grid_cache* c, void* stream) {
  if (!c) return set_error(GRID_E_INVALID_ARG, "grid_cache_clear: bad arguments");
  GRID_CUDA(cudaMemsetAsync(c->d.hdr, 0, (size_t)c->d.n * 16 * 4, (cudaStream_t)stream));
  GRID_CUDA(cudaMemsetAsync(c->d.stats, 0, 4 * 8, (cudaStream_t)stream));
  return GRID_OK;
}

extern "C" int grid_cache_stats(const grid_cache* c, int64_t out[4]) {
  if (!c || !out) return set_error(GRID_E_INVALID_ARG, "grid_cache_stats: bad arguments");
  unsigned long long st[3];
  std::vector<uint32_t> hdr((size_t)c->d.n * 16);
  GRID_CUDA(cudaMemcpy(st, c->d.stats, 3 * 8, cudaMemcpyDeviceToHost));
  GRID_CUDA(cudaMemcpy(hdr.data(), c->d.hdr, hdr.size() * 4, cudaMemcpyDeviceToHost));
  int64_t ready = 0;
  for (int i = 0; i < c->d.n; ++i) ready += hdr[(size_t)i * 16] == 2u;
  out[0] = (int64_t)st[0];
  out[1] = (int64_t)st[1];
  out[2] = (int64_t)st[2];
  out[3] = ready;
  return GRID_OK;
}

extern "C" int grid_masks_cached(const grid_spec* s, const grid_configs* c, grid_cache* cache, uint32_t* d_mask,
                                 int32_t* d_status, void* d_logits, int32_t dtype, int64_t row_stride, void* stream) {
  if (!s || !c || !cache || !d_mask || !d_status || cache->s != s ||
      (d_logits && (row_stride < s->t.V || (dtype != GRID_DTYPE_F32 && dtype != GRID_DTYPE_BF16))))
    return set_error(GRID_E_INVALID_ARG, "grid_masks_cached: bad arguments (the cache must belong to the spec)");
  MaskScratch m{c->ctx, c->rng, c->sel, c->verd0, c->verd1, c->A2, c->vcbits,
                c->surv, c->vsurv, c->cap, c->vcap, c->words_v};
  m.cache = cache->d;
  FusedLogits lg;
  lg.p = d_logits;
  lg.dtype = dtype;
  lg.stride = row_stride;
  return launch_masks(s, c->c, m, c->B, d_mask, d_status, (cudaStream_t)stream, c->ev[0] ? c->ev : nullptr, lg);
}

extern "C" int grid_advance_masks(const grid_spec* s, const grid_configs* in, grid_configs* out, grid_cache* cache,
                                  const int32_t* d_tokens, int32_t n_steps, uint32_t* d_mask, int32_t* d_status,
                                  void* d_logits, int32_t dtype, int64_t row_stride, void* stream) {
  if (!s || !in || !out || !d_tokens || !d_mask || !d_status || n_steps < 0 || in->B != out->B || in->D != out->D)
    return set_error(GRID_E_INVALID_ARG, "grid_advance_masks: bad arguments");
  if (cache && cache->s != s)
    return set_error(GRID_E_INVALID_ARG, "grid_advance_masks: the cache must belong to the spec");
  if (d_logits && (row_stride < s->t.V || (dtype != GRID_DTYPE_F32 && dtype != GRID_DTYPE_BF16)))
    return set_error(GRID_E_INVALID_ARG, "grid_advance_masks: bad logits arguments");
  if ((in->c.hs != nullptr) != (out->c.hs != nullptr))
    return set_error(GRID_E_INVALID_ARG,
                     "grid_advance_masks: audit must be enabled on both configurations or on neither");
  MaskScratch m{out->ctx, out->rng, out->sel, out->verd0, out->verd1, out->A2, out->vcbits,
                out->surv, out->vsurv, out->cap, out->vcap, out->words_v};
  if (cache) m.cache = cache->d;
  FusedLogits lg;
  lg.p = d_logits;
  lg.dtype = dtype;
  lg.stride = row_stride;
  const AdvArgs adv{in->c, d_tokens, n_steps, in != out ? 1 : 0};
  return launch_masks(s, out->c, m, out->B, d_mask, d_status, (cudaStream_t)stream, out->ev[0] ? out->ev : nullptr,
                      lg, &adv);
}

extern "C" int grid_spec_set_work_counters(grid_spec* s, unsigned long long* d_counters) {
  if (!s) return set_error(GRID_E_INVALID_ARG, "grid_spec_set_work_counters: bad arguments");
  s->walk_work = d_counters;
  return GRID_OK;
}

extern "C" int grid_configs_set_events(grid_configs* c, void* const* events, int32_t n_events) {
  if (!c || (n_events != 0 && n_events != kMaskKernels + 1) || (n_events && !events))
    return set_error(GRID_E_INVALID_ARG, "grid_configs_set_events: pass 0 or 5 events");
  for (int i = 0; i <= kMaskKernels; ++i) {
    c->ev[i] = n_events ? static_cast<cudaEvent_t>(events[i]) : nullptr;
    if (n_events && !c->ev[i]) {
      for (int k = 0; k <= kMaskKernels; ++k) c->ev[k] = nullptr;
      return set_error(GRID_E_INVALID_ARG, "grid_configs_set_events: null event");
    }
  }
  return GRID_OK;
}

// ---------------------------------------------------------------------------
// grid_masks_static: the mask step without any allocation.
//
// Some callers cannot allocate device memory when they need a mask: a serving
// engine whose own pool has reserved the device memory up front (a driver
// allocation would fail, or fragment the pool), or one that cannot afford the
// device-wide synchronization that freeing memory implies in the middle of a
// decoding step.  Such a caller keeps the parser configurations in device
// memory it already owns and passes them in; the scratch of the step (row
// contexts, class selections, survivor lists, verdict bitmaps) comes from the
// fixed array below instead of from a grid_configs.  The array is part of the
// library's device image: the CUDA runtime reserves it on every device where
// the library's kernels are loaded and keeps it until the process exits.
constexpr size_t kStaticScratchBytes = size_t(8) << 20;
constexpr int kStaticMaxDevices = 64;
static __device__ __align__(256) uint8_t g_static_scratch[kStaticScratchBytes];

namespace {
// In host code `g_static_scratch` names a host-side shadow of the array, not
// device memory; kernels get the device address found at set-up.
std::mutex g_static_mu;
uint8_t* g_static_dev[kStaticMaxDevices] = {};

// Offsets of the step's buffers inside the array (each 256-byte aligned),
// sized exactly as grid_configs_create sizes the same buffers.
struct StaticCarve {
  size_t ctx, rng, sel, verd0, verd1, A2, vcbits, surv, vsurv, total;
};

StaticCarve carve_static(const grid_spec* s, int B, int words_v) {
  StaticCarve c{};
  size_t at = 0;
  auto take = [&](size_t bytes) {
    const size_t o = at;
    at += (std::max<size_t>(bytes, 16) + 255) & ~size_t(255);
    return o;
  };
  c.ctx = take((size_t)B * sizeof(RowCtx));
  c.rng = take((size_t)B * sizeof(RowRanges));
  c.sel = take((size_t)B * 2 * std::max(1, s->t.nselw) * 4);
  c.verd0 = take((size_t)B * words_v * 4);
  c.verd1 = take((size_t)B * words_v * 4);
  c.A2 = take((size_t)B * 2 * s->t.T1 * 16);
  c.vcbits = take((size_t)B * 2 * std::max(1, s->vcw) * 4);
  c.surv = take((size_t)B * 2 * std::max(1, s->max_cd) * 4);
  c.vsurv = take((size_t)B * 2 * std::max(1, s->max_vc) * 4);
  c.total = at;
  return c;
}
}  // namespace

extern "C" int grid_masks_static(const grid_spec* s, const uint16_t* d_stack, const int32_t* d_depth,
                                 const int32_t* d_dfa_state, const int32_t* d_lex_node, const int32_t* d_flags,
                                 int32_t B, int32_t stack_stride, uint32_t* d_mask, int32_t* d_status,
                                 void* stream) {
  if (!s || !d_stack || !d_depth || !d_dfa_state || !d_lex_node || !d_flags || !d_mask || !d_status || B <= 0)
    return set_error(GRID_E_INVALID_ARG, "grid_masks_static: bad arguments");
  const Tables& t = s->t;
  if (B > kMaxRows)
    return set_error(GRID_E_TOO_LARGE, "grid_masks_static: more than " + std::to_string(kMaxRows) + " rows");
  if (stack_stride != t.D)
    return set_error(GRID_E_INVALID_ARG, "grid_masks_static: stack_stride " + std::to_string(stack_stride) +
                                             " differs from the grammar's max_depth " + std::to_string(t.D));
  int dev = 0;
  GRID_CUDA(cudaGetDevice(&dev));
  if (dev != s->device)
    return set_error(GRID_E_INVALID_ARG, "grid_masks_static: the spec lives on device " + std::to_string(s->device) +
                                             ", the current device is " + std::to_string(dev));
  if (dev < 0 || dev >= kStaticMaxDevices)
    return set_error(GRID_E_INVALID_ARG, "grid_masks_static: device ordinal " + std::to_string(dev) +
                                             " is beyond the " + std::to_string(kStaticMaxDevices) + " supported");
  const int words_v = t.W;
  const StaticCarve cv = carve_static(s, B, words_v);
  if (cv.total > kStaticScratchBytes)
    return set_error(GRID_E_TOO_LARGE, "grid_masks_static: B=" + std::to_string(B) + " needs " +
                                           std::to_string(cv.total) + " bytes of scratch with this spec, more than "
                                           "the " + std::to_string(kStaticScratchBytes) +
                                           "-byte static area; use grid_masks with a grid_configs instead");
  uint8_t* area = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_static_mu);
    if (!g_static_dev[dev]) {  // set-up, once per device
      void* p = nullptr;
      const cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch);
      if (e != cudaSuccess || !p)
        return set_error(GRID_E_CUDA, std::string("grid_masks_static: cudaGetSymbolAddress: ") +
                                          cudaGetErrorString(e));
      g_static_dev[dev] = static_cast<uint8_t*>(p);
    }
    area = g_static_dev[dev];
  }
  const MaskScratch m{reinterpret_cast<RowCtx*>(area + cv.ctx),
                      reinterpret_cast<RowRanges*>(area + cv.rng),
                      reinterpret_cast<uint32_t*>(area + cv.sel),
                      reinterpret_cast<uint32_t*>(area + cv.verd0),
                      reinterpret_cast<uint32_t*>(area + cv.verd1),
                      reinterpret_cast<uint32_t*>(area + cv.A2),
                      reinterpret_cast<uint32_t*>(area + cv.vcbits),
                      reinterpret_cast<int32_t*>(area + cv.surv),
                      reinterpret_cast<int32_t*>(area + cv.vsurv),
                      std::max(1, s->max_cd),
                      std::max(1, s->max_vc),
                      words_v};
  // the kernels only read the configurations
  const DevConfigs c{const_cast<uint16_t*>(d_stack), const_cast<int32_t*>(d_depth),
                     const_cast<int32_t*>(d_dfa_state), const_cast<int32_t*>(d_lex_node),
                     const_cast<int32_t*>(d_flags)};
  // What must start at zero is cleared by k_row itself on every call: the
  // verdict bitmaps and verdict-class bits (its clearing blocks) and each
  // row's queue, survivor and completion counters.  The other buffers are
  // written before they are read within the call, so the previous call's
  // contents do not matter.
  return launch_masks(s, c, m, B, d_mask, d_status, (cudaStream_t)stream, nullptr);
}

extern "C" int grid_apply_mask(const uint32_t* d_mask, void* d_logits, int32_t dtype, int32_t B, int32_t V,
                               int64_t row_stride, void* stream) {
  if (!d_mask || !d_logits || B <= 0 || V <= 0 || row_stride < V ||
      (dtype != GRID_DTYPE_F32 && dtype != GRID_DTYPE_BF16))
    return set_error(GRID_E_INVALID_ARG, "grid_apply_mask: bad arguments");
  cudaStream_t st = (cudaStream_t)stream;
  const int W = (V + 31) / 32;
  const int esz = dtype == GRID_DTYPE_F32 ? 4 : 2;
  const int vec_ok = ((uintptr_t)d_logits % 32 == 0) && ((row_stride * esz) % 32 == 0);  // 256-bit sectors
  if (B > 65535) return set_error(GRID_E_TOO_LARGE, "grid_apply_mask: more than 65535 rows in one call");
  const int sectors = (V * esz + 31) / 32;  // 32-byte sectors per row
  const int per_row = std::max(1, std::min((sectors + 255) / 256, (g_sms * 4 + B - 1) / B));
  const dim3 grid(per_row, B);
  if (dtype == GRID_DTYPE_F32)
    GRID_CUDA(launch_pdl(k_apply<float>, grid, dim3(256), 0, st, d_mask, (float*)d_logits, B, V, W,
                         (long long)row_stride, vec_ok));
  else
    GRID_CUDA(launch_pdl(k_apply<uint16_t>, grid, dim3(256), 0, st, d_mask, (uint16_t*)d_logits, B, V, W,
                         (long long)row_stride, vec_ok));
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
