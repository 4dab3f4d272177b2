// Host-side state shared by the translation units of libgrid: the spec and
// configuration objects behind the C ABI handles, the per-row scratch of a
// mask step, and the launchers of the mask step and the parser step.
#pragma once

#include <cuda_runtime.h>

#include <algorithm>
#include <string>
#include <vector>

#include "grid_blake2b.cuh"
#include "grid_device.cuh"

#define GRID_CUDA(call)                                                                  \
  do {                                                                                   \
    cudaError_t e_ = (call);                                                             \
    if (e_ != cudaSuccess)                                                               \
      return set_error(GRID_E_CUDA, std::string(#call) + ": " + cudaGetErrorString(e_)); \
  } while (0)

namespace grid {

// Per-row scratch of one grid_masks call.
struct RowCtx {
  uint32_t A0[4];   // allowed terminals at sigma
  uint32_t A1[4];   // allowed terminals at sigma' (after the forced emission)
  int32_t q, lx, depth, tbl0;
  uint32_t pc0, wc0;  // category bits of the pending lexeme's trie node
  int32_t emit_ok, eos_ok, status, complete;
  unsigned long long pack_done;  // k_pack blocks done with the row (low half) and with a set bit (high half)
  int32_t keep1, m1;
  int32_t work0;          // next item of the row's walk queue
  int32_t nrange;         // items over the continuing first-byte ranges (rows without a CI table)
  int32_t nsurv[2];       // CD spellings that survived k_filter, per context (0: sigma, 1: sigma')
  int32_t nvs[2];         // verdict classes that survived k_filter, per context
  int32_t nrng;
  int32_t chit, cfill;  // mask-cache entry this row reads (hit) or fills (miss), or -1
  uint32_t kill[8];  // bit b: first byte b ends the pending lexeme
  uint16_t ovl1[kMaxOvl];
};

// Continuing first-byte ranges of a row without a CI table.
struct RowRanges {
  int32_t lo[256];
  int32_t hi[256];
  int32_t cpre[257];
};

struct DevConfigs {
  uint16_t* stack;  // B*D
  int32_t* depth;
  int32_t* q;
  int32_t* lx;
  int32_t* flags;   // bit 0 = complete
  uint64_t* hs;     // B*D rolling node hashes parallel to the stacks (audit on), or NULL
};

struct Arena {
  std::vector<void*> owned;
  template <typename T>
  int upload(const std::vector<T>& v, const T** out) {
    void* p = nullptr;
    size_t n = std::max<size_t>(v.size(), 1) * sizeof(T);
    GRID_CUDA(cudaMalloc(&p, n));
    owned.push_back(p);
    if (!v.empty()) GRID_CUDA(cudaMemcpy(p, v.data(), v.size() * sizeof(T), cudaMemcpyHostToDevice));
    *out = static_cast<const T*>(p);
    return GRID_OK;
  }
  int alloc(size_t n, void** out) {
    GRID_CUDA(cudaMalloc(out, std::max<size_t>(n, 16)));
    owned.push_back(*out);
    return GRID_OK;
  }
  void release() {
    for (void* p : owned) cudaFree(p);
    owned.clear();
  }
};

// Buffers of one mask step (owned by a grid_configs, or carved out of the
// static area of grid_masks_static).
// Device view of a configuration-keyed mask cache (grid_cache): per entry a
// 16-word header -- [0] state (0 empty, 1 being filled, 2 ready), [1] kind
// (1 = identifier position: a lexer state without a CI table), [2] lexer
// state, [3] emit_ok, [4..7] A(sigma), [8..11] A(sigma') -- and W words of
// the values of the context-independent bits (ci) and W words marking the
// ids whose bits are the stack-dependent residue (sel).  n == 0: no cache.
struct CacheDev {
  uint32_t* hdr = nullptr;
  uint32_t* ci = nullptr;
  uint32_t* sel = nullptr;
  unsigned long long* stats = nullptr;  // [0] lookups, [1] hits, [2] fills claimed
  int n = 0;                            // entries, a power of two
};

struct MaskScratch {
  RowCtx* ctx;
  RowRanges* rng;
  uint32_t *sel, *verd0, *verd1, *A2, *vcbits;
  int32_t *surv, *vsurv;
  int cap, vcap, words_v;
  CacheDev cache;
};

// Logits to mask in the same pass as the mask (grid_masks_apply), or none.
struct FusedLogits {
  void* p = nullptr;
  int dtype = GRID_DTYPE_F32;
  long long stride = 0;
};

// Tokens to feed before the mask step, in its first kernel
// (grid_advance_masks): from cin into the configurations being masked.
struct AdvArgs {
  DevConfigs cin;
  const int32_t* tokens;
  int n_steps;
  int copy;  // 1: cin and the masked configurations are distinct (out of place)
};

constexpr int kMaskKernels = 4;  // k_row, k_filter, k_walk, k_pack

extern int g_sms;  // SM count of the current device, set by grid_specialize

}  // namespace grid

// Device tables of the reserve completion (grid_reserve), built by
// grid_specialize from the grammar's completion tables and the vocabulary.
struct ReserveTables {
  int ok = 0;            // 1 when built
  int NC = 1;            // categories (at least 1: the row stride of lx_wdist)
  int E = 0;             // search entries per row
  const int32_t* item_off = nullptr;  // S + 1: kernel items of each state
  const int32_t* item_p = nullptr;    // production of each kernel item
  const int32_t* item_d = nullptr;    // dot of each kernel item (the length of alpha)
  const uint32_t* item_cost = nullptr;  // tokens of beta's cheapest rendering
  const int32_t* prod_off = nullptr;  // P + 1
  const int32_t* prod_rhs = nullptr;  // symbols: < T1 terminal, else T1 + nonterminal
  const int32_t* ny_off = nullptr;    // NNT + 1: the cheapest terminal yield of each nonterminal
  const int32_t* ny = nullptr;
  const int32_t* rend_off = nullptr;  // T1 + 1: the tokens rendering each terminal
  const int32_t* rend_tok = nullptr;
  const uint16_t* lx_wdist = nullptr;  // LN * NC
  const uint8_t* lx_wbyte = nullptr;
  const uint8_t* dfa_tdist = nullptr;  // Q * T1
  const uint8_t* dfa_tbyte = nullptr;
  const int16_t* sep_byte = nullptr;   // Q
  const int32_t* byte_tok = nullptr;   // 256: the id spelling each single byte, or -1
};

struct grid_spec {
  const grid_grammar* g = nullptr;
  const grid_vocab* v = nullptr;
  grid::Tables t;
  grid::Arena mem;
  int device = 0;
  int sms = 152;
  int n1 = 0;  // walk chunks of the start state's CD list
  int walk_blocks = 0;  // persistent k_walk grid: resident blocks per SM x SMs
  int max_cd = 0;       // longest CD list of a table
  int vcw = 0;          // words of the largest table's verdict-class bitset
  int n_vc = 0;         // verdict classes over all tables
  int max_vc = 0;       // verdict classes of the largest table
  uint8_t fingerprint[16] = {};  // BLAKE2b-128 of the grammar and vocabulary fingerprints
  ReserveTables rt;
  unsigned long long* walk_work = nullptr;  // measurement hook: k_walk's work counters (4), or NULL
};

struct grid_configs {
  int B = 0, D = 0, words_v = 0;
  grid::DevConfigs c;
  grid::RowCtx* ctx = nullptr;
  grid::RowRanges* rng = nullptr;
  uint32_t* sel = nullptr;
  uint32_t* verd0 = nullptr;
  uint32_t* verd1 = nullptr;
  uint32_t* A2 = nullptr;
  uint32_t* vcbits = nullptr;
  int32_t* surv = nullptr;
  int32_t* vsurv = nullptr;
  int cap = 0, vcap = 0;
  int32_t* aux = nullptr;  // 4 x B ints of per-row working state for forced spans and reserves
  int32_t* rscratch = nullptr;  // per-row search space of grid_reserve (entries and level heads)
  // audit chain (grid_configs_enable_audit): node hashes (c.hs), per-row
  // chain heads (16 bytes) and record counters
  uint8_t* heads = nullptr;
  uint64_t* steps = nullptr;
  cudaEvent_t ev[grid::kMaskKernels + 1] = {};  // optional per-kernel timing events
  grid::Arena mem;
};

namespace grid {

// The four kernels of one mask step (k_row, k_filter, k_walk, k_pack) on
// `st`; `ev` (5 events or NULL) is recorded before the first kernel and after
// each.  With lg.p set, k_pack also masks the logits; with adv set, k_row
// first feeds adv's tokens into c.
int launch_masks(const grid_spec* s, const DevConfigs& c, const MaskScratch& m, int B, uint32_t* d_mask,
                 int32_t* d_status, cudaStream_t st, const cudaEvent_t* ev, const FusedLogits& lg = FusedLogits(),
                 const AdvArgs* adv = nullptr);

// The parser step (k_advance) of B rows from `in` into `out` (copy = 1: out
// of place) on `st`.
int launch_advance(const grid_spec* s, const DevConfigs& in, const DevConfigs& out, int B, const int32_t* d_tokens,
                   int32_t n_steps, int32_t* d_status, int copy, cudaStream_t st);

// Reserve completion tables (grid_span.cu), built at the end of
// grid_specialize into s->rt (device memory owned by s->mem).
int build_reserve_tables(grid_spec* s);
// Bytes of grid_reserve's search space per row.
size_t reserve_scratch_bytes(const grid_spec* s);

// Audit chain (grid_audit.cu): a fresh chain and node hashes of the current
// stacks when audit is enabled on `c` (no-op otherwise), and one record per
// row with a non-negative token (records at d_records + b * rec_stride).
int audit_reset(const grid_spec* s, grid_configs* c, cudaStream_t st);
int audit_append(const grid_spec* s, grid_configs* c, const uint32_t* d_mask, const int32_t* d_tokens, uint32_t kind,
                 uint8_t* d_records, long long rec_stride, cudaStream_t st);

}  // namespace grid
