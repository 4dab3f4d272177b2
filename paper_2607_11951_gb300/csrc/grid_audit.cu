// Audit chain (GRID Sec. 6.4, "The audit chain"): every decoding step of a
// row appends a record (step, configuration hash, mask entry id, token,
// blocked count, kind, previous record's hash) chained by BLAKE2b-128 from a
// genesis constant; a seal record ends the log with the stop reason, the
// artifacts' fingerprint and mode flags.  The configuration hash is the
// rolling hash of the row's top stack node, carried in a hash stack parallel
// to the LR stack and updated by k_advance at O(1) per push.
//
// Record layout (80 bytes, little-endian): 0 u64 step, 8 u64 config_hash,
// 16 u8[16] mask_entry_id, 32 i32 token, 36 u32 blocked_count, 40 u32 kind,
// 44 u8[16] prev_hash, 60 u32 zero, 64 u8[16] hash = BLAKE2b-128(bytes 0..59).
//
// Mask entry id: the mask row's words in 1,024-byte chunks (256 words, the
// last one shorter), each hashed with BLAKE2b-128, then BLAKE2b-128 of
// "GRIDmask" || u32 V || u32 chunks || the chunk digests: a content address
// whose chunks the lanes of a warp hash at once.

#include "grid_state.cuh"

namespace grid {
namespace {

constexpr int kRecBytes = 80;
constexpr int kChunkWords = 256;

struct Digest16 {
  uint8_t b[16];
};

Digest16 genesis_digest() {
  Digest16 d;
  Blake2b h;
  h.init(16);
  h.update("GRID audit chain genesis", 24);
  h.final(d.b);
  return d;
}

// BLAKE2b-128 of n little-endian 32-bit words; whole 128-byte blocks are
// packed straight from the words.
__device__ void hash_words(const uint32_t* w, int n, uint8_t* out) {
  uint64_t h[8];
  for (int i = 0; i < 8; ++i) h[i] = Blake2bIV::at(i);
  h[0] ^= 0x01010000ull ^ 16ull;
  uint64_t m[16];
  uint64_t t = 0;
  int k = 0;
  while (n - k > 32) {  // a full block that is not the last one
    for (int j = 0; j < 16; ++j) m[j] = (uint64_t)w[k + 2 * j] | ((uint64_t)w[k + 2 * j + 1] << 32);
    t += 128;
    blake2b_compress(h, m, t, false);
    k += 32;
  }
  for (int j = 0; j < 16; ++j) {
    const int a = k + 2 * j, b = a + 1;
    m[j] = (a < n ? (uint64_t)w[a] : 0ull) | (b < n ? ((uint64_t)w[b] << 32) : 0ull);
  }
  t += (uint64_t)(n - k) * 4;
  blake2b_compress(h, m, t, true);
  for (int i = 0; i < 16; ++i) out[i] = (uint8_t)(h[i >> 3] >> (8 * (i & 7)));
}

__host__ __device__ void put_le(uint8_t* p, uint64_t x, int n) {
  for (int i = 0; i < n; ++i) p[i] = (uint8_t)(x >> (8 * i));
}

// Fill the record's fields (bytes 0..59), hash them, write the record, and
// advance the row's chain head and counter.
__device__ void write_record(uint8_t* rec, uint64_t step, uint64_t cfg_hash, const uint8_t* mask_id, int32_t token,
                             uint32_t blocked, uint32_t kind, uint8_t* head) {
  uint8_t r[kRecBytes];
  put_le(r, step, 8);
  put_le(r + 8, cfg_hash, 8);
  for (int i = 0; i < 16; ++i) r[16 + i] = mask_id[i];
  put_le(r + 32, (uint32_t)token, 4);
  put_le(r + 36, blocked, 4);
  put_le(r + 40, kind, 4);
  for (int i = 0; i < 16; ++i) r[44 + i] = head[i];
  put_le(r + 60, 0, 4);
  Blake2b h;
  h.init(16);
  h.update(r, 60);
  h.final(r + 64);
  for (int i = 0; i < kRecBytes; ++i) rec[i] = r[i];
  for (int i = 0; i < 16; ++i) head[i] = r[64 + i];
}

// One thread per row: the node hashes of the row's current stack from the
// root up, and a fresh chain (genesis head, record counter 0).
__global__ void k_audit_init(Tables t, DevConfigs c, uint8_t* __restrict__ heads, uint64_t* __restrict__ steps,
                             Digest16 gen, int B) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const uint16_t* st = c.stack + (size_t)b * t.D;
  uint64_t* hs = c.hs + (size_t)b * t.D;
  const int d = c.depth[b];
  uint64_t h = 0;
  hs[0] = 0;
  for (int i = 1; i < d; ++i) {
    h = node_hash(h, t.acc_sym[st[i]]);
    hs[i] = h;
  }
  for (int i = 0; i < 16; ++i) heads[(size_t)b * 16 + i] = gen.b[i];
  steps[b] = 0;
}

// One warp per row (rows whose token is negative get no record): the lanes
// hash the mask row's chunks and count its set bits, lane 0 makes the mask
// entry id and the record.
__global__ void k_audit_append(Tables t, DevConfigs c, const uint32_t* __restrict__ mask,
                               const int32_t* __restrict__ tokens, uint32_t kind, uint8_t* __restrict__ heads,
                               uint64_t* __restrict__ steps, uint8_t* __restrict__ records, long long rec_stride,
                               int B) {
  extern __shared__ uint8_t s_dig[];  // chunks x 16 bytes
  const int b = blockIdx.x, lane = threadIdx.x;
  if (b >= B) return;
  const int tok = tokens[b];
  if (tok < 0) return;
  const int W = t.W;
  const uint32_t* row = mask + (size_t)b * W;
  const int nch = (W + kChunkWords - 1) / kChunkWords;
  for (int ch = lane; ch < nch; ch += 32) hash_words(row + ch * kChunkWords, min(kChunkWords, W - ch * kChunkWords), s_dig + ch * 16);
  int cnt = 0;
  for (int w = lane; w < W; w += 32) cnt += __popc(row[w]);
  cnt = __reduce_add_sync(0xffffffffu, cnt);
  __syncwarp();
  if (lane != 0) return;
  uint8_t id[16];
  Blake2b h;
  h.init(16);
  h.update("GRIDmask", 8);
  h.put_u32((uint32_t)t.V);
  h.put_u32((uint32_t)nch);
  h.update(s_dig, (size_t)nch * 16);
  h.final(id);
  const uint64_t cfg = c.hs[(size_t)b * t.D + c.depth[b] - 1];
  const uint64_t step = steps[b];
  write_record(records + (size_t)b * rec_stride, step, cfg, id, tok, (uint32_t)(t.V - cnt), kind, heads + (size_t)b * 16);
  steps[b] = step + 1;
}

// The seal: kind 3, the final configuration's hash, the spec's fingerprint
// in place of a mask id, the stop reason as the token and the mode flags as
// the blocked count.
__global__ void k_audit_seal(Tables t, DevConfigs c, const int32_t* __restrict__ reason, uint32_t mode,
                             Digest16 fp, uint8_t* __restrict__ heads, uint64_t* __restrict__ steps,
                             uint8_t* __restrict__ records, int B) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const uint64_t cfg = c.hs[(size_t)b * t.D + c.depth[b] - 1];
  const uint64_t step = steps[b];
  write_record(records + (size_t)b * kRecBytes, step, cfg, fp.b, reason[b], mode, 3u, heads + (size_t)b * 16);
  steps[b] = step + 1;
}

}  // namespace

int audit_reset(const grid_spec* s, grid_configs* c, cudaStream_t st) {
  if (!c->c.hs) return GRID_OK;
  k_audit_init<<<(c->B + 127) / 128, 128, 0, st>>>(s->t, c->c, c->heads, c->steps, genesis_digest(), c->B);
  GRID_CUDA(cudaGetLastError());
  return GRID_OK;
}

int audit_append(const grid_spec* s, grid_configs* c, const uint32_t* d_mask, const int32_t* d_tokens, uint32_t kind,
                 uint8_t* d_records, long long rec_stride, cudaStream_t st) {
  const int nch = (s->t.W + kChunkWords - 1) / kChunkWords;
  k_audit_append<<<c->B, 32, (size_t)nch * 16, st>>>(s->t, c->c, d_mask, d_tokens, kind, c->heads, c->steps,
                                                     d_records, rec_stride, c->B);
  GRID_CUDA(cudaGetLastError());
  return GRID_OK;
}

}  // namespace grid

using namespace grid;

extern "C" int grid_configs_enable_audit(const grid_spec* s, grid_configs* c, void* stream) {
  if (!s || !c) return set_error(GRID_E_INVALID_ARG, "grid_configs_enable_audit: bad arguments");
  if (!c->c.hs) {
    int rc;
    if ((rc = c->mem.alloc((size_t)c->B * c->D * 8, (void**)&c->c.hs)) ||
        (rc = c->mem.alloc((size_t)c->B * 16, (void**)&c->heads)) || (rc = c->mem.alloc((size_t)c->B * 8, (void**)&c->steps)))
      return rc;
  }
  cudaStream_t st = (cudaStream_t)stream;
  int rc = audit_reset(s, c, st);
  if (rc) return rc;
  GRID_CUDA(cudaStreamSynchronize(st));
  return GRID_OK;
}

extern "C" int grid_audit_append(const grid_spec* s, grid_configs* c, const uint32_t* d_mask, const int32_t* d_tokens,
                                 int32_t kind, uint8_t* d_records, void* stream) {
  if (!s || !c || !d_mask || !d_tokens || !d_records || kind < 0)
    return set_error(GRID_E_INVALID_ARG, "grid_audit_append: bad arguments");
  if (!c->c.hs) return set_error(GRID_E_INVALID_ARG, "grid_audit_append: audit is not enabled on these configurations");
  return audit_append(s, c, d_mask, d_tokens, (uint32_t)kind, d_records, kRecBytes, (cudaStream_t)stream);
}

extern "C" int grid_audit_seal(const grid_spec* s, grid_configs* c, const int32_t* d_reason, uint32_t mode_flags,
                               uint8_t* d_records, void* stream) {
  if (!s || !c || !d_reason || !d_records) return set_error(GRID_E_INVALID_ARG, "grid_audit_seal: bad arguments");
  if (!c->c.hs) return set_error(GRID_E_INVALID_ARG, "grid_audit_seal: audit is not enabled on these configurations");
  Digest16 fp;
  for (int i = 0; i < 16; ++i) fp.b[i] = s->fingerprint[i];
  k_audit_seal<<<(c->B + 127) / 128, 128, 0, (cudaStream_t)stream>>>(s->t, c->c, d_reason, mode_flags, fp, c->heads,
                                                                     c->steps, d_records, c->B);
  GRID_CUDA(cudaGetLastError());
  return GRID_OK;
}

extern "C" int grid_audit_head(const grid_configs* c, int32_t row, uint8_t* head, uint64_t* n_records) {
  if (!c || !head || !n_records || row < 0 || row >= c->B) return set_error(GRID_E_INVALID_ARG, "grid_audit_head: bad arguments");
  if (!c->c.hs) return set_error(GRID_E_INVALID_ARG, "grid_audit_head: audit is not enabled on these configurations");
  GRID_CUDA(cudaMemcpy(head, c->heads + (size_t)row * 16, 16, cudaMemcpyDeviceToHost));
  GRID_CUDA(cudaMemcpy(n_records, c->steps + row, 8, cudaMemcpyDeviceToHost));
  return GRID_OK;
}

extern "C" int64_t grid_audit_verify(const uint8_t* records, int64_t n, const uint8_t* genesis) {
  if (!records || n < 0) return set_error(GRID_E_INVALID_ARG, "grid_audit_verify: bad arguments");
  uint8_t prev[16];
  if (genesis) {
    for (int i = 0; i < 16; ++i) prev[i] = genesis[i];
  } else {
    const Digest16 g = genesis_digest();
    for (int i = 0; i < 16; ++i) prev[i] = g.b[i];
  }
  for (int64_t k = 0; k < n; ++k) {
    const uint8_t* r = records + k * kRecBytes;
    uint64_t step = 0;
    for (int i = 0; i < 8; ++i) step |= (uint64_t)r[i] << (8 * i);
    bool ok = step == (uint64_t)k && r[60] == 0 && r[61] == 0 && r[62] == 0 && r[63] == 0;
    for (int i = 0; i < 16 && ok; ++i) ok = r[44 + i] == prev[i];
    uint8_t h[16];
    Blake2b b;
    b.init(16);
    b.update(r, 60);
    b.final(h);
    for (int i = 0; i < 16 && ok; ++i) ok = r[64 + i] == h[i];
    if (!ok) return k;
    for (int i = 0; i < 16; ++i) prev[i] = h[i];
  }
  return -1;
}

extern "C" int grid_audit_genesis(uint8_t* out) {
  if (!out) return set_error(GRID_E_INVALID_ARG, "grid_audit_genesis: bad arguments");
  const Digest16 g = genesis_digest();
  for (int i = 0; i < 16; ++i) out[i] = g.b[i];
  return GRID_OK;
}

extern "C" int grid_blake2b(const void* data, size_t n, uint8_t* out, int32_t out_bytes) {
  if ((!data && n) || !out || out_bytes < 1 || out_bytes > 64) return set_error(GRID_E_INVALID_ARG, "grid_blake2b: bad arguments");
  Blake2b b;
  b.init(out_bytes);
  b.update(data, n);
  b.final(out);
  return GRID_OK;
}

extern "C" int grid_fingerprint(const grid_grammar* g, const grid_vocab* v, const grid_spec* s, uint8_t* out) {
  if (!out || ((g != nullptr) + (v != nullptr) + (s != nullptr)) != 1)
    return set_error(GRID_E_INVALID_ARG, "grid_fingerprint: pass exactly one of grammar, vocabulary, spec");
  const uint8_t* f = g ? g->h.fingerprint : v ? v->h.fingerprint : s->fingerprint;
  for (int i = 0; i < 16; ++i) out[i] = f[i];
  return GRID_OK;
}
