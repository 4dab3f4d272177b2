// Jump-forward forced spans (GRID Sec. 6.1, step 6 of the per-token hot
// path): while a row's mask admits exactly one token id, that token is
// forced; it is appended to the row's span and the row is advanced by it,
// without sampling.  Everything runs on the device: per span position one
// mask step, one kernel that finds each row's forced token (or stops the
// row), and one parser step whose no-op token (-1) leaves stopped rows alone.

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
