// BLAKE2b (RFC 7693), written from the RFC's description, for the audit
// chain: the rolling configuration hash of every stack node and the
// content-addressed ids and chain links of the audit records.  Unkeyed;
// digests of 1..64 bytes; callable from host and device code.
#pragma once

#include <cstddef>
#include <cstdint>

#ifdef __CUDACC__
#define GRID_HD __host__ __device__ __forceinline__
#else
#define GRID_HD inline
#endif

namespace grid {

// initialization vector (RFC 7693, Sec. 2.6): the SHA-512 initial hash values
struct Blake2bIV {
  static GRID_HD uint64_t at(int i) {
    return i == 0 ? 0x6a09e667f3bcc908ull
           : i == 1 ? 0xbb67ae8584caa73bull
           : i == 2 ? 0x3c6ef372fe94f82bull
           : i == 3 ? 0xa54ff53a5f1d36f1ull
           : i == 4 ? 0x510e527fade682d1ull
           : i == 5 ? 0x9b05688c2b3e6c1full
           : i == 6 ? 0x1f83d9abfb41bd6bull
                    : 0x5be0cd19137e2179ull;
  }
};

// message word schedule sigma (RFC 7693, Sec. 2.7), rows 0..9; rounds 10 and
// 11 reuse rows 0 and 1.  Row r, entry i is packed as nibble i of word r.
GRID_HD int blake2b_sigma(int r, int i) {
  constexpr uint64_t rows[10] = {
      0xfedcba9876543210ull, 0x357b20c16df984aeull, 0x491763eadf250c8bull, 0x8f04a562ebcd1397ull,
      0xd386cb1efa427509ull, 0x91ef57d438b0a6c2ull, 0xb8293670a4def15cull, 0xa2684f05931ce7bdull,
      0x5a417d2c803b9ef6ull, 0x0dc3e9bf5167482aull};
  return (int)((rows[r] >> (4 * i)) & 0xFu);
}

GRID_HD uint64_t blake2b_rotr(uint64_t x, int n) { return (x >> n) | (x << (64 - n)); }

GRID_HD void blake2b_g(uint64_t* v, int a, int b, int c, int d, uint64_t x, uint64_t y) {
  v[a] = v[a] + v[b] + x;
  v[d] = blake2b_rotr(v[d] ^ v[a], 32);
  v[c] = v[c] + v[d];
  v[b] = blake2b_rotr(v[b] ^ v[c], 24);
  v[a] = v[a] + v[b] + y;
  v[d] = blake2b_rotr(v[d] ^ v[a], 16);
  v[c] = v[c] + v[d];
  v[b] = blake2b_rotr(v[b] ^ v[c], 63);
}

// Compression function F (RFC 7693, Sec. 3.2) of one 128-byte block m (16
// little-endian words) into state h, with byte counter t and final flag.
GRID_HD void blake2b_compress(uint64_t* h, const uint64_t* m, uint64_t t, bool last) {
  uint64_t v[16];
  for (int i = 0; i < 8; ++i) {
    v[i] = h[i];
    v[i + 8] = Blake2bIV::at(i);
  }
  v[12] ^= t;  // the counter's high word stays zero for messages below 2^64 bytes
  if (last) v[14] = ~v[14];
  for (int r = 0; r < 12; ++r) {
    const int s = r % 10;
    blake2b_g(v, 0, 4, 8, 12, m[blake2b_sigma(s, 0)], m[blake2b_sigma(s, 1)]);
    blake2b_g(v, 1, 5, 9, 13, m[blake2b_sigma(s, 2)], m[blake2b_sigma(s, 3)]);
    blake2b_g(v, 2, 6, 10, 14, m[blake2b_sigma(s, 4)], m[blake2b_sigma(s, 5)]);
    blake2b_g(v, 3, 7, 11, 15, m[blake2b_sigma(s, 6)], m[blake2b_sigma(s, 7)]);
    blake2b_g(v, 0, 5, 10, 15, m[blake2b_sigma(s, 8)], m[blake2b_sigma(s, 9)]);
    blake2b_g(v, 1, 6, 11, 12, m[blake2b_sigma(s, 10)], m[blake2b_sigma(s, 11)]);
    blake2b_g(v, 2, 7, 8, 13, m[blake2b_sigma(s, 12)], m[blake2b_sigma(s, 13)]);
    blake2b_g(v, 3, 4, 9, 14, m[blake2b_sigma(s, 14)], m[blake2b_sigma(s, 15)]);
  }
  for (int i = 0; i < 8; ++i) h[i] ^= v[i] ^ v[i + 8];
}

// Incremental hashing over byte pieces.
struct Blake2b {
  uint64_t h[8];
  uint64_t buf[16];
  uint64_t t;
  int fill;  // bytes in buf
  int outlen;
  GRID_HD void init(int out_bytes) {
    outlen = out_bytes;
    for (int i = 0; i < 8; ++i) h[i] = Blake2bIV::at(i);
    h[0] ^= 0x01010000ull ^ (uint64_t)out_bytes;  // parameter block: digest length, no key, fanout 1, depth 1
    for (int i = 0; i < 16; ++i) buf[i] = 0;
    t = 0;
    fill = 0;
  }
  GRID_HD void put_byte(uint8_t x) {
    if (fill == 128) {  // a full block is compressed only once more input follows
      t += 128;
      blake2b_compress(h, buf, t, false);
      for (int i = 0; i < 16; ++i) buf[i] = 0;
      fill = 0;
    }
    buf[fill >> 3] |= (uint64_t)x << (8 * (fill & 7));
    ++fill;
  }
  GRID_HD void update(const void* p, size_t n) {
    const uint8_t* b = static_cast<const uint8_t*>(p);
    size_t i = 0;
    while (i < n && (fill & 7)) put_byte(b[i++]);  // to a word boundary
    // whole little-endian words while the block has room and input follows it
    for (; i + 8 <= n; i += 8) {
      if (fill == 128) {
        t += 128;
        blake2b_compress(h, buf, t, false);
        for (int k = 0; k < 16; ++k) buf[k] = 0;
        fill = 0;
      }
      uint64_t w = 0;
      for (int k = 0; k < 8; ++k) w |= (uint64_t)b[i + k] << (8 * k);
      buf[fill >> 3] = w;
      fill += 8;
    }
    for (; i < n; ++i) put_byte(b[i]);
  }
  GRID_HD void put_u32(uint32_t x) {
    for (int i = 0; i < 4; ++i) put_byte((uint8_t)(x >> (8 * i)));
  }
  GRID_HD void put_u64(uint64_t x) {
    for (int i = 0; i < 8; ++i) put_byte((uint8_t)(x >> (8 * i)));
  }
  GRID_HD void final(uint8_t* out) {
    t += (uint64_t)fill;
    blake2b_compress(h, buf, t, true);
    for (int i = 0; i < outlen; ++i) out[i] = (uint8_t)(h[i >> 3] >> (8 * (i & 7)));
  }
};

// H(node) = low64(BLAKE2b-128(H(parent) || u32(kind) || u32(id))): the
// rolling configuration hash of a stack node entered by a terminal (kind 0,
// id = terminal index) or by the goto on a nonterminal (kind 1, id = rank of
// the nonterminal's name in byte order among the grammar's nonterminals).
GRID_HD uint64_t node_hash(uint64_t parent, uint32_t sym) {
  Blake2b b;
  b.init(16);
  b.put_u64(parent);
  b.put_u32(sym >> 16);
  b.put_u32(sym & 0xFFFFu);
  uint8_t d[16];
  b.final(d);
  uint64_t x = 0;
  for (int i = 0; i < 8; ++i) x |= (uint64_t)d[i] << (8 * i);
  return x;
}

}  // namespace grid
