// Internal host-side structures shared by grid_host.cpp (compiler, vocabulary)
// and grid_kernels.cu (device upload, kernels).
#pragma once

#include <cstdint>
#include <string>
#include <vector>

#include "../../include/grid.h"

namespace grid {

constexpr int kMaxTerms = 128;   // terminal bitmasks are 4 x uint32 (incl. $end)
constexpr int kDead = 0;         // DFA state numbering: 0 = dead, 1 = start
constexpr int kStart = 1;
constexpr int16_t kAccept = 0x7FFF;  // ACTION code for ACCEPT

// Thread-local error reporting.
int set_error(int code, const std::string& msg);

// Compiled grammar (Sec. 2 layers L1-L3), host copy of every device table.
struct HostGrammar {
  // terminals: 0..n_term-1 in priority order, $end = n_term, T1 = n_term + 1
  int n_term = 0;
  int T1 = 0;
  std::vector<std::string> term_names;
  uint32_t ignored[4] = {0, 0, 0, 0};
  uint32_t catmask[4] = {0, 0, 0, 0};
  int n_cat = 0;
  std::vector<int> cat_term;  // category index -> terminal id

  // minimised union lexer DFA
  int Q = 0, C = 0;
  uint8_t byte_class[256];
  std::vector<uint16_t> next;  // Q*C
  std::vector<uint32_t> acc;   // Q*4 terminal bitmask accepted at q
  std::vector<uint32_t> live;  // Q*4 terminals with an accepting state reachable

  // LALR(1)
  int S = 0, NNT = 0, P = 0;
  std::vector<int16_t> action;  // S*T1: 0 error, s+1 shift s, -(p+1) reduce p, kAccept
  std::vector<uint16_t> go;     // S*NNT
  std::vector<uint8_t> plen;    // P
  std::vector<uint16_t> plhs;   // P

  // identifier trie over the union of all lexicons (node 0 = root)
  int LN = 0;
  std::vector<int32_t> lx_cstart;  // LN+1 CSR offsets of children (sorted by byte)
  std::vector<uint8_t> lx_cbyte;
  std::vector<int32_t> lx_cnode;
  std::vector<uint32_t> lx_pcats;  // category bits c with node string in Prefix(W_c)
  std::vector<uint32_t> lx_wcats;  // category bits c with node string in W_c

  int max_depth = 4096;

  // reserve completion (Sec. 5, Prop. 9): LR(0) kernel items per state
  // (production, dot), the productions' right-hand sides (< T1 terminal,
  // else T1 + nonterminal), per lexicon node and category the length of and
  // first byte towards the shortest word below (0xFFFF: none), per DFA state
  // and terminal the length of and first byte towards the shortest
  // accepting continuation (0xFF: none), per DFA state the byte that ends
  // the pending lexeme and starts an ignored one (-1: none), and per terminal
  // the lexeme that renders it (empty: none)
  std::vector<int32_t> kitem_off, kitem_p, kitem_d;
  std::vector<int32_t> prod_off, prod_rhs;
  std::vector<uint16_t> lx_wdist;
  std::vector<uint8_t> lx_wbyte;
  std::vector<uint8_t> dfa_tdist, dfa_tbyte;
  std::vector<int16_t> sep_byte;
  std::vector<std::string> render_lex;

  // audit: the symbol entering each LALR state (kind << 16 | id: kind 0 =
  // terminal id, kind 1 = rank of the nonterminal's name in byte order among
  // all nonterminals of the grammar text; 0xFFFFFFFF for the start state)
  std::vector<uint32_t> acc_sym;
  uint8_t fingerprint[16] = {};  // BLAKE2b-128 of the compile inputs
};

// Byte trie of the vocabulary (Def. 3), stored as the lexicographically sorted
// distinct spellings (= DFS order of the trie): the spellings that start with
// one byte, and so one subtree of the root, are contiguous.
struct HostVocab {
  int V = 0;
  int eos = -1;
  int NS = 0;
  std::vector<int32_t> spell_off;   // NS+1
  std::vector<uint8_t> spell_bytes;
  std::vector<int32_t> spell_of_id; // V, -1 for EOS/special
  std::vector<int32_t> first_of_byte;  // 257: spellings with first byte b are [f[b], f[b+1])
  bool byte_complete = false;
  uint8_t fingerprint[16] = {};  // BLAKE2b-128 of the vocabulary inputs
};

}  // namespace grid

struct grid_grammar {
  grid::HostGrammar h;
};

struct grid_vocab {
  grid::HostVocab h;
};
