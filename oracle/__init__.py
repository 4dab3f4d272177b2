"""Plain CPU oracle for GRID's cold full-vocabulary mask -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package.  The product
path (the CUDA library and its Python binding) never calls it.

What it computes (GRID, Def. 4): for a configuration with current output w,
bit t of the mask is 1 iff t is neither EOS nor special and w.bytes(t) is a
viable prefix of the constrained language L (Def. 2); the EOS bit is 1 iff w is
a complete sentence of L (Sec. 3.2, "EOS gating").  It follows the paper's own
executable-specification shape (Sec. 6.1): a brute-force trial parse of every
token, one byte at a time, from a copy of the configuration -- no trie, no
CI/CD split, no caching, no table compression.

Modules:
  regex.py    regular lexeme languages R_tau -> Thompson NFA -> union DFA (Sec. 2, L1)
  grammar.py  grammar text, L2 role projection, useless-symbol elimination (Sec. 2)
  lr1.py      canonical LR(1) tables (any LR(1) construction has the correct-prefix
              property that Prop. 3 relies on)
  core.py     configurations, maximal-munch contextual lexing, allowed-terminal
              simulation, trailing liveness, EOS gate, the mask (Sec. 3.2, 4.1)

Pins (tests/test_oracle_*.py) tie each part to something other than itself:
Python's ``re`` for the DFA, a textbook Earley recognizer for the LR(1) tables,
exhaustive brute force over short byte strings for the mask and the EOS bit, and
the worked example of Sec. 7.1.
"""
from .core import OracleGrammar, compile_grammar, Config  # noqa: F401
