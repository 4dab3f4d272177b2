"""Seeded synthetic inputs shared by the tests and the benchmark.

This package only *generates* inputs: grammar texts (read from ``grammars/``),
schema lexicons, byte-level vocabularies, sentence prefixes and logits.  It
contains none of the masking method's arithmetic (no lexing, parsing or mask
logic), so the CPU oracle and the CUDA path can both consume its outputs while
sharing no code with each other.

The paper's own workloads (Spider, JSONSchemaBench, the gpt2/Qwen tokenizers)
are not available; every generator here reproduces only their *shape* (vocab
sizes, token-length mix, prefix lengths, nesting depths), from a seed.
"""
import os

GRAMMAR_DIR = os.path.join(os.path.dirname(os.path.abspath(__file__)), "grammars")


def grammar_text(name: str) -> str:
    """Return the text of ``grammars/<name>.grid``."""
    with open(os.path.join(GRAMMAR_DIR, name + ".grid"), "r", encoding="utf-8") as f:
        return f.read()


def grammar_keywords(text: str):
    """Alphabetic literal terminals of a grammar file (used to keep generated
    identifiers disjoint from keywords).  Plain text scan of '%token NAME "lit"'."""
    out = []
    for line in text.splitlines():
        parts = line.split()
        if len(parts) >= 3 and parts[0] == "%token" and parts[2].startswith('"'):
            lit = parts[2].strip('"')
            if lit.isalpha():
                out.append(lit)
    return out
