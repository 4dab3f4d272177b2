"""Thin ctypes binding of libgrid (include/grid.h).

Argument marshalling only: every step of the mask path runs in the CUDA
library.  Functions keep the C names; the small classes own the opaque handles
and free them.  Device buffers are torch CUDA tensors (masks are int32 tensors
holding the uint32 words); streams default to torch's current stream.  If the
shared library has not been built, every call raises ``GridLibraryMissing``:
there is no fallback.
"""
from __future__ import annotations

import ctypes
import os

from .build import library_path

GRID_OK = 0
GRID_ST = {0: "OK", 1: "NONVIABLE", 2: "STACK_OVERFLOW", 3: "TOKEN_NOT_ALLOWED",
           4: "EMPTY_MASK", 5: "BOUND", 6: "COMPLETE"}
GRID_ST_OK, GRID_ST_NONVIABLE, GRID_ST_STACK_OVERFLOW, GRID_ST_TOKEN_NOT_ALLOWED = 0, 1, 2, 3
GRID_ST_EMPTY_MASK, GRID_ST_BOUND, GRID_ST_COMPLETE = 4, 5, 6
GRID_DTYPE_F32, GRID_DTYPE_BF16 = 0, 1

EXPORTED = ["grid_last_error", "grid_compile", "grid_grammar_free", "grid_grammar_info", "grid_grammar_lexicon_trie",
            "grid_load_vocab", "grid_vocab_free", "grid_vocab_info", "grid_specialize",
            "grid_spec_free", "grid_spec_info", "grid_configs_create", "grid_configs_free", "grid_configs_reset",
            "grid_advance", "grid_masks", "grid_masks_apply", "grid_advance_masks", "grid_configs_set_events", "grid_spec_set_work_counters", "grid_masks_static", "grid_forced_span",
            "grid_reserve", "grid_cache_create", "grid_cache_free", "grid_cache_clear", "grid_cache_stats",
            "grid_masks_cached", "grid_configs_enable_audit", "grid_audit_append", "grid_audit_seal", "grid_audit_head", "grid_audit_verify",
            "grid_audit_genesis", "grid_blake2b", "grid_fingerprint", "grid_apply_mask", "grid_configs_export"]


class GridLibraryMissing(RuntimeError):
    pass


class GridError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__("libgrid error %d: %s" % (code, msg))
        self.code = code


class _Lexicon(ctypes.Structure):
    _fields_ = [("category", ctypes.c_char_p), ("words", ctypes.c_void_p),
                ("offsets", ctypes.c_void_p), ("n_words", ctypes.c_int32)]


class _Options(ctypes.Structure):
    _fields_ = [("max_depth", ctypes.c_int32), ("reserved", ctypes.c_int32 * 7)]


_lib = None


def lib():
    """Load the in-tree libgrid.so (built by ``__graft_entry__.build()``)."""
    global _lib
    if _lib is not None:
        return _lib
    path = library_path()
    if not os.path.exists(path):
        raise GridLibraryMissing("libgrid.so not built at %s: run __graft_entry__.build()" % path)
    L = ctypes.CDLL(path)
    P, I32, I64, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
    sig = {
        "grid_last_error": (SZ, [ctypes.c_char_p, SZ]),
        "grid_compile": (I32, [ctypes.c_char_p, SZ, ctypes.c_char_p, P, I32, P, ctypes.POINTER(P)]),
        "grid_grammar_free": (None, [P]),
        "grid_grammar_info": (I32, [P, ctypes.POINTER(I64)]),
        "grid_grammar_lexicon_trie": (I32, [P, P, P, P, P, P, I64]),
        "grid_load_vocab": (I32, [P, P, I32, I32, P, I32, ctypes.POINTER(P)]),
        "grid_vocab_free": (None, [P]),
        "grid_vocab_info": (I32, [P, ctypes.POINTER(I64)]),
        "grid_specialize": (I32, [P, P, P, ctypes.POINTER(P)]),
        "grid_spec_free": (None, [P]),
        "grid_spec_info": (I32, [P, ctypes.POINTER(I64)]),
        "grid_configs_create": (I32, [P, I32, ctypes.POINTER(P)]),
        "grid_configs_free": (None, [P]),
        "grid_configs_reset": (I32, [P, P, P]),
        "grid_advance": (I32, [P, P, P, P, I32, P, P]),
        "grid_masks": (I32, [P, P, P, P, P]),
        "grid_masks_apply": (I32, [P, P, P, P, P, I32, I64, P]),
        "grid_advance_masks": (I32, [P, P, P, P, P, I32, P, P, P, I32, I64, P]),
        "grid_forced_span": (I32, [P, P, I32, P, P, P, P, P, P]),
        "grid_reserve": (I32, [P, P, P, P, I32, P, P, I32, P, P]),
        "grid_cache_create": (I32, [P, I32, ctypes.POINTER(P)]),
        "grid_cache_free": (None, [P]),
        "grid_cache_clear": (I32, [P, P]),
        "grid_cache_stats": (I32, [P, ctypes.POINTER(I64)]),
        "grid_masks_cached": (I32, [P, P, P, P, P, P, I32, I64, P]),
        "grid_configs_enable_audit": (I32, [P, P, P]),
        "grid_audit_append": (I32, [P, P, P, P, I32, P, P]),
        "grid_audit_seal": (I32, [P, P, P, ctypes.c_uint32, P, P]),
        "grid_audit_head": (I32, [P, I32, P, ctypes.POINTER(ctypes.c_uint64)]),
        "grid_audit_verify": (I64, [P, I64, P]),
        "grid_audit_genesis": (I32, [P]),
        "grid_blake2b": (I32, [P, SZ, P, I32]),
        "grid_fingerprint": (I32, [P, P, P, P]),
        "grid_configs_set_events": (I32, [P, P, I32]),
        "grid_spec_set_work_counters": (I32, [P, P]),
        "grid_masks_static": (I32, [P, P, P, P, P, P, I32, I32, P, P, P]),
        "grid_apply_mask": (I32, [P, P, I32, I32, I32, I64, P]),
        "grid_configs_export": (I32, [P, I32, P, I32, P, P, P, P]),
    }
    for name, (res, args) in sig.items():
        f = getattr(L, name)
        f.restype = res
        f.argtypes = args
    _lib = L
    return L


def last_error() -> str:
    buf = ctypes.create_string_buffer(4096)
    lib().grid_last_error(buf, 4096)
    return buf.value.decode(errors="replace")


def _check(rc):
    if rc != GRID_OK:
        raise GridError(rc, last_error())


def _stream(stream):
    if stream is None:
        import torch
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr())


def _i32(*xs):
    """Each tensor is a contiguous int32 CUDA tensor."""
    import torch
    for x in xs:
        assert x.is_contiguous() and x.is_cuda and x.dtype == torch.int32, "contiguous int32 CUDA tensor expected"


def _u8_records(records):
    import torch
    assert records.is_contiguous() and records.is_cuda and records.dtype == torch.uint8 and records.shape[-1] == 80, \
        "uint8 CUDA records [..., 80] expected"


def _pack(items):
    """list of bytes -> (contiguous buffer, int64 offsets) kept alive by the caller."""
    import numpy as np
    data = b"".join(items)
    offs = np.zeros(len(items) + 1, dtype=np.int64)
    if items:
        np.cumsum(np.fromiter(map(len, items), dtype=np.int64, count=len(items)), out=offs[1:])
    buf = ctypes.create_string_buffer(data, max(1, len(data)))
    return buf, np.ctypeslib.as_ctypes(offs)


# ---------------------------------------------------------------------------
def grid_compile(text: str, role_keep=None, lexicons=None, max_depth: int = 4096):
    """Returns a grid_grammar handle (c_void_p).  ``role_keep`` is None (all
    productions) or a list of kept production tags; ``lexicons`` maps a
    category terminal name to its word list."""
    L = lib()
    raw = text.encode()
    keep = None if role_keep is None else ",".join(role_keep).encode()
    lex = lexicons or {}
    arr = (_Lexicon * max(1, len(lex)))()
    keep_alive = []
    for i, (cat, words) in enumerate(lex.items()):
        ws = [w if isinstance(w, bytes) else w.encode() for w in words]
        buf, offs = _pack(ws)
        c = cat.encode()
        keep_alive += [buf, offs, c]
        arr[i].category = c
        arr[i].words = ctypes.cast(buf, ctypes.c_void_p)
        arr[i].offsets = ctypes.cast(offs, ctypes.c_void_p)
        arr[i].n_words = len(ws)
    opt = _Options(max_depth, (ctypes.c_int32 * 7)())
    out = ctypes.c_void_p()
    _check(L.grid_compile(raw, len(raw), keep, ctypes.cast(arr, ctypes.c_void_p), len(lex),
                          ctypes.byref(opt), ctypes.byref(out)))
    return out


def grid_grammar_info(g):
    out = (ctypes.c_int64 * 8)()
    _check(lib().grid_grammar_info(g, out))
    keys = ["terminals", "lalr_states", "nonterminals", "productions", "dfa_states",
            "byte_classes", "lexicon_nodes", "categories"]
    return dict(zip(keys, list(out)))


def grid_grammar_lexicon_trie(g):
    """The identifier trie's arrays (numpy): cstart, cbyte, cnode, pcats, wcats."""
    import numpy as np
    n = grid_grammar_info(g)["lexicon_nodes"]
    cstart = np.zeros(n + 1, np.int32)
    cbyte = np.zeros(max(1, n - 1), np.uint8)
    cnode = np.zeros(max(1, n - 1), np.int32)
    pc = np.zeros(n, np.uint32)
    wc = np.zeros(n, np.uint32)
    p = lambda a: a.ctypes.data_as(ctypes.c_void_p)
    _check(lib().grid_grammar_lexicon_trie(g, p(cstart), p(cbyte), p(cnode), p(pc), p(wc), n))
    return cstart, cbyte[:max(0, n - 1)], cnode[:max(0, n - 1)], pc, wc


def grid_load_vocab(tokens, eos: int, specials=()):
    L = lib()
    buf, offs = _pack(tokens)
    sp = (ctypes.c_int32 * max(1, len(specials)))(*specials)
    out = ctypes.c_void_p()
    _check(L.grid_load_vocab(ctypes.cast(buf, ctypes.c_void_p), ctypes.cast(offs, ctypes.c_void_p),
                             len(tokens), eos, ctypes.cast(sp, ctypes.c_void_p), len(specials),
                             ctypes.byref(out)))
    return out


def grid_vocab_info(v):
    out = (ctypes.c_int64 * 4)()
    _check(lib().grid_vocab_info(v, out))
    return dict(zip(["V", "spellings", "byte_complete", "bytes"], list(out)))


def grid_specialize(g, v, stream=None):
    out = ctypes.c_void_p()
    _check(lib().grid_specialize(g, v, _stream(stream), ctypes.byref(out)))
    return out


def grid_spec_info(spec):
    out = (ctypes.c_int64 * 8)()
    _check(lib().grid_spec_info(spec, out))
    keys = ["ci_tables", "ci_classes", "cd_start", "cd_total", "staged_bytes", "verdict_classes",
            "flags", "spellings"]
    d = dict(zip(keys, list(out)))
    d["ci_on"] = d["flags"] & 1
    d["vc_in_codes"] = (d["flags"] >> 1) & 1
    return d


def grid_configs_create(spec, B: int):
    out = ctypes.c_void_p()
    _check(lib().grid_configs_create(spec, B, ctypes.byref(out)))
    return out


def grid_configs_reset(spec, cfg, stream=None):
    _check(lib().grid_configs_reset(spec, cfg, _stream(stream)))


def grid_advance(spec, cin, cout, tokens, status, stream=None):
    """tokens: int32 CUDA tensor [B] or [B, n_steps]; status: int32 CUDA tensor [B].
    ``cin`` / ``cout`` are handles, or Configs objects (then B is checked)."""
    import torch
    n = 1 if tokens.dim() == 1 else tokens.shape[1]
    assert tokens.is_contiguous() and status.is_contiguous() and tokens.is_cuda and status.is_cuda
    assert tokens.dtype == torch.int32 and status.dtype == torch.int32 and tokens.dim() in (1, 2)
    B = getattr(cout, "B", None)
    assert B is None or (tokens.shape[0] == B and tuple(status.shape) == (B,)), "tokens [B] or [B, n], status [B]"
    _check(lib().grid_advance(getattr(spec, "h", spec), getattr(cin, "h", cin), getattr(cout, "h", cout),
                              _ptr(tokens), n, _ptr(status), _stream(stream)))


def grid_masks(spec, cfg, mask, status, stream=None):
    """mask: int32 CUDA tensor [B, ceil(V/32)] (uint32 words); status: int32 [B].
    ``spec`` and ``cfg`` are handles, or Spec / Configs objects (then the
    shapes are checked against V and B)."""
    import torch
    assert mask.is_contiguous() and status.is_contiguous() and mask.is_cuda and status.is_cuda
    assert mask.dtype == torch.int32 and status.dtype == torch.int32 and mask.dim() == 2
    B, W = getattr(cfg, "B", None), getattr(spec, "W", None)
    assert B is None or (mask.shape[0] == B and tuple(status.shape) == (B,)), "mask [B, W] and status [B] expected"
    assert W is None or mask.shape[1] == W, "mask [B, ceil(V/32)] expected"
    _check(lib().grid_masks(getattr(spec, "h", spec), getattr(cfg, "h", cfg), _ptr(mask), _ptr(status),
                            _stream(stream)))


def grid_masks_apply(spec, cfg, mask, status, logits, stream=None):
    """grid_masks plus the -inf fill of ``logits`` (float32 or bfloat16 CUDA
    tensor [B, >=V], unit stride along V) in the same pass."""
    import torch
    dt = {torch.float32: GRID_DTYPE_F32, torch.bfloat16: GRID_DTYPE_BF16}[logits.dtype]
    assert mask.is_contiguous() and status.is_contiguous() and mask.is_cuda and status.is_cuda and logits.is_cuda
    assert mask.dtype == torch.int32 and status.dtype == torch.int32 and mask.dim() == 2 and logits.dim() == 2
    assert logits.stride(1) == 1 and logits.shape[0] == mask.shape[0]
    B, W = getattr(cfg, "B", None), getattr(spec, "W", None)
    assert B is None or (mask.shape[0] == B and tuple(status.shape) == (B,)), "mask [B, W] and status [B] expected"
    assert W is None or mask.shape[1] == W, "mask [B, ceil(V/32)] expected"
    _check(lib().grid_masks_apply(getattr(spec, "h", spec), getattr(cfg, "h", cfg), _ptr(mask), _ptr(status),
                                  _ptr(logits), dt, logits.stride(0), _stream(stream)))


def grid_advance_masks(spec, cin, cout, tokens, mask, status, logits=None, stream=None, cache=None):
    """grid_advance of ``tokens`` (int32 CUDA tensor [B] or [B, n_steps]) from
    cin into cout, then the masks of cout (and, with ``logits``, their -inf
    fill) in one launch sequence, through ``cache`` (a Cache) if given;
    status: the advance's error for a row whose token was refused, else the
    mask step's."""
    import torch
    n = 1 if tokens.dim() == 1 else tokens.shape[1]
    assert tokens.is_contiguous() and tokens.dtype == torch.int32 and tokens.is_cuda
    assert mask.is_contiguous() and status.is_contiguous() and mask.dtype == torch.int32
    assert status.dtype == torch.int32 and mask.is_cuda and status.is_cuda and mask.dim() == 2
    B, W = getattr(cout, "B", None), getattr(spec, "W", None)
    assert B is None or (mask.shape[0] == B and tuple(status.shape) == (B,) and tokens.shape[0] == B), \
        "tokens [B] or [B, n], mask [B, W] and status [B] expected"
    assert W is None or mask.shape[1] == W, "mask [B, ceil(V/32)] expected"
    spec, cin, cout = getattr(spec, "h", spec), getattr(cin, "h", cin), getattr(cout, "h", cout)
    lp, dt, stride = ctypes.c_void_p(None), GRID_DTYPE_F32, 0
    if logits is not None:
        dt = {torch.float32: GRID_DTYPE_F32, torch.bfloat16: GRID_DTYPE_BF16}[logits.dtype]
        assert logits.is_cuda and logits.dim() == 2 and logits.stride(1) == 1
        assert B is None or logits.shape[0] == B, "logits [B, >=V] expected"
        lp, stride = _ptr(logits), logits.stride(0)
    ch = ctypes.c_void_p(None) if cache is None else getattr(cache, "h", cache)
    _check(lib().grid_advance_masks(spec, cin, cout, ch, _ptr(tokens), n, _ptr(mask), _ptr(status), lp, dt, stride,
                                    _stream(stream)))


def grid_forced_span(spec, cfg, max_span, mask, span, span_len, status, records=None, stream=None):
    """Jump-forward: span int32 CUDA tensor [B, max_span], span_len and status
    int32 [B], mask int32 [B, W] (the final configurations' masks); with audit
    on, records is a uint8 CUDA tensor [B, max_span, 80]."""
    _i32(mask, span, span_len, status)
    assert span.dim() == 2 and span.shape[1] == max_span and mask.dim() == 2
    assert span.shape[0] == mask.shape[0] == span_len.shape[0] == status.shape[0], "one row per configuration"
    rp = ctypes.c_void_p(None) if records is None else _ptr(records)
    if records is not None:
        _u8_records(records)
        assert records.numel() == span.shape[0] * max_span * 80
    _check(lib().grid_forced_span(spec, cfg, max_span, _ptr(mask), _ptr(span), _ptr(span_len), _ptr(status), rp,
                                  _stream(stream)))


def grid_reserve(spec, cfg, cost, tokens, status, budget=None, safety=0, fire=None, stream=None):
    """cost, status (and budget, fire) int32 CUDA tensors [B]; tokens int32 [B, cap]."""
    _i32(cost, tokens, status, *[x for x in (budget, fire) if x is not None])
    assert tokens.dim() == 2 and cost.shape[0] == tokens.shape[0] == status.shape[0], "one row per configuration"
    assert all(x.shape[0] == cost.shape[0] for x in (budget, fire) if x is not None)
    nul = ctypes.c_void_p(None)
    _check(lib().grid_reserve(spec, cfg, _ptr(cost), _ptr(tokens), tokens.shape[1], _ptr(status),
                              nul if budget is None else _ptr(budget), safety, nul if fire is None else _ptr(fire),
                              _stream(stream)))


def grid_masks_cached(spec, cfg, cache, mask, status, logits=None, stream=None):
    """grid_masks (logits None) or grid_masks_apply through a mask cache."""
    _i32(mask, status)
    assert mask.dim() == 2 and mask.shape[0] == status.shape[0]
    B, W = getattr(cfg, "B", None), getattr(spec, "W", None)
    assert B is None or mask.shape[0] == B, "mask [B, W] and status [B] expected"
    assert W is None or mask.shape[1] == W, "mask [B, ceil(V/32)] expected"
    if logits is None:
        lp, dt, stride = ctypes.c_void_p(None), GRID_DTYPE_F32, 0
    else:
        import torch
        assert logits.stride(1) == 1 and logits.is_cuda and logits.dim() == 2 and logits.shape[0] == mask.shape[0]
        lp, stride = _ptr(logits), logits.stride(0)
        dt = {torch.float32: GRID_DTYPE_F32, torch.bfloat16: GRID_DTYPE_BF16}[logits.dtype]
    _check(lib().grid_masks_cached(getattr(spec, "h", spec), getattr(cfg, "h", cfg), getattr(cache, "h", cache),
                                   _ptr(mask), _ptr(status), lp, dt, stride, _stream(stream)))


class Cache:
    """A configuration-keyed mask cache of a spec (n_entries a power of two)."""

    def __init__(self, spec, n_entries=1024):
        self.spec = spec
        out = ctypes.c_void_p()
        _check(lib().grid_cache_create(spec.h, n_entries, ctypes.byref(out)))
        self.h = out

    def clear(self, stream=None):
        _check(lib().grid_cache_clear(self.h, _stream(stream)))

    def stats(self):
        out = (ctypes.c_int64 * 4)()
        _check(lib().grid_cache_stats(self.h, out))
        return dict(zip(["lookups", "hits", "fills", "ready"], list(out)))

    def __del__(self):
        if getattr(self, "h", None) and _lib is not None:
            _lib.grid_cache_free(self.h)
            self.h = None


def grid_configs_enable_audit(spec, cfg, stream=None):
    _check(lib().grid_configs_enable_audit(spec, cfg, _stream(stream)))


def grid_audit_append(spec, cfg, mask, tokens, kind, records, stream=None):
    """records: uint8 CUDA tensor [B, 80]; tokens int32 [B] (-1 = no record)."""
    _u8_records(records)
    _i32(mask, tokens)
    _check(lib().grid_audit_append(spec, cfg, _ptr(mask), _ptr(tokens), kind, _ptr(records), _stream(stream)))


def grid_audit_seal(spec, cfg, reason, mode_flags, records, stream=None):
    _u8_records(records)
    _i32(reason)
    _check(lib().grid_audit_seal(spec, cfg, _ptr(reason), mode_flags, _ptr(records), _stream(stream)))


def grid_audit_head(cfg, row):
    head = (ctypes.c_uint8 * 16)()
    n = ctypes.c_uint64()
    _check(lib().grid_audit_head(cfg, row, head, ctypes.byref(n)))
    return bytes(head), n.value


def grid_audit_verify(records: bytes, genesis: bytes | None = None) -> int:
    """records: the concatenated 80-byte records of one row, in order."""
    assert len(records) % 80 == 0
    buf = ctypes.create_string_buffer(bytes(records), max(1, len(records)))
    g = None if genesis is None else ctypes.create_string_buffer(genesis, 16)
    r = lib().grid_audit_verify(buf, len(records) // 80, g)
    if r < -1:
        _check(int(r))
    return int(r)


def grid_audit_genesis() -> bytes:
    out = (ctypes.c_uint8 * 16)()
    _check(lib().grid_audit_genesis(out))
    return bytes(out)


def grid_blake2b(data: bytes, out_bytes: int = 64) -> bytes:
    out = (ctypes.c_uint8 * out_bytes)()
    buf = ctypes.create_string_buffer(data, max(1, len(data)))
    _check(lib().grid_blake2b(buf, len(data), out, out_bytes))
    return bytes(out)


def grid_fingerprint(grammar=None, vocab=None, spec=None) -> bytes:
    out = (ctypes.c_uint8 * 16)()
    h = lambda x: None if x is None else getattr(x, "h", x)
    _check(lib().grid_fingerprint(h(grammar), h(vocab), h(spec), out))
    return bytes(out)


def grid_configs_set_events(cfg, events):
    """events: 5 torch.cuda.Event(enable_timing=True) recorded around the four
    kernels of every later grid_masks on cfg; an empty list stops it."""
    arr = (ctypes.c_void_p * max(1, len(events)))(*[e.cuda_event for e in events])
    _check(lib().grid_configs_set_events(cfg, ctypes.cast(arr, ctypes.c_void_p), len(events)))


def grid_spec_set_work_counters(spec, counters):
    """counters: int64 CUDA tensor [6] (zeroed by the caller), or None to stop."""
    if counters is not None:
        assert counters.is_cuda and counters.numel() >= 6 and counters.element_size() == 8
    _check(lib().grid_spec_set_work_counters(spec, ctypes.c_void_p(None) if counters is None else _ptr(counters)))


def grid_masks_static(spec, stack, depth, dfa_state, lex_node, flags, mask, status, stream=None):
    """grid_masks for callers that cannot allocate: the configurations come as
    device arrays the caller owns (stack: int16/uint16 CUDA tensor [B, max_depth]
    holding uint16 LALR states; depth, dfa_state, lex_node, flags: int32 [B]),
    and the step's scratch is the library's fixed static device area.  ``spec``
    is a Spec (then the mask's width is checked too) or its handle."""
    import torch
    B = depth.shape[0]
    dev = stack.device
    for x in (stack, depth, dfa_state, lex_node, flags, mask, status):
        assert x.is_contiguous() and x.is_cuda and x.device == dev, "device tensors on one device expected"
    for x in (depth, dfa_state, lex_node, flags, status):
        assert x.dtype == torch.int32 and tuple(x.shape) == (B,), "int32 [B] expected"
    assert stack.dim() == 2 and stack.shape[0] == B and stack.element_size() == 2
    W = getattr(spec, "W", None)
    assert mask.dtype == torch.int32 and mask.dim() == 2 and mask.shape[0] == B, "int32 [B, ceil(V/32)] mask expected"
    assert W is None or mask.shape[1] == W, "int32 [B, ceil(V/32)] mask expected"
    spec = getattr(spec, "h", spec)
    _check(lib().grid_masks_static(spec, _ptr(stack), _ptr(depth), _ptr(dfa_state), _ptr(lex_node), _ptr(flags),
                                   B, stack.shape[1], _ptr(mask), _ptr(status), _stream(stream)))


def grid_apply_mask(mask, logits, stream=None):
    """In place on a float32 or bfloat16 CUDA tensor [B, >=V] (row stride = stride(0))."""
    import torch
    dt = {torch.float32: GRID_DTYPE_F32, torch.bfloat16: GRID_DTYPE_BF16}[logits.dtype]
    B, V = logits.shape
    assert logits.stride(1) == 1 and logits.is_cuda
    assert mask.is_contiguous() and mask.is_cuda and mask.dtype == torch.int32 and mask.dim() == 2
    assert mask.shape[0] == B and mask.shape[1] * 32 >= V, "mask [B, >= ceil(V/32)] for logits [B, V]"
    _check(lib().grid_apply_mask(_ptr(mask), _ptr(logits), dt, B, V, logits.stride(0), _stream(stream)))


def grid_apply_mask_raw(mask, logits_ptr: int, dtype: int, B: int, V: int, row_stride: int, stream=None):
    _check(lib().grid_apply_mask(_ptr(mask), ctypes.c_void_p(logits_ptr), dtype, B, V, row_stride,
                                 _stream(stream)))


def grid_configs_export(cfg, row: int, cap: int = 1 << 16):
    stack = (ctypes.c_int32 * cap)()
    d, q, lx, fl = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
    _check(lib().grid_configs_export(cfg, row, stack, cap, ctypes.byref(d), ctypes.byref(q),
                                     ctypes.byref(lx), ctypes.byref(fl)))
    return dict(stack=list(stack[:min(d.value, cap)]), depth=d.value, dfa_state=q.value,
                lex_node=lx.value, flags=fl.value)


# ---------------------------------------------------------------------------
class Grammar:
    def __init__(self, text, role_keep=None, lexicons=None, max_depth=4096):
        self.h = grid_compile(text, role_keep, lexicons, max_depth)

    def info(self):
        return grid_grammar_info(self.h)

    def __del__(self):
        if getattr(self, "h", None) and _lib is not None:
            _lib.grid_grammar_free(self.h)
            self.h = None


class Vocab:
    def __init__(self, tokens, eos, specials=()):
        self.V = len(tokens)
        self.eos = eos
        self.h = grid_load_vocab(tokens, eos, specials)

    def info(self):
        return grid_vocab_info(self.h)

    def __del__(self):
        if getattr(self, "h", None) and _lib is not None:
            _lib.grid_vocab_free(self.h)
            self.h = None


class Spec:
    """(grammar, vocabulary) tables on the device plus the CI classes."""

    def __init__(self, grammar: Grammar, vocab: Vocab, stream=None):
        self.grammar, self.vocab = grammar, vocab
        self.V = vocab.V
        self.W = (vocab.V + 31) // 32
        self.h = grid_specialize(grammar.h, vocab.h, stream)

    def info(self):
        return grid_spec_info(self.h)

    def __del__(self):
        if getattr(self, "h", None) and _lib is not None:
            _lib.grid_spec_free(self.h)
            self.h = None


class Configs:
    def __init__(self, spec: Spec, B: int):
        self.spec, self.B = spec, B
        self.h = grid_configs_create(spec.h, B)

    def reset(self, stream=None):
        grid_configs_reset(self.spec.h, self.h, stream)

    def export(self, row):
        return grid_configs_export(self.h, row)

    def __del__(self):
        if getattr(self, "h", None) and _lib is not None:
            _lib.grid_configs_free(self.h)
            self.h = None
