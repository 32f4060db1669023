"""fp64 CPU oracle of the verify step (test infrastructure).

This package is test infrastructure: only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import it.  The product path (the CUDA
library and its binding) never loads it, and it imports nothing from the product.

It wraps ``oracle.cpp`` (a plain fp64 statement of the verify step of lossless
Psi-Spec decoding: Sec. 4.2 and Appendix B.3, Algorithm "Lossless Psi-Spec decoding
(Linear Sampler)") with ``ctypes``.  Arrays go in and out as numpy arrays; bf16
tensors travel as their uint16 bit patterns.

Every function of ``oracle.cpp`` is pinned by ``tests/test_oracle_*.py`` against
facts the paper and the mathematics fix (exact losslessness by enumeration, the
closed-form acceptance rate, chi-square, special cases, dense-attention brute force).
"""

from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.cpp")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``oracle.cpp`` into ``liboracle.so`` (plain g++, -O2, no fast-math)."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["g++", "-std=c++17", "-O2", "-fno-fast-math", "-ffp-contract=off", "-fPIC",
           "-shared", "-pthread", _SRC, "-o", tmp]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            i32, i64, f64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
            lib.oracle_hardware_threads.restype = ctypes.c_int
            lib.oracle_softmax.argtypes = [P, i64, f64, P]
            lib.oracle_softmax.restype = ctypes.c_int
            lib.oracle_argmax.argtypes = [P, i64]
            lib.oracle_argmax.restype = i64
            lib.oracle_inverse_cdf.argtypes = [P, i64, f64, P]
            lib.oracle_inverse_cdf.restype = i64
            lib.oracle_accept_probs.argtypes = [i32, i64, P, P, P, P, i32, P, P, P, P, P, P, P]
            lib.oracle_accept_probs.restype = ctypes.c_int
            lib.oracle_accept_probs_many.argtypes = [i64, i32, i64, P, P, P, P, i32, P, P, P,
                                                     i32]
            lib.oracle_accept_probs_many.restype = ctypes.c_int
            lib.oracle_accept_block.argtypes = [i32, i32, i64, i32, P, P, P, P, P, P, P, P,
                                                P, P, P, P, i32]
            lib.oracle_accept_block.restype = ctypes.c_int
            lib.oracle_sample_block.argtypes = [i32, i32, i64, i32, P, P, P, P, P, P, P, P, P, P,
                                                i32]
            lib.oracle_sample_block.restype = ctypes.c_int
            lib.oracle_filter_row.argtypes = [P, i64, i32, f64, P, P]
            lib.oracle_filter_row.restype = ctypes.c_int
            lib.oracle_accept_block_filtered.argtypes = [i32, i32, i64, i32, P, P, P, P, P, P,
                                                         P, P, P, P, P, P, P, P, P, i32]
            lib.oracle_accept_block_filtered.restype = ctypes.c_int
            lib.oracle_verify_attention.argtypes = [i32, i32, i32, i32, i32, i32, i32, i32, f64,
                                                    P, P, P, P, P, P, P, P, i64, P, i32]
            lib.oracle_verify_attention.restype = ctypes.c_int
            lib.oracle_verify_attention_tree.argtypes = [i32, i32, i32, i32, i32, i32, i32, i32,
                                                         f64, P, P, P, P, P, P, P, P, P, i64, P,
                                                         i32]
            lib.oracle_verify_attention_tree.restype = ctypes.c_int
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def hardware_threads() -> int:
    return int(_load().oracle_hardware_threads())


def softmax(logits, temperature: float):
    """softmax(logits / T) of one row in fp64; raises on an undefined row."""
    lib = _load()
    l = _c(logits, np.float64)
    p = np.empty_like(l)
    rc = lib.oracle_softmax(_ptr(l), l.size, float(temperature), _ptr(p))
    if rc:
        raise ValueError("softmax undefined for this row")
    return p


def argmax(row) -> int:
    r = _c(row, np.float64)
    return int(_load().oracle_argmax(_ptr(r), r.size))


def inverse_cdf(weights, u: float):
    """(token, margin) of the inverse-CDF draw from unnormalised weights."""
    w = _c(weights, np.float64)
    m = np.zeros(1, np.float64)
    x = _load().oracle_inverse_cdf(_ptr(w), w.size, float(u), _ptr(m))
    return int(x), float(m[0])


def accept_probs(p_rows, q_rows, tokens, uniforms, greedy: bool = False):
    """The verify decision of one sequence on fp64 probability rows.

    Returns a dict with n, out_tokens, num_emitted, p_tok, q_tok, accept_margin,
    sample_margin (see ``oracle_accept_probs`` in oracle.cpp).
    """
    lib = _load()
    p = _c(p_rows, np.float64)
    gamma, vocab = p.shape
    q = None if greedy and q_rows is None else _c(q_rows, np.float64)
    t = _c(tokens, np.int32)
    u = _c(uniforms, np.float64)
    n = np.zeros(1, np.int32)
    ne = np.zeros(1, np.int32)
    out = np.empty(gamma + 1, np.int32)
    ptok = np.empty(gamma, np.float64)
    qtok = np.empty(gamma, np.float64)
    am = np.empty(gamma, np.float64)
    sm = np.empty(1, np.float64)
    rc = lib.oracle_accept_probs(gamma, vocab, _ptr(p), _ptr(q), _ptr(t), _ptr(u),
                                 1 if greedy else 0, _ptr(n), _ptr(out), _ptr(ne),
                                 _ptr(ptok), _ptr(qtok), _ptr(am), _ptr(sm))
    if rc:
        raise ValueError("token id out of range")
    return dict(n=int(n[0]), out_tokens=out, num_emitted=int(ne[0]), p_tok=ptok, q_tok=qtok,
                accept_margin=am, sample_margin=float(sm[0]))


def accept_probs_many(p_rows, q_rows, tokens, uniforms, greedy: bool = False,
                      nthreads: int = 0, lib=None):
    """accept_probs for many (tokens, uniforms) cases sharing the same rows.

    tokens: int [count][gamma]; uniforms: float [count][gamma].
    Returns (n [count], out_tokens [count][gamma+1], num_emitted [count]).
    ``lib`` optionally substitutes another build of oracle.cpp (mutation tests).
    """
    lib = lib or _load()
    p = _c(p_rows, np.float64)
    gamma, vocab = p.shape
    q = _c(q_rows, np.float64) if q_rows is not None else None
    t = _c(tokens, np.int32).reshape(-1, gamma)
    u = _c(uniforms, np.float64).reshape(-1, gamma)
    count = t.shape[0]
    n = np.empty(count, np.int32)
    ne = np.empty(count, np.int32)
    out = np.empty((count, gamma + 1), np.int32)
    rc = lib.oracle_accept_probs_many(count, gamma, vocab, _ptr(p), _ptr(q), _ptr(t), _ptr(u),
                                      1 if greedy else 0, _ptr(n), _ptr(out), _ptr(ne),
                                      int(nthreads))
    if rc:
        raise ValueError("token id out of range")
    return n, out, ne


def load_variant(src_text: str, tag: str):
    """Compile a modified copy of oracle.cpp (tests plant mistakes this way) and load it."""
    import tempfile
    d = tempfile.mkdtemp(prefix=f"oracle_{tag}_")
    src = os.path.join(d, "oracle.cpp")
    so = os.path.join(d, "liboracle.so")
    with open(src, "w") as f:
        f.write(src_text)
    subprocess.run(["g++", "-std=c++17", "-O1", "-fPIC", "-shared", "-pthread", src, "-o", so],
                   check=True)
    lib = ctypes.CDLL(so)
    P = ctypes.c_void_p
    i32, i64 = ctypes.c_int32, ctypes.c_int64
    lib.oracle_accept_probs_many.argtypes = [i64, i32, i64, P, P, P, P, i32, P, P, P, i32]
    lib.oracle_accept_probs_many.restype = ctypes.c_int
    lib.oracle_accept_block_filtered.argtypes = [i32, i32, i64, i32, P, P, P, P, P, P, P, P,
                                                 P, P, P, P, P, P, P, i32]
    lib.oracle_accept_block_filtered.restype = ctypes.c_int
    return lib


def source_text() -> str:
    with open(_SRC) as f:
        return f.read()


def accept_block(target_logits, drafter_logits, block_tokens, temperature, uniforms,
                 nthreads: int = 0):
    """The acceptance half of the verify step over a batch, from logits.

    target_logits / drafter_logits: [batch][gamma][vocab] float32, or uint16 bf16 bits.
    Returns a dict of numpy arrays: num_accepted, out_tokens, num_emitted, diag,
    accept_margin, sample_margin, status.
    """
    lib = _load()
    tl = np.ascontiguousarray(target_logits)
    dl = np.ascontiguousarray(drafter_logits)
    if tl.dtype == np.float32:
        dtype = 0
    elif tl.dtype == np.uint16:
        dtype = 1
    else:
        raise TypeError("logits must be float32 or uint16 (bf16 bits)")
    if dl.dtype != tl.dtype or dl.shape != tl.shape:
        raise TypeError("target and drafter logits must match in dtype and shape")
    batch, gamma, vocab = tl.shape
    bt = _c(block_tokens, np.int32)
    T = _c(temperature, np.float32)
    u = _c(uniforms, np.float32)
    na = np.empty(batch, np.int32)
    ne = np.empty(batch, np.int32)
    ot = np.empty((batch, gamma + 1), np.int32)
    diag = np.empty((batch, gamma, 2), np.float64)
    am = np.empty((batch, gamma), np.float64)
    sm = np.empty(batch, np.float64)
    st = np.empty(batch, np.int32)
    rc = lib.oracle_accept_block(batch, gamma, vocab, dtype, _ptr(tl), _ptr(dl), _ptr(bt),
                                 _ptr(T), _ptr(u), _ptr(na), _ptr(ot), _ptr(ne), _ptr(diag),
                                 _ptr(am), _ptr(sm), _ptr(st), int(nthreads))
    if rc:
        raise ValueError("invalid arguments to oracle_accept_block")
    return dict(num_accepted=na, out_tokens=ot, num_emitted=ne, diag=diag,
                accept_margin=am, sample_margin=sm, status=st)


def filter_row(p, top_k: int, top_p: float):
    """Top-k then top-p filtering of one probability row; returns (filtered row, margin)."""
    lib = _load()
    pr = _c(p, np.float64)
    out = np.empty_like(pr)
    m = np.empty(1, np.float64)
    rc = lib.oracle_filter_row(_ptr(pr), pr.size, int(top_k), float(top_p), _ptr(out), _ptr(m))
    if rc:
        raise ValueError("top_k must be >= 1 and top_p in (0, 1]")
    return out, float(m[0])


def accept_block_filtered(target_logits, drafter_logits, block_tokens, temperature, top_k, top_p,
                          uniforms, nthreads: int = 0, lib=None):
    """accept_block with top-k / top-p filtering of both distributions (per sequence).

    Returns the accept_block dict plus filter_margin (the smallest top-p margin of the
    rows a sequence uses); status 3 marks a top_k / top_p outside its range.
    """
    lib = lib or _load()
    tl = np.ascontiguousarray(target_logits)
    dl = np.ascontiguousarray(drafter_logits)
    if tl.dtype == np.float32:
        dtype = 0
    elif tl.dtype == np.uint16:
        dtype = 1
    else:
        raise TypeError("logits must be float32 or uint16 (bf16 bits)")
    if dl.dtype != tl.dtype or dl.shape != tl.shape:
        raise TypeError("target and drafter logits must match in dtype and shape")
    batch, gamma, vocab = tl.shape
    bt = _c(block_tokens, np.int32)
    T = _c(temperature, np.float32)
    K = _c(np.broadcast_to(np.asarray(top_k, np.int32), (batch,)), np.int32)
    P = _c(np.broadcast_to(np.asarray(top_p, np.float32), (batch,)), np.float32)
    u = _c(uniforms, np.float32)
    na = np.empty(batch, np.int32)
    ne = np.empty(batch, np.int32)
    ot = np.empty((batch, gamma + 1), np.int32)
    diag = np.empty((batch, gamma, 2), np.float64)
    am = np.empty((batch, gamma), np.float64)
    sm = np.empty(batch, np.float64)
    fm = np.empty(batch, np.float64)
    st = np.empty(batch, np.int32)
    rc = lib.oracle_accept_block_filtered(batch, gamma, vocab, dtype, _ptr(tl), _ptr(dl), _ptr(bt),
                                          _ptr(T), _ptr(K), _ptr(P), _ptr(u), _ptr(na), _ptr(ot),
                                          _ptr(ne), _ptr(diag), _ptr(am), _ptr(sm), _ptr(fm),
                                          _ptr(st), int(nthreads))
    if rc:
        raise ValueError("invalid arguments to oracle_accept_block_filtered")
    return dict(num_accepted=na, out_tokens=ot, num_emitted=ne, diag=diag,
                accept_margin=am, sample_margin=sm, filter_margin=fm, status=st)


def sample_block(drafter_logits, temperature, uniforms, top_k=None, top_p=None,
                 nthreads: int = 0):
    """Draft-side sampling of every block token from its drafter row (see
    ``oracle_sample_block`` in oracle.cpp). Returns a dict of tokens, q_tok, margin,
    filter_margin, status."""
    lib = _load()
    dl = np.ascontiguousarray(drafter_logits)
    if dl.dtype == np.float32:
        dtype = 0
    elif dl.dtype == np.uint16:
        dtype = 1
    else:
        raise TypeError("logits must be float32 or uint16 (bf16 bits)")
    batch, gamma, vocab = dl.shape
    T = _c(temperature, np.float32)
    u = _c(uniforms, np.float32)
    K = P = None
    if top_k is not None:
        K = _c(np.broadcast_to(np.asarray(top_k, np.int32), (batch,)), np.int32)
        P = _c(np.broadcast_to(np.asarray(top_p, np.float32), (batch,)), np.float32)
    tok = np.empty((batch, gamma), np.int32)
    qt = np.empty((batch, gamma), np.float64)
    mg = np.empty((batch, gamma), np.float64)
    fm = np.empty((batch, gamma), np.float64)
    st = np.empty(batch, np.int32)
    rc = lib.oracle_sample_block(batch, gamma, vocab, dtype, _ptr(dl), _ptr(T),
                                 None if K is None else _ptr(K), None if P is None else _ptr(P),
                                 _ptr(u), _ptr(tok), _ptr(qt), _ptr(mg), _ptr(fm), _ptr(st),
                                 int(nthreads))
    if rc:
        raise ValueError("invalid arguments to oracle_sample_block")
    return dict(tokens=tok, q_tok=qt, margin=mg, filter_margin=fm, status=st)


def noise_tokens(words, vocab: int):
    """Alg. line 1 (z ~ U[V], i.i.d.): token = floor(x * V / 2^32) of each 32-bit random
    word x, i.e. the word's position in [0, 1) scaled to the vocabulary."""
    w = np.asarray(words, dtype=np.uint64)
    return ((w * np.uint64(vocab)) >> np.uint64(32)).astype(np.int32)


def commit_kv(kv_len, num_accepted, page_table, page_size: int, gamma: int, free_pages,
              free_count: int, reserve: bool = True):
    """Roll a paged KV cache back to the accepted prefix of a verify step, sequence by
    sequence in batch order (plain loops).

    kv_len[b] = ctx_b + gamma on entry (the block's keys were written for the verify
    pass). The step keeps x^{L+1} and the n-1 accepted drafts (n = num_accepted + 1), so
    kv_len becomes ctx_b + n; a sequence whose step failed (num_accepted = -1) keeps
    ctx_b. The keys past the new length are stale and are overwritten by the next block.
      * reserve: the sequence keeps its pages and pops from the top of the free list the
        pages it lacks for gamma more keys. Requests are served in batch order; request
        b is granted iff the requests of sequences 0..b together fit in the list (a
        refused request still counts against the later ones, so the grants are a prefix
        of the batch order). A refused sequence, or one whose table cannot hold the
        pages, gets none (flag 2; its length is still committed).
      * otherwise (the sequence stops here): pages wholly past the new length are pushed
        onto the free list in batch order, with the same prefix rule against the list's
        capacity; their table entries become -1. A sequence whose pages do not fit keeps
        them (flag 2).
    A sequence with kv_len outside [gamma, max_pages * page_size] or num_accepted outside
    [-1, gamma - 1] is left unchanged (flag 1).

    Returns (kv_len', page_table', free_pages', free_count', flags[b]: 0, 1 or 2)."""
    kv = np.array(kv_len, dtype=np.int64)
    na = np.asarray(num_accepted, dtype=np.int64)
    table = np.array(page_table, dtype=np.int32, copy=True)
    free = np.array(free_pages, dtype=np.int32, copy=True)
    count = int(free_count)
    B, max_pages = table.shape
    new = kv.copy()
    flags = np.zeros(B, np.int32)
    for b in range(B):
        if kv[b] < gamma or kv[b] > max_pages * page_size or na[b] < -1 or na[b] > gamma - 1:
            flags[b] = 1
            continue
        new[b] = kv[b] - gamma + (na[b] + 1 if na[b] >= 0 else 0)
    capacity = len(free)
    asked = 0  # pages requested (reserve) or offered (release) by sequences 0..b-1
    top = count
    for b in range(B):
        if flags[b]:
            continue
        have = -(-int(kv[b]) // page_size)
        if reserve:
            want = -(-int(new[b] + gamma) // page_size)
            if want > max_pages:
                flags[b] = 2
                continue
            need = want - have
            if need > 0 and asked + need > count:
                flags[b] = 2
                asked += need
                continue
            for i in range(need):
                table[b, have + i] = free[count - 1 - asked - i]
            asked += need
            if need > 0:
                top = count - asked
        else:
            keep = -(-int(new[b]) // page_size)
            give = have - keep
            if give > 0 and count + asked + give > capacity:
                flags[b] = 2
                asked += give
                continue
            for i in range(give):
                free[count + asked + i] = table[b, keep + i]
                table[b, keep + i] = -1
            asked += give
            if give > 0:
                top = count + asked
    return new.astype(np.int32), table, free, top, flags


def _rows_f64(logits):
    a = np.asarray(logits)
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return a.astype(np.float64)


def build_tree(drafter_logits, temperature, root_tokens, top_k: int, budget: int):
    """The tree sampler's candidate tree (Sec. 3.3, "Tree Sampler": the top K tokens at
    each block position, pruned to the top ``budget`` prefixes by log-probability), by
    best-first search in plain loops.

    Position d = 1 .. gamma-1 of the block draws from drafter row d; its candidates are
    the top_k tokens of log q_d = log softmax(row / T) (T = temperature[b], or 1 at
    T = 0), ranked by probability, equal ones by lower token id. Node 0 is the root (the
    free token x^{L+1} = root_tokens[b]); a node at depth d < gamma - 1 offers its next
    unused candidate of position d + 1 as a child, scored score(node) + log q_{d+1}.
    Each of ``budget`` steps takes the best offered child (equal scores: the lower
    parent index) as the next node. Since scores only fall along a path, the nodes are
    the top ``budget`` prefixes and every node's parent precedes it.

    Returns a dict: tokens, parents, depth (int32 [batch][budget+1]), mask (uint64
    [batch][budget+1]: bit i of node j set iff node i is j or an ancestor of j), score
    (fp64), margin (fp64 [batch]: the smallest gap between the taken child's score and
    the best other offer over all steps; +inf if there never was another offer), and the
    ranked candidates: cand_tokens (int32 [batch][gamma][min(top_k, vocab)], row 0 -1)
    and cand_logq (their log q, fp64).
    """
    dl = _rows_f64(drafter_logits)
    B, G, V = dl.shape
    N = budget + 1
    if N > 64:
        raise ValueError("a tree holds at most 64 nodes")
    Kc = min(top_k, V)
    out = dict(tokens=np.full((B, N), -1, np.int32), parents=np.full((B, N), -1, np.int32),
               depth=np.zeros((B, N), np.int32), mask=np.zeros((B, N), np.uint64),
               score=np.zeros((B, N), np.float64), margin=np.full(B, np.inf),
               cand_tokens=np.full((B, G, Kc), -1, np.int32),
               cand_logq=np.full((B, G, Kc), np.nan, np.float64))
    for b in range(B):
        T = float(np.float32(temperature[b]))
        T = T if T > 0 else 1.0
        logq, top = [None], [None]
        for d in range(1, G):
            z = dl[b, d] / T
            m = z.max()
            lq = z - m - np.log(np.exp(z - m).sum())
            order = sorted(range(V), key=lambda x: (-lq[x], x))[:min(top_k, V)]
            logq.append(lq)
            top.append(order)
            out["cand_tokens"][b, d] = order
            out["cand_logq"][b, d] = lq[order]
        tokens, parents, depth, score = [int(root_tokens[b])], [-1], [0], [0.0]
        nxt = [0]
        margin = np.inf
        for _ in range(budget):
            offers = []
            for u in range(len(tokens)):
                d = depth[u] + 1
                if d < G and nxt[u] < len(top[d]):
                    c = top[d][nxt[u]]
                    offers.append((score[u] + logq[d][c], u, c))
            if not offers:
                raise ValueError("the tree ran out of candidates before the budget")
            best = max(offers, key=lambda o: (o[0], -o[1]))
            others = [o[0] for o in offers if o is not best]
            if others:
                margin = min(margin, best[0] - max(others))
            sc, u, c = best
            tokens.append(c)
            parents.append(u)
            depth.append(depth[u] + 1)
            score.append(sc)
            nxt[u] += 1
            nxt.append(0)
        for j in range(N):
            bits, a = 0, j
            while a >= 0:
                bits |= 1 << a
                a = parents[a]
            out["mask"][b, j] = np.uint64(bits)
        out["tokens"][b] = tokens
        out["parents"][b] = parents
        out["depth"][b] = depth
        out["score"][b] = score
        out["margin"][b] = margin
    return out


def accept_tree_greedy(target_logits, tokens, parents):
    """Greedy (T = 0) verification of a candidate tree: from the root, move to the child
    whose token is the lowest-index argmax of the current node's target row (children
    in node order); stop when there is none, and emit that argmax as the final token.
    target row j is the verifier's distribution of the token after node j.

    Returns a dict: path (int32 [batch][N], node indices, -1 padded), num_accepted
    (path length - 1), out_tokens (int32 [batch][N+1]: the path's tokens, then the final
    token, -1 padded), num_emitted (path length + 1)."""
    tl = _rows_f64(target_logits)
    B, N, V = tl.shape
    path = np.full((B, N), -1, np.int32)
    out = np.full((B, N + 1), -1, np.int32)
    na = np.zeros(B, np.int32)
    ne = np.zeros(B, np.int32)
    for b in range(B):
        cur, walk = 0, [0]
        while True:
            a = int(np.argmax(tl[b, cur]))
            nxt = next((c for c in range(N) if parents[b, c] == cur and tokens[b, c] == a), None)
            if nxt is None:
                break
            walk.append(nxt)
            cur = nxt
        path[b, :len(walk)] = walk
        toks = [int(tokens[b, x]) for x in walk] + [int(np.argmax(tl[b, cur]))]
        out[b, :len(toks)] = toks
        na[b] = len(walk) - 1
        ne[b] = len(walk) + 1
    return dict(path=path, num_accepted=na, out_tokens=out, num_emitted=ne)


def accept_tree_sampled(target_logits, tokens, parents, temperature, uniforms):
    """Sampled (T > 0) verification of a candidate tree whose nodes are deterministic
    candidates (Sec. 4.2: candidates verified at once as a prefix tree, with the
    standard rejection correction; Sec. 3.3, "Tree Sampler"), lossless for the target.

    At the current node (the root first) with target distribution p = softmax(row / T)
    of its target row, its children are tried in node order. A child is a point-mass
    proposal (q = one-hot at its token), so the rule min(1, p'/q) accepts it with
    probability p'(token), where p' is what is left of p at this node: p with the
    tokens of the children rejected so far removed, renormalised (the residual
    Norm([p' - q]_+) of a rejected point mass). Child c is accepted iff
    uniforms[c] <= p'(tokens[c]); the walk then moves to c. If no child is accepted (or
    the node has none), the final token is the inverse-CDF draw from p' with
    uniforms[0]. A sequence with T <= 0 takes the greedy walk (accept_tree_greedy).

    target_logits [batch][N][V] (float32, or uint16 bf16 bits), tokens / parents int32
    [batch][N] (parents[0] = -1, parents[c] < c), temperature float32 [batch], uniforms
    float32 [batch][N] in (0, 1]. Returns a dict: path, num_accepted, out_tokens,
    num_emitted (as accept_tree_greedy), accept_margin float64 [batch][N] (|u - p'| of
    each test taken at node c's entry, +inf elsewhere), sample_margin float64 [batch]
    (the final draw's inverse-CDF margin over the remaining mass), status int32 [batch]
    (0; 1: a node row with NaN, or for a tempered sequence +inf or no finite logit; 2: a
    token outside [0, V) or parents that are not a tree; such a sequence gets -1
    outputs and num_emitted 0)."""
    tl = _rows_f64(target_logits)
    B, N, V = tl.shape
    tok = np.asarray(tokens, dtype=np.int64)
    par = np.asarray(parents, dtype=np.int64)
    T = np.asarray(temperature, dtype=np.float32)
    u = np.asarray(uniforms, dtype=np.float32).astype(np.float64)
    path = np.full((B, N), -1, np.int32)
    out = np.full((B, N + 1), -1, np.int32)
    na = np.full(B, -1, np.int32)
    ne = np.zeros(B, np.int32)
    am = np.full((B, N), np.inf)
    sm = np.full(B, np.inf)
    st = np.zeros(B, np.int32)
    for b in range(B):
        if (np.any(tok[b] < 0) or np.any(tok[b] >= V) or par[b, 0] != -1 or
                any(not (0 <= par[b, c] < c) for c in range(1, N))):
            st[b] = 2
            continue
        tempered = float(T[b]) > 0.0
        # every node row must be usable: no NaN; tempered rows also no +inf and a finite max
        rows_bad = np.isnan(tl[b]).any() or (tempered and (
            np.isposinf(tl[b]).any() or not np.isfinite(tl[b].max(axis=1)).all()))
        if rows_bad:
            st[b] = 1
            continue
        if not tempered:
            g = accept_tree_greedy(tl[b:b + 1], tok[b:b + 1], par[b:b + 1])
            path[b], out[b], na[b], ne[b] = g["path"][0], g["out_tokens"][0], \
                g["num_accepted"][0], g["num_emitted"][0]
            continue
        cur, walk, final = 0, [0], None
        while True:
            prob = softmax(tl[b, cur], float(T[b]))
            w = prob.copy()
            nxt = None
            for c in range(1, N):
                if par[b, c] != cur:
                    continue
                S = w.sum()
                ratio = w[tok[b, c]] / S if S > 0.0 else 1.0
                am[b, c] = abs(u[b, c] - min(1.0, ratio))
                if u[b, c] <= ratio:
                    nxt = c
                    break
                w[tok[b, c]] = 0.0  # the rejected candidate leaves the distribution
            if nxt is not None:
                walk.append(nxt)
                cur = nxt
                continue
            S = w.sum()
            if not S > 0.0:  # only through rounding: draw from p itself
                w, S = prob, prob.sum()
            final, margin = inverse_cdf(w, u[b, 0])
            sm[b] = margin / S
            break
        path[b, :len(walk)] = walk
        toks = [int(tok[b, x]) for x in walk] + [int(final)]
        out[b, :len(toks)] = toks
        na[b] = len(walk) - 1
        ne[b] = len(walk) + 1
    return dict(path=path, num_accepted=na, out_tokens=out, num_emitted=ne, accept_margin=am,
                sample_margin=sm, status=st)


def compact_tree_kv(k_cache, v_cache, page_table, kv_len, num_nodes: int, path, num_accepted):
    """Keep the accepted path of a verified tree in the paged KV cache: the block's node
    keys sit at positions ctx .. ctx + num_nodes - 1 (kv_len = ctx + num_nodes); the key
    and value of path node path[d] move to position ctx + d for d = 1 .. n - 1
    (n = num_accepted + 1; the root stays at ctx), and kv_len becomes ctx + n (ctx when
    num_accepted = -1). Returns new (k_cache, v_cache, kv_len)."""
    k = np.array(k_cache, copy=True)
    v = np.array(v_cache, copy=True)
    kl = np.array(kv_len, dtype=np.int32, copy=True)
    P = k.shape[2]
    for b in range(len(kl)):
        ctx = int(kv_len[b]) - num_nodes
        n = int(num_accepted[b]) + 1 if num_accepted[b] >= 0 else 0
        for d in range(1, n):
            src, dst = ctx + int(path[b, d]), ctx + d
            ps, pd = page_table[b, src // P], page_table[b, dst // P]
            k[pd, :, dst % P] = k[ps, :, src % P]
            v[pd, :, dst % P] = v[ps, :, src % P]
        kl[b] = ctx + n
    return k, v, kl


def lm_head_stats(hidden, weight, temperature, rows_per_seq: int, tokens=None, rows=None,
                  chunk: int = 8192):
    """The target's LM head and the acceptance's row statistics (Sec. 4.2 verifier pass;
    Appendix B.3 reads p = softmax(l / T) through its normaliser, maximum and drafted
    logits): l = hidden . weight^T in fp64 on the exactly decoded bf16 operands (a
    matmul per chunk of vocab rows), then per row r (sequence r // rows_per_seq):
    max, the lowest index of the max, sum_v exp((l_v - max) / T) (T <= 0 sums at T = 1)
    and l at tokens[r] (NaN where tokens is None or the token is outside [0, vocab)).

    hidden: uint16 bf16 bits [rows][H]; weight: uint16 [vocab][H]; rows: optional row
    indices to compute. Returns a dict: row_max, row_sum, row_argmax, token_logit (over
    the selected rows), logits (fp64 [selected rows][vocab]) and abs_bound (fp64, per
    row: max_v sum_i |h_i w_vi|, which bounds a logit's accumulation error)."""
    h = _rows_f64(hidden)
    sel = np.arange(h.shape[0]) if rows is None else np.asarray(rows, dtype=np.int64)
    hs = h[sel]
    V = weight.shape[0]
    logits = np.empty((len(sel), V), np.float64)
    bound = np.zeros(len(sel), np.float64)
    for v0 in range(0, V, chunk):
        w = _rows_f64(weight[v0:v0 + chunk])
        logits[:, v0:v0 + chunk] = hs @ w.T
        bound = np.maximum(bound, (np.abs(hs) @ np.abs(w).T).max(axis=1))
    out = dict(row_max=np.empty(len(sel)), row_sum=np.empty(len(sel)),
               row_argmax=np.empty(len(sel), np.int64), token_logit=np.full(len(sel), np.nan),
               logits=logits, abs_bound=bound)
    for i, r in enumerate(sel):
        T = float(np.float32(temperature[r // rows_per_seq]))
        T = T if T > 0 else 1.0
        l = logits[i]
        m = l.max()
        out["row_max"][i] = m
        out["row_argmax"][i] = int(np.argmax(l))
        out["row_sum"][i] = np.exp((l - m) / T).sum()
        if tokens is not None and 0 <= int(tokens[r]) < V:
            out["token_logit"][i] = l[int(tokens[r])]
    return out


def verify_attention(q, k_cache, v_cache, page_table, kv_len, gamma: int, softmax_scale=None,
                     rows=None, nthreads: int = 0, tree_mask=None):
    """fp64 block-causal paged GQA attention.

    q: uint16 bf16 bits [batch][gamma][Hq][D]; k_cache, v_cache: uint16
    [num_pages][Hkv][page_size][D]; page_table: int32 [batch][max_pages];
    kv_len: int32 [batch].  rows: optional int array [n][3] of (b, j, h) to compute.
    tree_mask: optional uint64 [batch][gamma]: block query j sees the block keys whose
    bits are set (tree attention) instead of the first j + 1.
    Returns (out fp64 [batch][gamma][Hq][D], lse fp64 [batch][gamma][Hq], status).
    Rows not listed in ``rows`` are left NaN.
    """
    lib = _load()
    qa = _c(q, np.uint16)
    ka = _c(k_cache, np.uint16)
    va = _c(v_cache, np.uint16)
    pt = _c(page_table, np.int32)
    kl = _c(kv_len, np.int32)
    batch, g, Hq, D = qa.shape
    if g != gamma:
        raise ValueError("q's second dimension must equal gamma")
    num_pages, Hkv, page_size, D2 = ka.shape
    if D2 != D or va.shape != ka.shape:
        raise ValueError("cache shapes disagree with q")
    scale = 1.0 / np.sqrt(D) if softmax_scale is None else float(softmax_scale)
    out = np.full((batch, gamma, Hq, D), np.nan, np.float64)
    lse = np.full((batch, gamma, Hq), np.nan, np.float64)
    st = np.empty(batch, np.int32)
    r = None
    nrows = 0
    if rows is not None:
        r = _c(rows, np.int32).reshape(-1, 3)
        nrows = r.shape[0]
    tm = None if tree_mask is None else _c(tree_mask, np.uint64)
    rc = lib.oracle_verify_attention_tree(batch, gamma, Hq, Hkv, D, page_size, pt.shape[1],
                                          num_pages, scale, _ptr(qa), _ptr(ka), _ptr(va),
                                          _ptr(pt), _ptr(kl), _ptr(tm), _ptr(out), _ptr(lse),
                                          _ptr(r), nrows, _ptr(st), int(nthreads))
    if rc:
        raise ValueError("invalid arguments to oracle_verify_attention")
    return out, lse, st
