"""Shared test utilities: moving generator outputs to the device, running the CUDA path
through the C ABI, and comparing it with the oracle under the documented tolerances.

Tolerances (the arithmetic behind them is derived in the design notes):
  * accepted lengths and emitted tokens: bit-exact, except a decision or a draw whose
    uniform lies within TIE_MARGIN = 1e-6 (in probability units) of its threshold in
    the oracle; such ties are counted, and the rest of that sequence is not compared;
  * p_i(t_i), q_i(t_i): within 1e-5 relative;
  * attention outputs: within 1e-2 max-abs, and within 1e-2 of the largest output
    magnitude (|O| is ~1/sqrt(context) for random keys, so the absolute bound alone
    would accept an all-zero answer); log-sum-exp within 1e-3.
"""

from __future__ import annotations

import numpy as np
import torch

TIE_MARGIN = 1e-6
DIAG_RTOL = 1e-5
ATTN_ATOL = 1e-2
ATTN_RTOL_OF_MAX = 1e-2
LSE_ATOL = 1e-3


def bf16_dev(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).cuda()


def dev(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def logits_dev(a: np.ndarray) -> torch.Tensor:
    return bf16_dev(a) if a.dtype == np.uint16 else dev(a.astype(np.float32))


def accept_tensors(inp):
    return (logits_dev(inp.target_logits), logits_dev(inp.drafter_logits), dev(inp.block_tokens),
            dev(inp.temperature), dev(inp.uniforms))


def attn_tensors(inp):
    return (bf16_dev(inp.q), bf16_dev(inp.k_cache), bf16_dev(inp.v_cache), dev(inp.page_table),
            dev(inp.kv_len))


def gpu_accept(inp, ws=None):
    from paper_2609_04010_gb300 import binding
    r = binding.accept_block(*accept_tensors(inp), ws=ws)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in r.items() if v is not None}


def gpu_attention(inp, path=0, ws=None):
    from paper_2609_04010_gb300 import binding
    out, lse = binding.verify_attention(*attn_tensors(inp), path=path, ws=ws)
    torch.cuda.synchronize()
    return out.float().cpu().numpy(), lse.cpu().numpy()


def compare_accept(g, o, gamma, skip=()):
    """Compares GPU and oracle acceptance outputs; returns the list of ties.

    Sequences in ``skip`` are not compared. Raises AssertionError on any mismatch that
    is not a tie."""
    B = len(o["num_accepted"])
    ties = []
    for b in range(B):
        if b in skip:
            continue
        if o["status"][b] != 0:
            assert g["num_accepted"][b] == -1 and g["num_emitted"][b] == 0, b
            assert np.all(g["out_tokens"][b] == -1), b
            continue
        gn, on = int(g["num_accepted"][b]) + 1, int(o["num_accepted"][b]) + 1
        same = gn == on and np.array_equal(g["out_tokens"][b], o["out_tokens"][b]) and \
            g["num_emitted"][b] == o["num_emitted"][b]
        # the decisions both sides took agree in value
        for i in range(1, min(gn, on) + 1):
            if i >= gamma:
                break
            np.testing.assert_allclose(g["diag"][b, i], o["diag"][b, i], rtol=DIAG_RTOL, atol=0,
                                       err_msg=f"diag b={b} i={i}")
        if same:
            continue
        if gn != on:
            i = min(gn, on)
            m = o["accept_margin"][b, i]
            assert m < TIE_MARGIN, (
                f"seq {b}: GPU n={gn}, oracle n={on}, decision {i} margin {m:.3g}")
            ties.append((b, "decision", i, float(m)))
        else:
            np.testing.assert_array_equal(g["out_tokens"][b, :gn], o["out_tokens"][b, :on],
                                          err_msg=f"seq {b} accepted prefix")
            m = o["sample_margin"][b]
            assert m < TIE_MARGIN, (
                f"seq {b}: final token GPU {g['out_tokens'][b, gn]} oracle "
                f"{o['out_tokens'][b, on]}, margin {m:.3g}")
            ties.append((b, "draw", gn, float(m)))
    return ties


def sample_rows(inp, n, seed=0):
    rng = np.random.default_rng(seed)
    B, G, Hq = inp.q.shape[:3]
    rows = np.stack([rng.integers(0, B, n), rng.integers(0, G, n), rng.integers(0, Hq, n)], 1)
    # always include the first and last block positions of the first sequence
    extra = np.array([[0, 0, 0], [0, G - 1, Hq - 1], [B - 1, G - 1, 0]])
    return np.unique(np.concatenate([rows, extra]), axis=0).astype(np.int32)


def compare_attention(g_out, g_lse, o_out, o_lse, rows=None):
    if rows is not None:
        b, j, h = rows[:, 0], rows[:, 1], rows[:, 2]
        g_out, o_out, g_lse, o_lse = g_out[b, j, h], o_out[b, j, h], g_lse[b, j, h], o_lse[b, j, h]
    err = np.abs(g_out - o_out).max()
    scale = np.abs(o_out).max()
    fin = np.isfinite(o_lse)
    assert np.array_equal(fin, np.isfinite(g_lse)), "lse finiteness differs"
    lerr = np.abs(g_lse[fin] - o_lse[fin]).max() if fin.any() else 0.0
    assert err < ATTN_ATOL, f"attention max abs error {err}"
    assert err <= ATTN_RTOL_OF_MAX * scale, f"attention error {err} vs max |O| {scale}"
    assert lerr < LSE_ATOL, f"lse max abs error {lerr}"
    return float(err), float(lerr)
