"""GPU parity of the fused LM head + row statistics (spec_lm_head_stats) with the oracle.

Tolerances: the kernel accumulates in fp32 (tensor cores) and the oracle in fp64, so a
logit may differ by up to ERR = 2^-20 * sum_i |h_i w_vi| (the oracle's abs_bound). row_max
and token_logit within ERR; row_sum within 1e-4 relative plus 2 ERR / T (its
exponents shift by at most ERR / T); row_argmax exact unless the oracle's two largest
logits lie within 2 ERR; bf16 logits within one bf16 rounding of the oracle's plus ERR."""

import numpy as np
import pytest
import torch

from paper_2609_04010_gb300 import binding
from paper_2609_04010_gb300 import workloads as W

from helpers import bf16_dev, dev

pytestmark = pytest.mark.gpu


def gpu_lm(h, w, T, rps, tok=None, want_logits=False):
    r = binding.lm_head_stats(bf16_dev(h), bf16_dev(w), dev(T), rps,
                              tokens=None if tok is None else dev(tok), want_logits=want_logits)
    torch.cuda.synchronize()
    out = {}
    for k, v in r.items():
        out[k] = v.float().cpu().numpy() if k == "logits" else v.cpu().numpy()
    return out


def check(oracle_mod, h, w, T, rps, tok, rows=None):
    g = gpu_lm(h, w, T, rps, tok)
    o = oracle_mod.lm_head_stats(h, w, T, rps, tokens=tok, rows=rows)
    sel = np.arange(h.shape[0]) if rows is None else np.asarray(rows)
    err = 2.0 ** -20 * o["abs_bound"]
    Te = np.array([float(T[r // rps]) if T[r // rps] > 0 else 1.0 for r in sel])
    np.testing.assert_array_less(np.abs(g["row_max"][sel] - o["row_max"]), err + 1e-30)
    np.testing.assert_array_less(np.abs(g["row_sum"][sel] - o["row_sum"]),
                                 o["row_sum"] * (1e-4 + 2 * err / Te))
    srt = np.sort(o["logits"], axis=1)
    gap = srt[:, -1] - srt[:, -2] if o["logits"].shape[1] > 1 else np.full(len(sel), np.inf)
    clear = gap > 2 * err
    np.testing.assert_array_equal(g["row_argmax"][sel][clear], o["row_argmax"][clear])
    if tok is not None:
        ok = ~np.isnan(o["token_logit"])
        np.testing.assert_array_equal(np.isnan(g["token_logit"][sel]), ~ok)
        np.testing.assert_array_less(np.abs(g["token_logit"][sel][ok] - o["token_logit"][ok]), err[ok] + 1e-30)
    return g, o


@pytest.mark.parametrize("R,H,V,rps", [(7, 64, 300, 7), (200, 512, 5000, 16), (130, 1000, 777, 13),
                                       (64, 2048, 32000, 8), (1, 8, 1, 1)])
def test_lm_head_shapes(oracle_mod, R, H, V, rps):
    h, w, T, tok = W.make_lm_inputs(R, H, V, rps, temperature=[1.0, 0.0, 0.7], seed=R + V)
    check(oracle_mod, h, w, T, rps, tok)


def test_lm_head_llama8b_shape_all_rows(oracle_mod):
    # the verify step's rows at the Llama-3-8B head: 8 sequences x 8 positions, 4096 -> 128,256
    h, w, T, tok = W.make_lm_inputs(64, 4096, 128256, 8, seed=5)
    check(oracle_mod, h, w, T, 8, tok)


def test_lm_head_logits_output(oracle_mod):
    h, w, T, tok = W.make_lm_inputs(40, 256, 3000, 8, seed=6)
    g = gpu_lm(h, w, T, 8, tok, want_logits=True)
    o = oracle_mod.lm_head_stats(h, w, T, 8, tokens=tok)
    ref = o["logits"]
    err = 2.0 ** -20 * o["abs_bound"][:, None]
    # within one bf16 rounding (relative 2^-8) of the oracle's logit, plus ERR
    assert np.all(np.abs(g["logits"] - ref) <= np.abs(ref) * 2.0 ** -8 + err + 1e-30)
    srt = np.sort(ref, axis=1)
    clear = srt[:, -1] - srt[:, -2] > 2 * err[:, 0]
    np.testing.assert_array_equal(g["row_argmax"][clear], np.argmax(ref, axis=1)[clear])


def test_lm_head_token_edges_and_bad_rows(oracle_mod):
    h, w, T, tok = W.make_lm_inputs(12, 128, 1000, 4, seed=7)
    tok = tok.copy()
    tok[1] = -1
    tok[2] = 1000
    tok[3] = 999
    h = h.copy()
    h[5, 17] = np.uint16(0x7FC0)  # NaN
    ws = binding.new_workspace(1 << 20)
    r = binding.lm_head_stats(bf16_dev(h), bf16_dev(w), dev(T), 4, tokens=dev(tok), ws=ws)
    torch.cuda.synchronize()
    assert binding.read_device_status(ws)[1] == binding.FLAG_BAD_LOGITS
    g = {k: v.cpu().numpy() for k, v in r.items()}
    assert g["row_argmax"][5] == -1
    assert np.isnan(g["token_logit"][1]) and np.isnan(g["token_logit"][2])
    good = [i for i in range(12) if i != 5]
    o = oracle_mod.lm_head_stats(h, w, T, 4, tokens=tok, rows=good)
    np.testing.assert_array_equal(g["row_argmax"][good], o["row_argmax"])
    assert abs(g["token_logit"][3] - o["token_logit"][good.index(3)]) < 1e-3
