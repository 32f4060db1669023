"""GPU parity on the sweep workload, all of it: gamma in {1, 2, 4, 8, 16, 32} x batch in
{1, 8, 32, 128}, 32 query / 8 KV heads, head_dim 128, ragged contexts uniform in
[256, 16,384] in 16-token pages, vocabulary 151,936 bf16 logits, drafter noise
sigma in {0.1, 1, 3}, temperatures {0, 1}: the 24 attention shapes and the 144
acceptance points.

Inputs are drawn on the device (workloads.make_*_inputs_device; the host generator
cannot fill billions of values in test time). The kernels always run on the full batch
in the launch configuration the benchmark uses (automatic kernel choice), so the full
size paths (stream-K splits and merges, ragged last tiles, the widest grids) run; the
oracle checks what it can compute in seconds:
  * attention: one row of every (sequence, KV head) unit, and every sequence's last
    block position, within 1e-2 max-abs (and of max |O|) and lse within 1e-3;
  * acceptance: the first min(batch, 8) sequences of each point bit-exact but for
    counted ties (a uniform within 1e-6 of its threshold in the oracle); every sequence
    of every point structurally (the accepted prefix is the block's, the count and
    padding agree); and at T = 0 every sequence against the greedy chain computed with
    torch's argmax (lowest index on ties, the rule's reading)."""

import numpy as np
import pytest
import torch

from paper_2609_04010_gb300 import binding
from paper_2609_04010_gb300 import workloads as W

from helpers import TIE_MARGIN, compare_accept, compare_attention

pytestmark = pytest.mark.gpu

VOCAB = 151936
ORACLE_SEQS = 8


def unit_rows(batch, gamma, hq, hkv, seed):
    """(b, j, h) rows: one random row of every (sequence, KV head) unit, and the last
    block position of every sequence (random head)."""
    rng = np.random.default_rng(seed)
    group = hq // hkv
    rows = []
    for b in range(batch):
        for g in range(hkv):
            rows.append((b, int(rng.integers(gamma)), g * group + int(rng.integers(group))))
        rows.append((b, gamma - 1, int(rng.integers(hq))))
    return np.unique(np.array(rows, np.int32), axis=0)


@pytest.mark.parametrize("batch", W.SWEEP_BATCHES)
@pytest.mark.parametrize("gamma", W.SWEEP_GAMMAS)
def test_sweep_attention(oracle_mod, gamma, batch):
    wl = W.sweep_workload(gamma, batch)
    seed = 7000 + gamma * 1000 + batch
    di = W.make_attn_inputs_device(batch, gamma, wl.num_q_heads, wl.num_kv_heads, wl.head_dim,
                                   wl.page_size, wl.ctx, seed=seed)
    out, lse = binding.verify_attention(di.q, di.k_cache, di.v_cache, di.page_table, di.kv_len,
                                        path=binding.ATTN_AUTO)
    torch.cuda.synchronize()
    rows = unit_rows(batch, gamma, wl.num_q_heads, wl.num_kv_heads, seed)
    h = di.host()
    del di
    o_out, o_lse, st = oracle_mod.verify_attention(h.q, h.k_cache, h.v_cache, h.page_table,
                                                   h.kv_len, gamma, rows=rows)
    assert np.all(st == 0)
    err, lerr = compare_attention(out.float().cpu().numpy(), lse.cpu().numpy(), o_out, o_lse,
                                  rows)
    print(f"sweep attention g{gamma} b{batch}: {len(rows)} rows, max ctx "
          f"{int(h.kv_len.max()) - gamma}, err {err:.2e}, lse err {lerr:.2e}")


def check_structure(g, inp_tokens, gamma):
    """Every sequence: emitted = accepted + 2 in [2, gamma + 1], the emitted prefix is the
    block's first token and its accepted drafts, the final token a vocabulary id, the
    rest -1 padding."""
    na, ot, ne = g["num_accepted"], g["out_tokens"], g["num_emitted"]
    assert np.all((na >= 0) & (na <= gamma - 1))
    assert np.all(ne == na + 2)
    for b in range(len(na)):
        n = int(na[b]) + 1
        assert np.array_equal(ot[b, :n], inp_tokens[b, :n]), b
        assert 0 <= ot[b, n] < VOCAB, b
        assert np.all(ot[b, n + 1:] == -1), b


def greedy_chain(di, gamma):
    """(num_accepted, final token) of every sequence under the T = 0 rule, from torch's
    argmax of the target rows (lowest index among equal maxima)."""
    am = torch.argmax(di.target_logits, dim=-1).to(torch.int32)  # [batch][gamma]
    tok = di.block_tokens
    if gamma > 1:
        match = (tok[:, 1:] == am[:, :-1]).to(torch.int32)  # draft i vs target row i-1
        acc = torch.cumprod(match, dim=1).sum(dim=1)
    else:
        acc = torch.zeros(tok.shape[0], dtype=torch.int64, device=tok.device)
    final = am.gather(1, acc.view(-1, 1).long()).view(-1)
    return acc.cpu().numpy(), final.cpu().numpy()


@pytest.mark.parametrize("batch", W.SWEEP_BATCHES)
@pytest.mark.parametrize("gamma", W.SWEEP_GAMMAS)
def test_sweep_accept(oracle_mod, gamma, batch):
    total_ties, checked = 0, 0
    for sigma in W.SWEEP_SIGMAS:
        for T in W.SWEEP_TEMPS:
            seed = int(gamma * 100000 + batch * 100 + sigma * 10 + T)
            di = W.make_accept_inputs_device(batch, gamma, VOCAB, 3.0, sigma, T, seed=seed)
            r = binding.accept_block(di.target_logits, di.drafter_logits, di.block_tokens,
                                     di.temperature, di.uniforms)
            torch.cuda.synchronize()
            g = {k: v.cpu().numpy() for k, v in r.items()}
            tokens = di.block_tokens.cpu().numpy()
            check_structure(g, tokens, gamma)
            if T == 0.0:
                acc, final = greedy_chain(di, gamma)
                np.testing.assert_array_equal(g["num_accepted"], acc)
                np.testing.assert_array_equal(g["out_tokens"][np.arange(batch), acc + 1], final)
            n = min(batch, ORACLE_SEQS)
            h = di.host(n)
            del di
            o = oracle_mod.accept_block(h.target_logits, h.drafter_logits, h.block_tokens,
                                        h.temperature, h.uniforms)
            assert np.all(o["status"] == 0)
            ties = compare_accept({k: v[:n] for k, v in g.items()}, o, gamma)
            assert len(ties) <= max(1, int(0.02 * n)), (sigma, T, ties)
            assert all(t[3] < TIE_MARGIN for t in ties)
            total_ties += len(ties)
            checked += n
    print(f"sweep accept g{gamma} b{batch}: {checked} sequences vs the oracle "
          f"(6 points), ties {total_ties}")
