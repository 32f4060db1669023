"""GPU parity of the acceptance half of the verify step (spec_accept_block) with the
oracle, through the C ABI, on the same seeded inputs.

Accepted lengths and emitted tokens must match bit for bit except ties (a uniform
within 1e-6 of its threshold in the oracle), which are counted; p_i(t_i) and
q_i(t_i) must agree within 1e-5 relative."""

import numpy as np
import pytest
import torch
from scipy import stats

from paper_2609_04010_gb300 import binding
from paper_2609_04010_gb300 import workloads as W

from helpers import accept_tensors, compare_accept, gpu_accept

pytestmark = pytest.mark.gpu


def oracle_accept(oracle_mod, inp):
    return oracle_mod.accept_block(inp.target_logits, inp.drafter_logits, inp.block_tokens,
                                   inp.temperature, inp.uniforms)


def check(oracle_mod, inp, max_tie_frac=0.02):
    g = gpu_accept(inp)
    o = oracle_accept(oracle_mod, inp)
    ties = compare_accept(g, o, inp.gamma)
    assert len(ties) <= max(1, int(max_tie_frac * inp.batch)), ties
    ok = o["status"] == 0
    assert np.all(g["num_emitted"][ok] == g["num_accepted"][ok] + 2)
    assert np.all((g["num_emitted"][ok] >= 2) & (g["num_emitted"][ok] <= inp.gamma + 1))
    return g, o, ties


@pytest.mark.parametrize("name", ["tiny", "llama8b", "serve64", "long70b"])
def test_named_workloads(oracle_mod, name):
    inp = W.workload(name).accept_inputs(seed=0)
    g, o, ties = check(oracle_mod, inp)
    print(f"{name}: mean accepted {g['num_accepted'].mean():.3f}, ties {len(ties)}")


SWEEP_POINTS = [(1, 1, 1.0, 1.0), (2, 8, 0.1, 1.0), (4, 32, 3.0, 0.0), (8, 8, 1.0, 1.0),
                (16, 8, 0.1, 1.0), (32, 8, 3.0, 1.0), (32, 1, 0.1, 0.0), (16, 32, 1.0, 0.0),
                (4, 128, 0.1, 1.0)]


@pytest.mark.parametrize("gamma,batch,sigma,T", SWEEP_POINTS)
def test_sweep_points(oracle_mod, gamma, batch, sigma, T):
    inp = W.sweep_workload(gamma, batch, sigma, T).accept_inputs(seed=gamma * 1000 + batch)
    check(oracle_mod, inp)


@pytest.mark.parametrize("vocab,dtype", [(1, "f32"), (7, "f32"), (8, "bf16"), (8191, "bf16"),
                                         (8193, "bf16"), (16392, "bf16"), (40000, "f32"),
                                         (24577, "f32")])
def test_vocab_edges(oracle_mod, vocab, dtype):
    inp = W.make_accept_inputs(12, 5, vocab, dtype, 3.0, 1.0, [1.0, 0.0, 0.5], seed=vocab)
    check(oracle_mod, inp, max_tie_frac=0.1)


def test_gamma_one_is_a_plain_decode_step(oracle_mod):
    inp = W.make_accept_inputs(40, 1, 5000, "bf16", 3.0, 1.0, [1.0, 0.0], seed=3)
    g, o, _ = check(oracle_mod, inp)
    assert np.all(g["num_accepted"] == 0) and np.all(g["num_emitted"] == 2)


def test_identical_drafter_accepts_every_draft(oracle_mod):
    inp = W.make_accept_inputs(16, 8, 30000, "bf16", 3.0, 0.0, 1.0, seed=4)
    g, o, _ = check(oracle_mod, inp)
    assert np.all(g["num_accepted"] == 7)


def test_masked_vocabulary_entries(oracle_mod):
    inp = W.make_accept_inputs(8, 6, 40000, "bf16", 3.0, 1.0, [1.0, 0.0], seed=5)
    ninf = np.uint16(0xFF80)
    inp.target_logits[:, :, 8192:16384] = ninf   # a whole chunk masked
    inp.drafter_logits[:, 2:, 100:900] = ninf    # a partial range masked
    inp.target_logits[3, 1, 30000:] = ninf
    check(oracle_mod, inp)


def test_greedy_ties_pick_lowest_index(oracle_mod):
    inp = W.make_accept_inputs(8, 4, 20000, "bf16", 1.0, 1.0, 0.0, seed=6)
    big = W.f32_to_bf16_bits(np.array([50.0], np.float32))[0]
    for b in range(8):
        for j in range(4):
            inp.target_logits[b, j, [777 + b, 15000 + j, 19999]] = big  # exact ties
    inp.block_tokens[:4, 1] = np.arange(4) + 777  # drafts equal to the lowest tied index
    g, o, _ = check(oracle_mod, inp)
    for b in range(8):
        n = g["num_accepted"][b] + 1
        assert g["out_tokens"][b, n] == 777 + b


def test_bad_inputs_flagged_without_disturbing_others(oracle_mod):
    inp = W.make_accept_inputs(6, 4, 10000, "f32", 3.0, 1.0, [1.0, 0.0, 1.0, 1.0, 0.0, 1.0],
                               seed=7)
    inp.block_tokens[1, 2] = 10000
    inp.target_logits[2, 3, 17] = np.nan
    inp.drafter_logits[3, 1, 5] = np.inf
    inp.target_logits[4, 0, 9] = np.nan  # greedy row
    ws_args = accept_tensors(inp)
    a0 = binding.accept_block(*ws_args)  # warm up a workspace-free call
    res = {k: torch.empty_like(v) if v is not None else None for k, v in a0.items()}
    args = binding.accept_args(*ws_args, res["num_accepted"], res["out_tokens"],
                               res["num_emitted"], res["diag"])
    ws = binding.new_workspace(binding.workspace_size(accept=args))
    binding.accept_block_args(args, ws)
    code, flags = binding.read_device_status(ws)
    assert code == 5 and flags == (binding.FLAG_BAD_TOKEN | binding.FLAG_BAD_LOGITS)
    assert binding.read_device_status(ws) == (0, 0)  # reading cleared it
    g = {k: v.cpu().numpy() for k, v in res.items()}
    o = oracle_accept(oracle_mod, inp)
    assert list(o["status"]) == [0, 2, 1, 1, 1, 0]
    compare_accept(g, o, inp.gamma)


def test_deterministic_and_workspace_reusable(oracle_mod):
    inp = W.make_accept_inputs(32, 8, 50000, "bf16", 3.0, 1.0, [1.0, 0.0, 0.7], seed=8)
    t = accept_tensors(inp)
    first = binding.accept_block(*t)
    args0 = binding.accept_args(*t, first["num_accepted"], first["out_tokens"],
                                first["num_emitted"], first["diag"])
    ws = binding.new_workspace(binding.workspace_size(accept=args0))
    outs = []
    for _ in range(3):
        r = binding.accept_block(*t, ws=ws)
        outs.append({k: v.cpu().numpy() for k, v in r.items()})
    for r in outs[1:]:
        for k in r:
            np.testing.assert_array_equal(r[k], outs[0][k])
    # the counters returned to zero: the whole workspace past the partials is reusable,
    # and a fresh workspace gives the same answer
    fresh = binding.accept_block(*t)
    np.testing.assert_array_equal(fresh["out_tokens"].cpu().numpy(), outs[0]["out_tokens"])


def _complete(rng, out, ne, p):
    gamma, V = p.shape
    x = np.empty((out.shape[0], gamma), np.int64)
    n = ne - 1
    for k in range(1, gamma + 1):
        fresh = rng.choice(V, size=out.shape[0], p=p[k - 1])
        x[:, k - 1] = np.where(k <= n, out[:, k], fresh)
    return x


def test_gpu_output_distribution_chi_square():
    """10^6 GPU verify steps at vocab 8, gamma 3 against the target product distribution."""
    from scipy import special
    rng = np.random.default_rng(21)
    gamma, V, T = 3, 8, 1.0
    target = (rng.standard_normal((gamma, V)) * 1.5).astype(np.float32)
    drafter = np.empty_like(target)
    drafter[0] = rng.standard_normal(V).astype(np.float32)
    drafter[1:] = target[:-1] + rng.standard_normal((gamma - 1, V)).astype(np.float32)
    p = special.softmax(target.astype(np.float64), axis=-1)
    q = special.softmax(drafter.astype(np.float64), axis=-1)
    N, chunk = 1_000_000, 62_500
    xs = []
    tl = torch.from_numpy(np.broadcast_to(target, (chunk, gamma, V)).copy()).cuda()
    dl = torch.from_numpy(np.broadcast_to(drafter, (chunk, gamma, V)).copy()).cuda()
    temp = torch.full((chunk,), T, dtype=torch.float32, device="cuda")
    for c in range(N // chunk):
        tok = np.zeros((chunk, gamma), np.int32)
        for i in range(gamma):
            tok[:, i] = rng.choice(V, size=chunk, p=q[i])
        u = binding.philox_uniforms(W.uniform_seed(1000 + c), chunk * gamma).view(chunk, gamma)
        r = binding.accept_block(tl, dl, torch.from_numpy(tok).cuda(), temp, u, want_diag=False)
        xs.append(_complete(rng, r["out_tokens"].cpu().numpy(), r["num_emitted"].cpu().numpy(), p))
    x = np.concatenate(xs)
    flat = np.ravel_multi_index(tuple(x[:, k] for k in range(gamma)), (V,) * gamma)
    obs = np.bincount(flat, minlength=V ** gamma).astype(np.float64)
    P = p[0]
    for r_ in p[1:]:
        P = np.multiply.outer(P, r_)
    exp = P.ravel() * N
    small = exp < 5
    o = np.append(obs[~small], obs[small].sum())
    e = np.append(exp[~small], exp[small].sum())
    assert stats.chisquare(o, e).pvalue > 1e-3


def test_unused_drafter_row_is_never_read():
    # the classic convention's spare leading drafter row may hold anything, even NaN:
    # the unfiltered and the filtered acceptance give the same outputs and raise no flag
    from helpers import dev, logits_dev
    inp = W.workload("llama8b").accept_inputs(seed=3)
    dl = inp.drafter_logits.copy()
    dl[:, 0, :] = np.uint16(0x7FC0) if dl.dtype == np.uint16 else np.nan
    B = inp.batch
    tl, tok, T, u = (logits_dev(inp.target_logits), dev(inp.block_tokens), dev(inp.temperature),
                     dev(inp.uniforms))
    top_k, top_p = dev(np.full(B, 50, np.int32)), dev(np.full(B, 0.95, np.float32))
    for filtered in (False, True):
        outs = []
        for d in (inp.drafter_logits, dl):
            ws = binding.new_workspace(1 << 28)
            if filtered:
                r = binding.accept_block_filtered(tl, logits_dev(d), tok, T, top_k, top_p, u,
                                                  max_top_k=50, ws=ws)
            else:
                r = binding.accept_block(tl, logits_dev(d), tok, T, u, ws=ws)
            torch.cuda.synchronize()
            assert binding.read_device_status(ws) == (0, 0)
            outs.append({k: v.cpu().numpy() for k, v in r.items() if v is not None})
        for k in ("num_accepted", "out_tokens", "num_emitted"):
            np.testing.assert_array_equal(outs[0][k], outs[1][k])
        assert np.all(outs[1]["out_tokens"][:, 0] == inp.block_tokens[:, 0])


def test_gpu_mean_accepted_matches_closed_form():
    """The GPU's accepted-draft counts over 200,000 seeded steps against the closed form
    (Leviathan et al.'s acceptance rate, the TV link of Sec. 3.2): with fixed rows,
    P(a >= k) = prod_{i <= k} alpha_i, alpha_i = sum_x min(p_{i-1}(x), q_i(x)), and
    E[a] = sum_k P(a >= k). The mean and every tail probability must lie within 5
    standard errors."""
    from scipy import special
    rng = np.random.default_rng(33)
    gamma, V, T = 6, 64, 1.0
    target = (rng.standard_normal((gamma, V)) * 2.0).astype(np.float32)
    drafter = np.empty_like(target)
    drafter[0] = rng.standard_normal(V).astype(np.float32)
    drafter[1:] = target[:-1] + rng.standard_normal((gamma - 1, V)).astype(np.float32) * 0.7
    p = special.softmax(target.astype(np.float64) / T, axis=-1)
    q = special.softmax(drafter.astype(np.float64) / T, axis=-1)
    alpha = np.array([np.minimum(p[i - 1], q[i]).sum() for i in range(1, gamma)])
    tail = np.cumprod(alpha)                 # P(a >= k), k = 1 .. gamma-1
    expect = tail.sum()
    N, chunk = 200_000, 50_000
    tl = torch.from_numpy(np.broadcast_to(target, (chunk, gamma, V)).copy()).cuda()
    dl = torch.from_numpy(np.broadcast_to(drafter, (chunk, gamma, V)).copy()).cuda()
    temp = torch.full((chunk,), T, dtype=torch.float32, device="cuda")
    counts = []
    for c in range(N // chunk):
        tok = np.zeros((chunk, gamma), np.int32)
        for i in range(gamma):
            tok[:, i] = rng.choice(V, size=chunk, p=q[i])
        u = binding.philox_uniforms(W.uniform_seed(5000 + c), chunk * gamma).view(chunk, gamma)
        r = binding.accept_block(tl, dl, torch.from_numpy(tok).cuda(), temp, u, want_diag=False)
        counts.append(r["num_accepted"].cpu().numpy())
    a = np.concatenate(counts).astype(np.float64)
    se = a.std() / np.sqrt(N)
    assert abs(a.mean() - expect) < 5 * se, (a.mean(), expect, se)
    for k in range(1, gamma):
        f = (a >= k).mean()
        se_k = np.sqrt(tail[k - 1] * (1 - tail[k - 1]) / N)
        assert abs(f - tail[k - 1]) < 5 * se_k + 1e-12, (k, f, tail[k - 1])
    print(f"mean accepted {a.mean():.4f} vs closed form {expect:.4f} (se {se:.4f})")
