"""The ReMDM remasking sampler (NEXT row) on the GPU, through the C ABI,
against the oracle and the shared Philox generator."""
import numpy as np
import pytest

import workloads as wl
from oracle import tadm_oracle as O

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def T():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()
    from paper_2609_37924_gb300 import tadm
    return tadm


def nucleus_valid(logits, mask_id, top_p, u, tok, tol=1e-5):
    """A draw that differs from the oracle's is valid when it lies in the
    fp64 nucleus (or ties its threshold within tol) and u * mass sits within
    tol of one of its CDF edges: fp32 vs fp64 sums moved a boundary."""
    l = logits.astype(np.float64).copy()
    l[mask_id] = -np.inf
    q = np.exp(l - l.max())
    desc = np.sort(q)[::-1]
    k = int(np.searchsorted(np.cumsum(desc), top_p * q.sum(), side="left"))
    tau = desc[min(k, desc.size - 1)]
    if tok == mask_id or q[tok] < tau * (1.0 - tol):
        return False
    qn = np.where(q >= tau * (1.0 - tol), q, 0.0)
    c = np.cumsum(qn)
    goal = u * c[-1]
    return min(abs(c[tok] - goal), abs(c[tok] - qn[tok] - goal)) <= tol * c[-1] or c[tok] - qn[tok] <= goal < c[tok]


def test_remdm_draws_are_the_shared_philox_bit_exactly(T):
    """The kernel's Philox4x32-10 draws equal the generator module's, also
    for block indices above 2^32."""
    for seed, step, B, R in ((3, 0, 2, 37), (0xDEADBEEF12345, 1_000_000, 4, 1100)):
        out = torch.empty((B, R, 3), dtype=torch.float32, device="cuda")
        T.tadm_remdm_uniforms(seed, step, B, R, out)
        torch.cuda.synchronize()
        assert np.array_equal(out.cpu().numpy().astype(np.float64), wl.remdm_uniforms(seed, step, B, R))


@pytest.mark.parametrize("V,top_p,sigma,p_un", [(1000, 0.9, 0.2, 0.4), (32768, 0.9, 0.05, 0.7), (257, 1.0, 0.5, 1.0),
                                            (60000, 0.9, 0.1, 0.3)])   # 60000: rows too long for shared memory
def test_remdm_update_matches_the_oracle(T, V, top_p, sigma, p_un):
    """One reverse step from the same logits: actions (keep / remask /
    unmask) bit-exact, tokens equal to the oracle's or valid at a CDF edge."""
    B, R, first, mask, seed, step = 3, 300, 40, V - 1, 1234, 7
    rng = np.random.default_rng(V)
    z = np.where(rng.random((B, R)) < 0.5, mask, rng.integers(0, V - 1, (B, R))).astype(np.int32)
    z[:, :first] = rng.integers(0, V - 1, (B, first))
    scale = np.where(rng.random((B * R, 1)) < 0.5, 0.3, 3.0)     # flat and peaked rows
    logits = (rng.standard_normal((B * R, V)) * scale).astype(np.float32)
    zt = torch.from_numpy(z).cuda()
    act = torch.empty(B * R, dtype=torch.int32, device="cuda")
    T.tadm_remdm_update(zt, torch.from_numpy(logits).cuda(), first, mask, sigma, p_un, top_p, seed, step, act)
    torch.cuda.synchronize()
    zg, ag = zt.cpu().numpy(), act.cpu().numpy().reshape(B, R)
    u = wl.remdm_uniforms(seed, step, B, R)
    exact = total = 0
    for b in range(B):
        zo, ao = O.remdm_step(z[b], logits[b * R:(b + 1) * R], first, sigma, p_un, top_p, u[b], mask)
        assert np.array_equal(ag[b], ao)
        assert np.array_equal(zg[b][ao != 2], zo[ao != 2])
        for r in np.nonzero(ao == 2)[0]:
            total += 1
            if zg[b, r] == zo[r]:
                exact += 1
            else:
                assert nucleus_valid(logits[b * R + r], mask, top_p, u[b, r, 2], zg[b, r]), (b, r, zg[b, r], zo[r])
    assert total > 50 and exact >= 0.99 * total, (exact, total)


def test_remdm_token_frequencies_follow_the_nucleus(T):
    """4096 independent draws from one distribution: the empirical
    frequencies match the renormalised nucleus probabilities."""
    V, R, mask, top_p = 24, 4096, 23, 0.8
    row = np.linspace(-2.0, 2.0, V).astype(np.float32)[::-1].copy()
    logits = np.tile(row, (R, 1))
    z = np.full((1, R), mask, np.int32)
    zt = torch.from_numpy(z).cuda()
    act = torch.empty(R, dtype=torch.int32, device="cuda")
    T.tadm_remdm_update(zt, torch.from_numpy(logits).cuda(), 0, mask, 0.0, 1.0, top_p, 99, 0, act)
    torch.cuda.synchronize()
    got = np.bincount(zt.cpu().numpy().ravel(), minlength=V) / R
    q = np.exp(row.astype(np.float64) - row[:mask].max())
    q[mask] = 0.0
    desc = np.sort(q)[::-1]
    tau = desc[np.searchsorted(np.cumsum(desc), top_p * q.sum())]
    want = np.where(q >= tau, q, 0.0)
    want /= want.sum()
    assert got[mask] == 0.0 and np.all(got[want == 0.0] == 0.0)
    assert 0.5 * np.abs(got - want).sum() < 0.03


def test_generate_remdm_matches_the_oracle_fp32(T):
    """Whole ReMDM-Cap generations of the fp32 tiny workload (K = 4): the
    GPU follows the oracle's trajectory (same draws, fp32 vs fp64 logits)."""
    w = wl.WORKLOADS["tiny"]
    m = w.model
    host = wl.make_weights(m, seed=0)
    tm = T.TadmModel(m, T.upload_weights(m, host), max_batch=1, max_rows=w.total_len)
    o = O.Oracle(m, host)
    prompts = wl.make_prompts(w)
    for kind, eta, seed in (("cap", 0.04, 5), ("loop", 0.02, 6)):
        out = torch.empty((1, w.total_len), dtype=torch.int32, device="cuda")
        scratch = torch.empty((w.gen_len, m.vocab), dtype=torch.float32, device="cuda")
        tm.tadm_generate_remdm(torch.from_numpy(prompts).cuda(), out, w.gen_len, w.steps_per_block, 4, kind, eta,
                               0.9, seed, scratch)
        tm.tadm_sync_status()
        got = out.cpu().numpy()
        ref = o.generate_remdm(prompts, w.gen_len, w.steps_per_block, 4, kind, eta, 0.9,
                               lambda n, s=seed: wl.remdm_uniforms(s, n, 1, w.total_len))
        assert np.all(got != m.mask_id) and np.array_equal(got[:, :w.prompt_len], prompts)
        assert float(np.mean(got == ref)) >= 0.98, (kind, float(np.mean(got == ref)))
        c = tm.tadm_get_counters()
        assert c["denoise_steps"] == w.steps_per_block and c["anchor_calls"] == (w.steps_per_block + 3) // 4
    tm.close()


def test_generate_remdm_bf16_completes(T):
    """bf16 test model, batch 4: every generated position ends unmasked, the
    prompt is untouched, and the same seed reproduces the same tokens."""
    m = wl.ModelConfig(vocab=4096, d_model=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=768, n_anchor=3,
                       n_denoise=2, dtype="bf16")
    B, P, G, steps = 4, 32, 160, 24
    w = wl.Workload("t", m, batch=B, prompt_len=P, gen_len=G, steps_per_block=steps, K=4)
    tm = T.TadmModel(m, T.upload_weights(m, wl.make_weights(m, seed=2)), max_batch=B, max_rows=P + G)
    p = torch.from_numpy(wl.make_prompts(w, batch=B, seed=3)).cuda()
    scratch = torch.empty((B * G, m.vocab), dtype=torch.float32, device="cuda")
    outs = []
    for _ in range(2):
        out = torch.empty((B, P + G), dtype=torch.int32, device="cuda")
        tm.tadm_generate_remdm(p, out, G, steps, 4, "cap", 0.04, 0.9, 17, scratch)
        tm.tadm_sync_status()
        outs.append(out.cpu().numpy())
    assert np.array_equal(outs[0], outs[1])
    assert np.all(outs[0] != m.mask_id) and np.array_equal(outs[0][:, :P], p.cpu().numpy())
    tm.close()
