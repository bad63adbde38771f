"""The entropy-bound sampler with self-conditioning (Alg. 2, NEXT row) on
the GPU, through the C ABI, against the oracle and the shared Philox
generator."""
import numpy as np
import pytest

import workloads as wl
from oracle import tadm_oracle as O

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

# fp32 sums of V terms: each lane adds V / 512 of them in order, a warp
# butterfly adds 32 lanes (5 levels) and one thread the 16 warp segments, so
# the relative error of Z and W stays below (V / 512 + 21) 2^-24 (3.1e-5 at
# V = 262144), plus a few ulp from exp and log.  The
# entropy is log Z - W / Z, so its error stays below that bound times
# (1 + |W / Z|) with W / Z = sum p a; the tests allow four times the bound.
def z_rel_bound(V):
    return (V / 512 + 21) * 2.0 ** -24


def h_tol(V, mean_a):
    return 4.0 * z_rel_bound(V) * (1.0 + abs(mean_a)) + 1e-6


@pytest.fixture(scope="module")
def T():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()
    from paper_2609_37924_gb300 import tadm
    return tadm


def rows_case(V, B, G, seed):
    rng = np.random.default_rng(seed)
    scale = np.where(rng.random((B * G, 1)) < 0.3, 12.0, np.where(rng.random((B * G, 1)) < 0.5, 0.3, 3.0))
    logits = (rng.standard_normal((B * G, V)) * scale).astype(np.float32)
    logits[:5, 7] = logits[:5].max(axis=1) + 40.0          # near one-hot rows (H ~ 0)
    logits[5, :] = 1.25                                      # all equal: argmax is id 0, H = log(V - 1)
    return logits


def draw_valid(l64, tau, mask, u, tok, tol=2e-5):
    """A draw that differs from the oracle's is valid when u * Z lies within
    tol * Z of an edge of tok's CDF interval (fp32 vs fp64 running sums)."""
    a = l64 / tau
    a[mask] = -np.inf
    e = np.exp(a - a.max())
    c = np.cumsum(e)
    goal = u * c[-1]
    return e[tok] > 0 and c[tok] - e[tok] - tol * c[-1] <= goal <= c[tok] + tol * c[-1]


@pytest.mark.parametrize("V", [1000, 32768, 60000, 262144])     # 60000, 262144: rows beyond shared memory
def test_eb_update_matches_the_oracle(T, V):
    """One Alg. 2 step from the same logits: argmax (n = 1) exact; entropy,
    Z and p = q / Z within the fp32 bound; draws equal to the oracle's or on
    a CDF edge; accepted set and re-noise tokens exact given the kernel's
    entropies (the oracle's accept rule run on them)."""
    B, R, first, mask, seed, step, tau = 2, 72, 8, V - 1, 4321, 5, 0.6
    G = R - first
    logits = rows_case(V, B, G, V)
    lt = torch.from_numpy(logits).cuda()
    z0 = np.random.default_rng(1).integers(0, V - 1, (B, R)).astype(np.int32)
    ent = torch.empty(B * G, dtype=torch.float32, device="cuda")
    probs = torch.empty((B * G, V), dtype=torch.float32, device="cuda")
    zsum = torch.empty(B * G, dtype=torch.float32, device="cuda")
    # n = 1: the argmax
    z = torch.from_numpy(z0).cuda()
    T.tadm_eb_update(z, lt, first, mask, tau, 0.1, True, seed, step, ent)
    am = z.cpu().numpy()
    # n > 1, eta = inf: every position keeps its draw
    z = torch.from_numpy(z0).cuda()
    T.tadm_eb_update(z, lt, first, mask, tau, float("inf"), False, seed, step, ent, probs, zsum)
    draws, H, Q = z.cpu().numpy(), ent.cpu().numpy().astype(np.float64), probs.cpu().numpy()
    Zg = zsum.cpu().numpy().astype(np.float64)
    # n > 1, eta = 0.5: accepted positions keep the draw, the rest re-noise
    z = torch.from_numpy(z0).cuda()
    T.tadm_eb_update(z, lt, first, mask, tau, 0.5, False, seed, step, ent)
    acc = z.cpu().numpy()
    torch.cuda.synchronize()
    u = wl.remdm_uniforms(seed, step, B, R)
    assert np.array_equal(am[:, :first], z0[:, :first]) and np.array_equal(draws[:, :first], z0[:, :first])
    edge = 0
    for b in range(B):
        for g in range(G):
            j = b * G + g
            l64 = logits[j].astype(np.float64)
            p, a_max, h, d = O.eb_row(l64, tau, mask, u[b, first + g, 0])
            assert am[b, first + g] == a_max, (b, g)
            mean_a = float(np.sum(p[p > 0] * (l64[p > 0] - l64[:mask].max()) / tau))
            assert abs(H[j] - h) <= h_tol(V, mean_a), (b, g, H[j], h)
            a = (l64 - l64[:mask].max()) / tau
            a[mask] = -np.inf
            Zo = np.exp(a).sum()
            assert abs(Zg[j] - Zo) <= 4.0 * z_rel_bound(V) * Zo, (b, g, Zg[j], Zo)
            assert np.allclose(Q[j] / Zg[j], p, rtol=5e-5 + 4.0 * z_rel_bound(V), atol=1e-12), (b, g)
            if draws[b, first + g] != d:
                edge += 1
                assert draw_valid(l64, tau, mask, u[b, first + g, 0], draws[b, first + g]), (b, g)
    assert edge <= 2, edge
    for b in range(B):
        Hb = H[b * G:(b + 1) * G]
        ok = O.eb_accept(Hb, 0.5)
        order = np.lexsort((np.arange(G), Hb))
        margin = np.abs(np.cumsum(Hb[order]) - Hb[order] - 0.5)
        close = np.zeros(G, bool)
        close[order[margin < 1e-9]] = True
        noise = np.floor(u[b, first:, 1] * (V - 1)).astype(np.int32)
        want = np.where(ok, draws[b, first:], noise)
        assert np.array_equal(acc[b, first:][~close], want[~close]), b
        assert ok.sum() >= 1 and np.all(acc[b, first:] != mask)


def test_eb_bf16_probabilities(T):
    """The bf16 q = exp((l - max) / tau) (the self-conditioning operand of
    bf16 models) is q rounded to bf16."""
    B, R, first, V = 1, 40, 8, 4096
    G = R - first
    logits = rows_case(V, B, G, 7)
    z = torch.zeros((B, R), dtype=torch.int32, device="cuda")
    ent = torch.empty(B * G, dtype=torch.float32, device="cuda")
    probs = torch.empty((B * G, V), dtype=torch.bfloat16, device="cuda")
    T.tadm_eb_update(z, torch.from_numpy(logits).cuda(), first, V - 1, 0.7, 0.1, False, 3, 0, ent, probs)
    got = probs.float().cpu().numpy()
    for j in range(G):
        l64 = logits[j].astype(np.float64)
        q = np.exp((l64 - l64[:V - 1].max()) / 0.7)
        q[V - 1] = 0.0
        assert np.allclose(got[j], q, rtol=2.0 ** -8 + 5e-5, atol=1e-30), j


def test_eb_draw_frequencies_follow_p(T):
    """4096 positions with the same logits, eta = inf: the draws' empirical
    frequencies match p."""
    V, G, tau = 24, 4096, 0.8
    row = np.linspace(-2.0, 2.0, V).astype(np.float32)[::-1].copy()
    logits = np.tile(row, (G, 1))
    z = torch.zeros((1, G), dtype=torch.int32, device="cuda")
    ent = torch.empty(G, dtype=torch.float32, device="cuda")
    T.tadm_eb_update(z, torch.from_numpy(logits).cuda(), 0, V - 1, tau, float("inf"), False, 99, 0, ent)
    got = np.bincount(z.cpu().numpy().ravel(), minlength=V) / G
    p = O.eb_row(row.astype(np.float64), tau, V - 1, 0.5)[0]
    assert got[V - 1] == 0.0 and 0.5 * np.abs(got - p).sum() < 0.03


@pytest.mark.parametrize("self_cond", [True, False])
def test_generate_entropy_bound_matches_the_oracle_fp32(T, self_cond):
    """Whole Alg. 2 generations of the fp32 tiny workload (T = 16, K = 2,
    eta = 0.1, tau 0.8 -> 0.4): the GPU follows the oracle's trajectory (same
    draws, fp32 vs fp64 logits)."""
    w = wl.WORKLOADS["tiny"]
    m = w.model
    host = wl.make_weights(m, seed=0)
    tm = T.TadmModel(m, T.upload_weights(m, host), max_batch=1, max_rows=w.total_len)
    o = O.Oracle(m, host)
    prompts = wl.make_prompts(w)
    steps, K, seed = 16, 2, 11
    out = torch.empty((1, w.total_len), dtype=torch.int32, device="cuda")
    nbytes = tm.tadm_eb_scratch_bytes(1, w.gen_len, self_cond)
    scratch = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    tm.tadm_generate_entropy_bound(torch.from_numpy(prompts).cuda(), out, w.gen_len, steps, K, 0.1, 0.8, 0.4, seed,
                                   scratch, self_cond)
    tm.tadm_sync_status()
    got = out.cpu().numpy()
    ref = o.generate_entropy_bound(prompts, w.gen_len, steps, K, 0.1, 0.8, 0.4,
                                   lambda i: wl.remdm_uniforms(seed, i, 1, w.total_len), self_cond=self_cond)
    assert np.all(got != m.mask_id) and np.array_equal(got[:, :w.prompt_len], prompts)
    assert float(np.mean(got == ref)) >= 0.98, float(np.mean(got == ref))
    c = tm.tadm_get_counters()
    assert c["denoise_steps"] == steps and c["anchor_calls"] == (steps + K - 1) // K
    tm.close()


def test_generate_entropy_bound_bf16_completes(T):
    """bf16 test model, batch 4, self-conditioning through the tcgen05 GEMM:
    the prompt is untouched, no MASK is left, the same seed reproduces the
    same tokens, and self-conditioning changes the result."""
    m = wl.ModelConfig(vocab=4096, d_model=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=768, n_anchor=3,
                       n_denoise=2, dtype="bf16")
    B, P, G, steps = 4, 32, 160, 12
    w = wl.Workload("t", m, batch=B, prompt_len=P, gen_len=G, steps_per_block=steps, K=3)
    tm = T.TadmModel(m, T.upload_weights(m, wl.make_weights(m, seed=2)), max_batch=B, max_rows=P + G)
    p = torch.from_numpy(wl.make_prompts(w, batch=B, seed=3)).cuda()
    scratch = torch.empty(tm.tadm_eb_scratch_bytes(B, G, True), dtype=torch.uint8, device="cuda")
    outs = []
    for sc in (True, True, False):
        out = torch.empty((B, P + G), dtype=torch.int32, device="cuda")
        tm.tadm_generate_entropy_bound(p, out, G, steps, 3, 0.1, 0.8, 0.4, 17, scratch, sc)
        tm.tadm_sync_status()
        outs.append(out.cpu().numpy())
    assert np.array_equal(outs[0], outs[1]) and not np.array_equal(outs[0], outs[2])
    assert np.all(outs[0] != m.mask_id) and np.array_equal(outs[0][:, :P], p.cpu().numpy())
    tm.close()


def test_eb_update_at_the_post_train_launch_shape(T):
    """The sampler launch of the post-train canvas workload (batch 8, 256
    generated positions after a 256-token prompt, V = 262144): on sampled
    rows argmax exact, entropy within the fp32 bound, draws exact or on a
    CDF edge; for every sequence the accepted set and re-noise tokens exact
    given the kernel's entropies; the prompt untouched and no MASK."""
    B, P, G, V, tau, eta, seed, step = 8, 256, 256, 262144, 0.6, 0.1, 77, 9
    R, mask = P + G, V - 1
    rng = np.random.default_rng(5)
    logits = np.empty((B * G, V), np.float32)
    for j in range(B * G):                          # mixed flat and peaked rows, as in the generation
        logits[j] = rng.standard_normal(V, dtype=np.float32) * np.float32((0.5, 2.0, 6.0)[j % 3])
    lt = torch.from_numpy(logits).cuda()
    z0 = rng.integers(0, V - 1, (B, R)).astype(np.int32)
    ent = torch.empty(B * G, dtype=torch.float32, device="cuda")
    z = torch.from_numpy(z0).cuda()
    T.tadm_eb_update(z, lt, P, mask, tau, eta, True, seed, step, ent)
    am = z.cpu().numpy()
    z = torch.from_numpy(z0).cuda()
    T.tadm_eb_update(z, lt, P, mask, tau, float("inf"), False, seed, step, ent)
    draws, H = z.cpu().numpy(), ent.cpu().numpy().astype(np.float64)
    z = torch.from_numpy(z0).cuda()
    T.tadm_eb_update(z, lt, P, mask, tau, eta, False, seed, step, ent)
    acc = z.cpu().numpy()
    torch.cuda.synchronize()
    u = wl.remdm_uniforms(seed, step, B, R)
    for out in (am, draws, acc):
        assert np.array_equal(out[:, :P], z0[:, :P]) and np.all(out[:, P:] != mask)
    edge = 0
    for j in rng.choice(B * G, 24, replace=False):
        b, g = divmod(int(j), G)
        l64 = logits[j].astype(np.float64)
        p, a_max, h, d = O.eb_row(l64, tau, mask, u[b, P + g, 0])
        assert am[b, P + g] == a_max, (b, g)
        mean_a = float(np.sum(p[p > 0] * (l64[p > 0] - l64[:mask].max()) / tau))
        assert abs(H[j] - h) <= h_tol(V, mean_a), (b, g, H[j], h)
        if draws[b, P + g] != d:
            edge += 1
            assert draw_valid(l64, tau, mask, u[b, P + g, 0], draws[b, P + g]), (b, g)
    assert edge <= 1, edge
    for b in range(B):
        Hb = H[b * G:(b + 1) * G]
        order = np.lexsort((np.arange(G), Hb))
        margin = np.abs(np.cumsum(Hb[order]) - Hb[order] - eta)
        close = np.zeros(G, bool)
        close[order[margin < 1e-9]] = True
        want = np.where(O.eb_accept(Hb, eta), draws[b, P:], np.floor(u[b, P:, 1] * (V - 1)).astype(np.int32))
        assert np.array_equal(acc[b, P:][~close], want[~close]), b


def test_generate_entropy_bound_one_step_bf16_argmax(T):
    """T = 1 on the bf16 test model: the output is the argmax of the fused
    prediction on step 1's noise canvas, taken by the sampler from the
    tcgen05 output head's per-tile partials.  Against the oracle's fp64
    logits (std 0.32): equal wherever the oracle's top-2 gap exceeds 2e-2,
    about 15x the bf16 path's typical logit error (rel-L2 4e-3, ~1.3e-3
    absolute), and >= 90 % overall."""
    m = wl.ModelConfig(vocab=4096, d_model=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=768, n_anchor=3,
                       n_denoise=2, dtype="bf16")
    B, P, G, seed = 2, 16, 48, 23
    w = wl.Workload("t", m, batch=B, prompt_len=P, gen_len=G, steps_per_block=1, K=1)
    host = wl.make_weights(m, seed=4)
    tm = T.TadmModel(m, T.upload_weights(m, host), max_batch=B, max_rows=P + G)
    prompts = wl.make_prompts(w, batch=B, seed=6)
    out = torch.empty((B, P + G), dtype=torch.int32, device="cuda")
    scratch = torch.empty(tm.tadm_eb_scratch_bytes(B, G, True), dtype=torch.uint8, device="cuda")
    tm.tadm_generate_entropy_bound(torch.from_numpy(prompts).cuda(), out, G, 1, 1, 0.1, 0.8, 0.4, seed, scratch, True)
    tm.tadm_sync_status()
    got = out.cpu().numpy()
    tm.close()
    o = O.Oracle(m, host)
    u = wl.remdm_uniforms(seed, 1, B, P + G)
    pos = np.arange(P + G)
    agree = total = 0
    for b in range(B):
        zb = np.concatenate([prompts[b], np.floor(u[b, P:, 1] * (m.vocab - 1)).astype(np.int32)])
        c = o.S(zb, pos, None)
        lg = o.lm_head(o.D_hidden(o.fuse(c, o.make_cache(c, o.A(c, pos, None))), pos, None))[P:]
        lg[:, m.mask_id] = -np.inf
        top2 = np.sort(lg, axis=1)[:, -2:]
        sure = top2[:, 1] - top2[:, 0] > 2e-2
        ref = np.argmax(lg, axis=1)
        assert np.array_equal(got[b, P:][sure], ref[sure]), b
        assert np.array_equal(got[b, :P], prompts[b])
        agree += int(np.sum(got[b, P:] == ref))
        total += G
    assert agree >= 0.90 * total, (agree, total)
