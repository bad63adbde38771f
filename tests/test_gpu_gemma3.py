"""Gemma-3 layer details on the GPU against the oracle: sliding-window
attention (local layers) on the tcgen05, mma.sync and fp32 attention kernels;
QK-norm in the QKV epilogue; sandwich norms; the local / global pattern with
its two RoPE bases; whole models in single-block and block mode (the window
then reaches across the committed context).  Tolerances as for the other
layers: 1e-4 relative for fp32 models, 2e-2 for bf16 ones."""
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


def bf16_tensor(shape, seed, std=1.0):
    bits = wl.normal(seed, 99, int(np.prod(shape)), 0.0, std, "bf16").reshape(shape)
    return torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).cuda(), O.widen(bits)


def f32_tensor(shape, seed, std=1.0):
    x = wl.normal(seed, 98, int(np.prod(shape)), 0.0, std, "f32").reshape(shape)
    return torch.from_numpy(x).cuda(), x.astype(np.float64)


def rel_l2(a, b):
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


# ------------------------------------------------------------------ windowed attention kernels
# pad 0 / stride % 8 == 0: tcgen05 kernel (key tiles below every row's window are skipped); pad 1: mma.sync
@pytest.mark.parametrize("hd,Hq,Hkv,rows,ctx,causal,window,pad", [
    (64, 4, 2, 300, 0, False, 64, 4), (64, 4, 2, 300, 0, True, 100, 4), (128, 4, 2, 260, 0, False, 130, 4),
    (128, 16, 8, 32, 1100, False, 1024, 0), (128, 16, 8, 32, 1100, True, 1024, 0), (128, 2, 1, 32, 700, False, 40, 0),
    (64, 8, 2, 20, 300, False, 7, 0), (128, 2, 1, 100, 130, True, 1, 0), (64, 4, 2, 48, 200, True, 500, 0),
    (128, 16, 8, 32, 1100, False, 1024, 1), (64, 4, 2, 300, 77, True, 33, 3)])
def test_window_attention_bf16(T, hd, Hq, Hkv, rows, ctx, causal, window, pad):
    B = 2
    L = ctx + rows
    stride = L + (-L) % 8 + pad
    q, qd = bf16_tensor((B, Hq, rows, hd), 5)
    k, kd = bf16_tensor((B, Hkv, stride, hd), 6)
    vt, vtd = bf16_tensor((B, Hkv, hd, stride), 7)       # V is passed transposed
    vd = vtd.transpose(0, 1, 3, 2)
    o = torch.empty((B * rows, Hq * hd), dtype=torch.bfloat16, device="cuda")
    T.tadm_attention(q, k, vt, o, Hq, Hkv, rows, ctx, causal, dtype=1, window=window)
    torch.cuda.synchronize()
    got = o.float().cpu().numpy().astype(np.float64).reshape(B, rows, Hq, hd)
    for b in range(B):
        ref = O.attention(qd[b], kd[b, :, :L], vd[b, :, :L], ctx + np.arange(rows), np.arange(L), causal,
                          window).transpose(1, 0, 2)
        assert rel_l2(got[b], ref) < 1e-2     # P is rounded to bf16 before P V


@pytest.mark.parametrize("hd,causal,window", [(64, False, 5), (64, True, 17), (32, False, 1)])
def test_window_attention_f32(T, hd, causal, window):
    B, Hq, Hkv, rows, ctx = 1, 4, 2, 45, 9
    stride = ctx + rows
    q, qd = f32_tensor((B, Hq, rows, hd), 8)
    k, kd = f32_tensor((B, Hkv, stride, hd), 9)
    v, vtd = f32_tensor((B, Hkv, hd, stride), 10)
    o = torch.empty((B * rows, Hq * hd), dtype=torch.float32, device="cuda")
    T.tadm_attention(q, k, v, o, Hq, Hkv, rows, ctx, causal, dtype=0, window=window)
    torch.cuda.synchronize()
    ref = O.attention(qd[0], kd[0], vtd[0].transpose(0, 2, 1), ctx + np.arange(rows), np.arange(stride), causal,
                      window).transpose(1, 0, 2)
    np.testing.assert_allclose(o.cpu().numpy().reshape(rows, Hq, hd), ref, rtol=1e-4, atol=1e-5)


# ------------------------------------------------------------------ whole models
G3 = dict(qk_norm=True, sandwich_norm=True, global_every=3, rope_theta_global=1e6)


def _setup(T, m, batch, rows, max_ctx=0, seed=1, affine_std=0.05):
    host = wl.make_weights(m, seed=seed, affine_std=affine_std)
    tm = T.TadmModel(m, T.upload_weights(m, host), max_batch=batch, max_rows=rows, max_ctx=max_ctx)
    return tm, O.Oracle(m, host)


def _step(tm, z, t, Tn, G, cache):
    B, R = z.shape
    zt = torch.from_numpy(z).cuda()
    logits = torch.empty((B * R, tm.model.vocab), dtype=torch.float32, device="cuda")
    tok = torch.empty(B * R, dtype=torch.int32, device="cuda")
    tm.tadm_denoise_step(zt, t, Tn, G, cache, logits=logits, tok=tok)
    tm.tadm_sync_status()
    return (zt.cpu().numpy(), logits.cpu().numpy().astype(np.float64).reshape(B, R, -1),
            tok.cpu().numpy().reshape(B, R))


def test_gemma3_fp32_block_mode_exact(T):
    """fp32 model (CUDA-core path) with every Gemma-3 detail, in block mode:
    a 40-token prompt, blocks of 16 and a window of 24, so that the local
    layers' windows cut into the committed context; the refresh, stale steps
    and commits against the oracle at the fp32 tolerance, the tokens exact."""
    m = wl.ModelConfig(vocab=512, d_model=128, n_heads=4, n_kv_heads=2, head_dim=32, ffn=256, n_shared=1,
                       n_anchor=3, n_denoise=2, dtype="f32", sliding_window=24, **G3)
    B, P, bl, Tn = 2, 40, 16, 4
    w = wl.Workload("t", m, batch=B, prompt_len=P, gen_len=3 * bl, steps_per_block=Tn, K=2, block_len=bl)
    tm, o = _setup(T, m, B, max(P, bl), max_ctx=P + 3 * bl)
    prompts = wl.make_prompts(w, batch=B, seed=9)
    tm.tadm_reset(B)
    tm.tadm_prefill(torch.from_numpy(prompts).cuda())
    sess = o.new_session(B)
    o.prefill(sess, prompts)
    cache = tm.new_cache(B, bl)
    for blk in range(3):
        zb = np.full((B, bl), m.mask_id, np.int32)
        for n in range(Tn):
            if n % 2 == 0:
                tm.tadm_anchor_forward(torch.from_numpy(zb).cuda(), Tn - n, cache)
                cache_o = o.anchor_forward(sess, zb)
            gz, gl, gt = _step(tm, zb, Tn - n, Tn, bl, cache)
            ref = o.denoise_step(sess, zb, cache_o, n, Tn, bl)
            assert rel_l2(gl, ref["logits"]) < 1e-4, (blk, n)
            assert np.array_equal(gz, ref["z"]), (blk, n)
            zb = gz
        tm.tadm_commit_block(torch.from_numpy(zb).cuda())
        o.commit_block(sess, zb)
    tm.tadm_sync_status()
    # the whole generation through tadm_generate equals the oracle's
    got = tm.generate(torch.from_numpy(prompts).cuda(), 3 * bl, Tn, 2, block_len=bl).cpu().numpy()
    ref = o.generate(prompts, 3 * bl, Tn, 2, block_len=bl)
    assert float(np.mean(got == ref)) >= 0.99


def test_gemma3_bf16_block_mode_split_k_projections(T):
    """bf16 Gemma-3 model (QK-norm, sandwich norms, a 48-key window) in block
    mode at batch 8 x 32-row blocks, d_model 1024: its 256-row QKV
    projections (split operand, K = 2048) run 256-wide CTA-pair tiles with
    split-K and the QKV epilogue in the ordered split-K reduction, and so do
    its 320-row prefill projections (the second pair tile ragged); the
    fp32-store sandwich projections split-K with the element-wise reduction.
    Teacher-forced steps (both sides continue from the oracle's canvas)
    across a commit."""
    m = wl.ModelConfig(vocab=2048, d_model=1024, n_heads=8, n_kv_heads=4, head_dim=64, ffn=2048, n_shared=1,
                       n_anchor=2, n_denoise=1, dtype="bf16", sliding_window=48, qkv_split=True, **G3)
    B, P, bl, Tn = 8, 40, 32, 4
    w = wl.Workload("t", m, batch=B, prompt_len=P, gen_len=2 * bl, steps_per_block=Tn, K=2, block_len=bl)
    tm, o = _setup(T, m, B, max(P, bl), max_ctx=P + 2 * bl)
    prompts = wl.make_prompts(w, batch=B, seed=9)
    tm.tadm_reset(B)
    tm.tadm_prefill(torch.from_numpy(prompts).cuda())
    sess = o.new_session(B)
    o.prefill(sess, prompts)
    cache = tm.new_cache(B, bl)
    worst = 0.0
    for blk in range(2):
        zb = np.full((B, bl), m.mask_id, np.int32)
        for n in range(Tn):
            if n % 2 == 0:
                tm.tadm_anchor_forward(torch.from_numpy(zb).cuda(), Tn - n, cache)
                cache_o = o.anchor_forward(sess, zb)
            gz, gl, gt = _step(tm, zb, Tn - n, Tn, bl, cache)
            ref = o.denoise_step(sess, zb, cache_o, n, Tn, bl)
            rel = rel_l2(gl, ref["logits"])
            worst = max(worst, rel)
            assert rel < 2e-2, (blk, n, rel)
            masked = zb == m.mask_id
            assert float(np.mean(gt[masked] == ref["tok"][masked])) >= 0.95, (blk, n)
            zb = ref["z"]
        tm.tadm_commit_block(torch.from_numpy(zb).cuda())
        o.commit_block(sess, zb)
    tm.tadm_sync_status()
    print(f"[gemma3 bf16 block mode, split-K projections] worst logits rel-L2 {worst:.3e}")


@pytest.mark.parametrize("fusion", ["gated_mlp", "paired_attn"])
def test_gemma3_bf16_single_block_stale_step(T, fusion):
    """bf16 model on tcgen05 (QK-norm in the QKV epilogue, sandwich norms,
    local layers with a 48-key window over a 200-row canvas, global layers on
    the second RoPE table): refresh, then a step on a later canvas with the
    stale cache."""
    extra = dict(fusion_rank=256, fusion_heads=4, glu="geglu", tied_lm_head=True) if fusion == "paired_attn" else {}
    m = wl.ModelConfig(vocab=4096, d_model=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=768, n_shared=1,
                       n_anchor=3, n_denoise=2, dtype="bf16", fusion=fusion, sliding_window=48, **G3, **extra)
    B, R = 2, 200
    w = wl.Workload("t", m, batch=B, prompt_len=40, gen_len=160, steps_per_block=16, K=4)
    tm, o = _setup(T, m, B, R)
    z0 = wl.random_canvas(w, B, R, 0.8, seed=7, start=40)
    z1 = wl.random_canvas(w, B, R, 0.5, seed=8, start=40)
    cache = tm.new_cache(B, R)
    tm.tadm_reset(B)
    tm.tadm_anchor_forward(torch.from_numpy(z0).cuda(), 16, cache)
    sess = o.new_session(B)
    cache_o = o.anchor_forward(sess, z0)
    gz, gl, gt = _step(tm, z1, 14, 16, 160, cache)
    ref = o.denoise_step(sess, z1, cache_o, 2, 16, 160)
    rel = rel_l2(gl, ref["logits"])
    assert rel < 2e-2, rel
    c2, t2 = O.confidence(gl.reshape(-1, m.vocab), m.mask_id)
    assert np.array_equal(gt.reshape(-1), t2)
    masked = z1 == m.mask_id
    assert float(np.mean(gt[masked] == ref["tok"][masked])) >= 0.95
    print(f"[gemma3 bf16 {fusion}] logits rel-L2 {rel:.3e}")


def test_posttrain_g3_full_width_reduced_depth():
    """'posttrain_g3' widths (d_model 5376, 32/16 heads of 128, FFN 21504
    GeGLU, vocab 262144, tied head, paired-attention fusion) with 1 + 5 + 1
    layers, so that layer 5 is global and the others local, a 256-key window
    and a 320-token prompt, batch 4: prefill, refresh and a stale step on the
    first block, whose local layers then see only part of the context."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()
    from paper_2609_37924_gb300 import TadmModel, upload_weights
    m = wl.get_workload("posttrain_g3", model_n_shared=1, model_n_anchor=5, model_n_denoise=1,
                        model_sliding_window=256).model
    B, P, bl, Tn, seed = 4, 320, 32, 32, 5
    w = wl.Workload("g3", m, batch=B, prompt_len=P, gen_len=4 * bl, steps_per_block=Tn, K=4, block_len=bl, seed=seed)
    host = wl.make_weights(m, seed=seed)
    tm = TadmModel(m, upload_weights(m, host), max_batch=B, max_rows=max(P, bl), max_ctx=P + 4 * bl)
    prompts = wl.make_prompts(w)
    z0 = np.full((B, bl), m.mask_id, np.int32)
    z1 = wl.random_canvas(w, B, bl, 0.6, seed=seed + 1)
    tm.tadm_reset(B)
    tm.tadm_prefill(torch.from_numpy(prompts).cuda())
    cache = tm.new_cache(B, bl)
    tm.tadm_anchor_forward(torch.from_numpy(z0).cuda(), Tn, cache)
    gz, gl, gt = _step(tm, z1, Tn - 1, Tn, bl, cache)
    del tm
    torch.cuda.empty_cache()
    b = B - 1
    o = O.Oracle(m, host)
    sess = o.new_session(1)
    o.prefill(sess, prompts[b:b + 1])
    cache_o = o.anchor_forward(sess, z0[b:b + 1])
    ref = o.denoise_step(sess, z1[b:b + 1], cache_o, 1, Tn, bl)
    rel = rel_l2(gl[b], ref["logits"][0])
    assert rel < 2e-2, rel
    masked = z1[b] == m.mask_id
    committed = masked & (gz[b] != m.mask_id)
    assert np.array_equal(gz[b][committed], ref["tok"][0][committed])
    agree = float(np.mean(gt[b][masked] == ref["tok"][0][masked]))
    assert agree >= 0.9, agree
    print(f"[fullsize posttrain_g3] logits rel-L2 {rel:.3e}, argmax agreement {agree:.4f}")
