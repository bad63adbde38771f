"""Kernel-level parity on the GPU, through the C ABI building blocks, against
the oracle (or its plain definitions) on the same seeded inputs."""
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


# ------------------------------------------------------------------------------- GEMM
@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (300, 520, 200), (1024, 768, 768), (77, 2304, 3072),
                                   (2048, 4096, 2048), (1, 256, 512)])
def test_gemm_bf16_tcgen05(T, M, N, K):
    A, a = bf16_tensor((M, K), 1)
    B, b = bf16_tensor((N, K), 2)
    C = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    T.tadm_gemm(A, B, C, dtype=1)
    torch.cuda.synchronize()
    ref = a @ b.T
    got = C.cpu().numpy().astype(np.float64)
    # fp32 accumulation of K exact bf16 products: error << 1e-5 of the row scale
    err = np.abs(got - ref).max() / (np.abs(a).max() * np.abs(b).max() * np.sqrt(K))
    assert np.isfinite(got).all() and err < 1e-5, err
    Cb = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    T.tadm_gemm(A, B, Cb, dtype=1)
    gb = Cb.float().cpu().numpy().astype(np.float64)
    assert np.all(np.abs(gb - ref) <= np.abs(ref) * 2.0 ** -8 + 1e-5 * np.sqrt(K))


@pytest.mark.parametrize("M,N,K", [(64, 64, 16), (100, 130, 70), (257, 1024, 256)])
def test_gemm_f32_cuda_cores(T, M, N, K):
    A, a = f32_tensor((M, K), 3)
    B, b = f32_tensor((N, K), 4)
    C = torch.empty((M, N), dtype=torch.float32, device="cuda")
    T.tadm_gemm(A, B, C, dtype=0)
    torch.cuda.synchronize()
    ref = a @ b.T
    err = np.abs(C.cpu().numpy() - ref).max() / np.sqrt(K)
    assert err < 1e-5, err


# -------------------------------------------------------------------------- attention
# kv_stride % 8 == 0 runs the tcgen05 kernel (128 virtual rows = query heads of
# a KV group x rows per CTA; 64-key tiles for hd 128 with < 256 virtual rows),
# the other strides the mma.sync kernel
@pytest.mark.parametrize("hd,Hq,Hkv,rows,ctx,causal,pad", [
    (64, 4, 4, 70, 0, False, 5), (64, 4, 2, 64, 0, True, 5), (128, 4, 2, 32, 37, False, 5),
    (128, 2, 1, 100, 130, True, 5), (64, 12, 12, 1024, 0, False, 0), (64, 4, 2, 300, 77, True, 3),
    (128, 4, 2, 260, 0, False, 4), (128, 2, 2, 512, 200, True, 0), (64, 2, 1, 200, 0, False, 1),
    # short rows on tcgen05: GQA group packing, heads straddling a 128-row tile, causal
    (128, 4, 2, 32, 37, False, 3), (128, 16, 8, 32, 200, True, 0), (64, 4, 2, 48, 40, True, 0),
    (128, 2, 1, 100, 130, True, 2), (64, 8, 2, 20, 300, False, 0),
    # hd 64 launches of more CTAs than SMs run the pipelined kernel (double-buffered S and P, 64-key
    # tiles): bidirectional, causal with a context and a ragged last tile, GQA
    (64, 12, 12, 1024, 0, True, 0), (64, 16, 8, 700, 100, True, 0), (64, 16, 4, 520, 44, False, 0)])
def test_attention_bf16(T, hd, Hq, Hkv, rows, ctx, causal, pad):
    B, stride = 2, ctx + rows + pad
    q, qd = bf16_tensor((B, Hq, rows, hd), 5)
    k, kd = bf16_tensor((B, Hkv, stride, hd), 6)
    vt, vtd = bf16_tensor((B, Hkv, hd, stride), 7)       # V is passed transposed
    v, vd = vt, vtd.transpose(0, 1, 3, 2)
    o = torch.empty((B * rows, Hq * hd), dtype=torch.bfloat16, device="cuda")
    T.tadm_attention(q, k, v, o, Hq, Hkv, rows, ctx, causal, dtype=1)
    torch.cuda.synchronize()
    got = o.float().cpu().numpy().astype(np.float64).reshape(B, rows, Hq, hd)
    L = ctx + rows
    for b in range(B):
        pos = ctx + np.arange(rows)
        kpos = np.arange(L)
        # keys < ctx are context: always visible; the causal test covers the rest
        ref = O.attention(qd[b], kd[b, :, :L], vd[b, :, :L], pos, kpos, causal).transpose(1, 0, 2)
        rel = np.linalg.norm(got[b] - ref) / np.linalg.norm(ref)
        assert rel < 1e-2, rel      # P is rounded to bf16 before P V


@pytest.mark.parametrize("hd,causal", [(64, False), (64, True), (32, False)])
def test_attention_f32(T, hd, causal):
    B, Hq, Hkv, rows, ctx = 1, 4, 2, 45, 9
    stride = ctx + rows
    q, qd = f32_tensor((B, Hq, rows, hd), 8)
    k, kd = f32_tensor((B, Hkv, stride, hd), 9)
    v, vtd = f32_tensor((B, Hkv, hd, stride), 10)        # V is passed transposed
    vd = vtd.transpose(0, 1, 3, 2)
    o = torch.empty((B * rows, Hq * hd), dtype=torch.float32, device="cuda")
    T.tadm_attention(q, k, v, o, Hq, Hkv, rows, ctx, causal, dtype=0)
    torch.cuda.synchronize()
    ref = O.attention(qd[0], kd[0], vd[0], ctx + np.arange(rows), np.arange(stride), causal).transpose(1, 0, 2)
    np.testing.assert_allclose(o.cpu().numpy().reshape(rows, Hq, hd), ref, rtol=1e-4, atol=1e-5)


# ------------------------------------------------------------------ confidence + top-k
def test_confidence_bit_exact_argmax(T):
    rows, V = 333, 32768
    lg, l64 = f32_tensor((rows, V), 11, std=2.0)
    host = lg.cpu().numpy()
    host[5, 100] = host[5, 200] = host[5].max() + 1.0        # tie -> lower id
    host[7, V - 1] = host[7].max() + 5.0                     # MASK largest -> excluded
    lg = torch.from_numpy(host).cuda()
    conf = torch.empty(rows, dtype=torch.float32, device="cuda")
    tok = torch.empty(rows, dtype=torch.int32, device="cuda")
    T.tadm_confidence(lg, V - 1, conf, tok)
    torch.cuda.synchronize()
    rc, rt = O.confidence(host.astype(np.float64), V - 1)
    assert np.array_equal(tok.cpu().numpy(), rt)
    assert tok.cpu().numpy()[5] == 100 and tok.cpu().numpy()[7] != V - 1
    # fp32 sum of V terms vs the fp64 sum: relative error bound ~ log2(V) * 2^-24 per term, use 4e-6
    assert np.max(np.abs(conf.cpu().numpy() - rc) / rc) < 4e-6


def test_topk_unmask_bit_exact_from_same_keys(T):
    B, R, mask = 6, 300, 999
    rng = np.random.default_rng(5)
    for k in (1, 3, 6, 40, 400):
        z = np.where(rng.random((B, R)) < 0.7, mask, rng.integers(0, 999, (B, R))).astype(np.int32)
        conf = rng.choice(np.float32([0.1, 0.25, 0.5, 0.75]), size=(B, R)).astype(np.float32)  # many ties
        tok = rng.integers(0, 999, (B, R)).astype(np.int32)
        zt = torch.from_numpy(z).cuda()
        sel = torch.empty((B, k), dtype=torch.int32, device="cuda")
        T.tadm_topk_unmask(zt, torch.from_numpy(conf).cuda(), torch.from_numpy(tok).cuda(), k, mask, sel)
        torch.cuda.synchronize()
        zg, sg = zt.cpu().numpy(), sel.cpu().numpy()
        for b in range(B):
            p = O.select_topk(z[b], conf[b].astype(np.float64), k, mask)
            zr = z[b].copy()
            zr[p] = tok[b, p]
            assert np.array_equal(zg[b], zr)
            assert list(sg[b, : p.size]) == list(p) and np.all(sg[b, p.size:] == -1)


@pytest.mark.parametrize("rows,d,V,dtype", [(300, 768, 32768, 1), (129, 256, 5000, 1), (70, 256, 1024, 0)])
def test_head_confidence_fused(T, rows, d, V, dtype):
    mk = bf16_tensor if dtype else f32_tensor
    x, xd = mk((rows, d), 12)
    w, wd = mk((V, d), 13, std=0.05)
    conf = torch.empty(rows, dtype=torch.float32, device="cuda")
    tok = torch.empty(rows, dtype=torch.int32, device="cuda")
    scratch = torch.empty(T.tadm_head_scratch_size(rows, V, dtype), dtype=torch.uint8, device="cuda")
    T.tadm_head_confidence(x, w, V - 1, conf, tok, scratch, dtype)
    logits = torch.empty((rows, V), dtype=torch.float32, device="cuda")
    T.tadm_gemm(x, w, logits, dtype=dtype)          # same accumulation, materialised
    torch.cuda.synchronize()
    rc, rt = O.confidence(logits.cpu().numpy().astype(np.float64), V - 1)
    assert np.array_equal(tok.cpu().numpy(), rt)
    assert np.max(np.abs(conf.cpu().numpy() - rc) / rc) < 4e-6
    lf = xd @ wd.T                                   # fp64 from the same inputs
    assert np.linalg.norm(logits.cpu().numpy() - lf) / np.linalg.norm(lf) < 1e-5


@pytest.mark.parametrize("hd,Hq,Hkv,rows,ctx,causal", [(128, 4, 2, 32, 40, False), (128, 4, 2, 32, 72, True),
                                                      (64, 4, 2, 32, 40, False)])
def test_attention_short_rows_tcgen05_as_accurate_as_mma_sync(T, hd, Hq, Hkv, rows, ctx, causal):
    """The same Q, K, V through the tcgen05 kernel (KV stride a multiple of 8)
    and the mma.sync kernel (stride one more): both within the bf16-P bound of
    the fp64 reference, and the tcgen05 error no larger than 1.5x the other's."""
    B = 2
    L = ctx + rows
    q, qd = bf16_tensor((B, Hq, rows, hd), 15)
    k8, kd = bf16_tensor((B, Hkv, L, hd), 16)
    vt8, vtd = bf16_tensor((B, Hkv, hd, L), 17)
    errs = []
    for stride in (L + (-L) % 8, L + (-L) % 8 + 1):
        k = torch.zeros((B, Hkv, stride, hd), dtype=torch.bfloat16, device="cuda")
        vt = torch.zeros((B, Hkv, hd, stride), dtype=torch.bfloat16, device="cuda")
        k[:, :, :L] = k8
        vt[..., :L] = vt8
        o = torch.empty((B * rows, Hq * hd), dtype=torch.bfloat16, device="cuda")
        T.tadm_attention(q, k, vt, o, Hq, Hkv, rows, ctx, causal, dtype=1)
        torch.cuda.synchronize()
        got = o.float().cpu().numpy().astype(np.float64).reshape(B, rows, Hq, hd)
        e = 0.0
        for b in range(B):
            ref = O.attention(qd[b], kd[b], vtd[b].transpose(0, 2, 1), ctx + np.arange(rows), np.arange(L),
                              causal).transpose(1, 0, 2)
            e = max(e, np.linalg.norm(got[b] - ref) / np.linalg.norm(ref))
        errs.append(e)
    print(f"[short-row attention hd {hd}] rel-L2 tcgen05 {errs[0]:.2e}  mma.sync {errs[1]:.2e}")
    assert errs[0] < 1e-2 and errs[1] < 1e-2
    assert errs[0] <= 1.5 * errs[1], errs


@pytest.mark.parametrize("B,Hq,Hkv,rows,ctx,causal", [
    (16, 16, 8, 32, 777, False),     # block-diffusion steps: 32 rows x a GQA group over a long context
    (8, 32, 16, 32, 1100, False),    # post-train widths
    (2, 16, 8, 500, 100, True),      # a causal commit / prefill pass over a context
    (1, 64, 64, 300, 0, False)])     # ragged rows, many heads
def test_attention_pipelined_hd128(T, B, Hq, Hkv, rows, ctx, causal):
    """hd 128 launches that fill 80-100 % of the SMs in one wave run the
    pipelined kernel (one CTA per SM, double-buffered S and P, four 32 KB K /
    V stages); the others attn_tc_kernel."""
    hd = 128
    L = ctx + rows
    stride = L + (-L) % 8
    q, qd = bf16_tensor((B, Hq, rows, hd), 25)
    k, kd = bf16_tensor((B, Hkv, stride, hd), 26)
    vt, vtd = bf16_tensor((B, Hkv, hd, stride), 27)
    o = torch.empty((B * rows, Hq * hd), dtype=torch.bfloat16, device="cuda")
    T.tadm_attention(q, k, vt, o, Hq, Hkv, rows, ctx, causal, dtype=1)
    torch.cuda.synchronize()
    got = o.float().cpu().numpy().astype(np.float64).reshape(B, rows, Hq, hd)
    for b in sorted({0, B - 1}):
        ref = O.attention(qd[b], kd[b, :, :L], vtd[b, :, :, :L].transpose(0, 2, 1), ctx + np.arange(rows),
                          np.arange(L), causal).transpose(1, 0, 2)
        rel = np.linalg.norm(got[b] - ref) / np.linalg.norm(ref)
        assert rel < 1e-2, (b, rel)
