"""Token-agreement floor of an ideal bf16 tensor-core path (test infrastructure).

A bf16 tensor-core implementation must round every GEMM / attention operand
to bf16: the normalised activations entering the QKV, gate/up and output-head
GEMMs, Q, K and V after RoPE, the softmax numerators P, the attention output,
the GLU product and the fusion MLP's inputs (App. C.2).  Everything else
(accumulation, residual stream, norms, softmax sums) can stay exact.  This
script runs the oracle's arithmetic with exactly those roundings added (an
``Oracle`` subclass; weights, sampler and loop are the oracle's) through the
teacher-forced agreement protocol of the GPU model tests, with the fp64
oracle as the teacher, and writes the agreement it reaches to
``tests/golden/bf16_floor_small.json``.

That number is the floor of the protocol: no bf16 path, however exact its
accumulation, does better except by luck of rounding, because on random-init
weights the last masked positions of a block have near-tied top-2 logits and
a rounding of relative size 2^-9 flips some of them.  The GPU test compares
its own agreement with it.

Run (about 40 minutes of CPU):  python tests/bf16_floor.py
"""
from __future__ import annotations

import json
import math
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))

import workloads as wl  # noqa: E402
from oracle import tadm_oracle as O  # noqa: E402

# the agreement protocol of test_committed_token_agreement_teacher_forced[small_workload_dims]
PROTOCOL = dict(workload="small", batch=8, prompt_len=64, gen_len=192, steps=32, K=4, weight_seed=7,
                affine_std=0.0, prompt_seed=17)


def to_bf16(x: np.ndarray) -> np.ndarray:
    """Round to the nearest bf16 value (ties to even), returned as float64.
    Goes through float32 first, as the GPU's fp32 accumulators do."""
    a = np.ascontiguousarray(x, dtype=np.float32)
    bits = a.view(np.uint32).astype(np.uint64)
    rounded = ((bits + 0x7FFF + ((bits >> 16) & 1)) >> 16) << 16
    return rounded.astype(np.uint32).view(np.float32).astype(np.float64)


# The tensor-core operand sites of the path, in the order the data meets them.
SITES = ("qkv_in", "qkv", "p", "o_in", "ffn_in", "down_in", "fusion_u", "fusion_hid", "head_in")


class Bf16Oracle(O.Oracle):
    """The oracle with bf16 operands at every tensor-core input, except the
    sites named in ``exact`` ("site" everywhere, "site@net" in one network:
    shared, anchor or denoise), which keep the oracle's arithmetic."""

    exact = frozenset()

    def _r(self, site, x):
        if site in self.exact or f"{site}@{self._net}" in self.exact:
            return x
        return to_bf16(x)

    def layer(self, name, x, pos, seq, causal, keep_kv):
        """O.Oracle.layer with the tensor-core operands rounded; block mode
        (KV context, causal passes) and the Gemma-3 options included."""
        self._net = name.split(".")[0]
        r = self._r
        m = self.m
        hd, Hq, Hkv, F = m.head_dim, m.n_heads, m.n_kv_heads, m.ffn
        L = x.shape[0]
        window, theta = self.layer_kind(name)
        n = r("qkv_in", O.rms_norm(x, self.W(name + "attn_norm"), m.norm_eps))
        qkv = O.linear(n, self.W(name + "wqkv"))
        q = qkv[:, : Hq * hd].reshape(L, Hq, hd).transpose(1, 0, 2)
        k = qkv[:, Hq * hd: (Hq + Hkv) * hd].reshape(L, Hkv, hd).transpose(1, 0, 2)
        v = qkv[:, (Hq + Hkv) * hd:].reshape(L, Hkv, hd).transpose(1, 0, 2)
        if getattr(m, "qk_norm", False):
            q = O.rms_norm(q, self.W(name + "q_norm"), m.norm_eps)
            k = O.rms_norm(k, self.W(name + "k_norm"), m.norm_eps)
        q, k = O.rope(q, pos, theta), O.rope(k, pos, theta)
        q, k, v = r("qkv", q), r("qkv", k), r("qkv", v)     # the K / V cache holds these bf16 values
        if seq is not None and name in seq.kv:
            kc, vc = seq.kv[name]
            k_all, v_all = np.concatenate([kc, k], axis=1), np.concatenate([vc, v], axis=1)
            k_pos = np.concatenate([np.arange(kc.shape[1]), pos])
        else:
            k_all, v_all, k_pos = k, v, pos
        o = self._attention(q, k_all, v_all, pos, k_pos, causal, window, "p")
        a = O.linear(r("o_in", o.transpose(1, 0, 2).reshape(L, Hq * hd)), self.W(name + "wo"))
        if getattr(m, "sandwich_norm", False):
            a = O.rms_norm(a, self.W(name + "post_attn_norm"), m.norm_eps)
        x = x + a
        n = r("ffn_in", O.rms_norm(x, self.W(name + "ffn_norm"), m.norm_eps))
        gu = O.linear(n, self.W(name + "wgu"))
        g, u = gu[:, :F], gu[:, F:]
        act = O.silu(g) if m.glu == "swiglu" else O.gelu_tanh(g)
        f = O.linear(r("down_in", act * u), self.W(name + "wdown"))
        if getattr(m, "sandwich_norm", False):
            f = O.rms_norm(f, self.W(name + "post_ffn_norm"), m.norm_eps)
        if keep_kv and seq is not None:
            if name in seq.kv:
                seq.kv[name] = [k_all, v_all]
            else:
                seq.kv[name] = [k, v]
        return x + f

    def _attention(self, q, k, v, q_pos, k_pos, causal, window, site):
        """O.attention with the unnormalised numerators P rounded at `site`
        (the row sums stay exact: fp32 on the GPU)."""
        Hq, _, hd = q.shape
        group = Hq // k.shape[0]
        out = np.empty_like(q)
        for h in range(Hq):
            s = q[h] @ k[h // group].T / math.sqrt(hd)
            if causal:
                s = np.where(k_pos[None, :] <= q_pos[:, None], s, O.NEG_INF)
            if window > 0:
                s = np.where(q_pos[:, None] - k_pos[None, :] < window, s, O.NEG_INF)
            pe = np.exp(s - s.max(axis=-1, keepdims=True))
            out[h] = (self._r(site, pe) @ v[h // group]) / pe.sum(axis=-1, keepdims=True)
        return out

    # paired-attention fusion (App. C.1): the GPU rounds the scaled inputs of
    # W_C / W_H, J, the mixer's Q, K, V, P and output, R (the W_1 input), the
    # SiLU hidden, F and M (the W_up input); Z, U, phi, R and the gate are fp32
    def mixer(self, Z, U):
        self._net = "fusion"
        r = self._r
        rk, H = self.m.fusion_rank, self.m.fusion_heads
        L = Z.shape[0]
        J = r("pa_j", np.concatenate([Z, U], axis=-1))
        wqkv = self.W("fusion.wqkv")
        q = r("pa_qkv", O.linear(J, wqkv[:rk]).reshape(L, H, rk // H).transpose(1, 0, 2))
        k = r("pa_qkv", O.linear(J, wqkv[rk:2 * rk]).reshape(L, H, rk // H).transpose(1, 0, 2))
        v = r("pa_qkv", O.linear(J, wqkv[2 * rk:]).reshape(L, H, rk // H).transpose(1, 0, 2))
        pos = np.arange(L)
        o = self._attention(q, k, v, pos, pos, False, 0, "pa_p").transpose(1, 0, 2).reshape(L, rk)
        R = Z + O.linear(r("pa_o", o), self.W("fusion.wo"))
        hid = r("pa_hid", O.silu(O.linear(r("pa_r", R), self.W("fusion.w1"))))
        return R + O.linear(hid, self.W("fusion.w2"))

    def paired_refresh(self, C0, H0):
        self._net = "fusion"
        r = self._r
        sC, sH = self._rms_scale(C0), self._rms_scale(H0)
        Z0 = O.linear(r("pa_in", C0 / sC), self.W("fusion.wc"))
        U = O.linear(r("pa_in", H0 / sH), self.W("fusion.wh"))
        return {"H0": H0, "C0": C0, "sC": sC, "sH": sH, "Z0": Z0, "U": U, "phi0": self.mixer(Z0, U)}

    def fusion_paired_attn(self, C, st):
        self._net = "fusion"
        r = self._r
        Z = O.linear(r("pa_in", C / st["sC"]), self.W("fusion.wc"))
        M = self.mixer(Z, st["U"]) - st["phi0"]
        self._net = "fusion"
        F = r("pa_f", np.concatenate([st["U"], st["Z0"], Z - st["Z0"], M], axis=-1))
        g = O.sigmoid(O.linear(O.silu(O.linear(F, self.W("fusion.wg1"))), self.W("fusion.wg2"), self.W("fusion.bg")))
        return st["H0"] + g * st["sH"] * O.linear(r("pa_m", M), self.W("fusion.wup"))

    def fusion_gated_mlp(self, c, h):
        self._net = "fusion"
        r = self._r
        m, d, eps = self.m, self.m.d_model, self.m.norm_eps
        s = O.layer_norm(c, self.W("fusion.ln_c.w"), self.W("fusion.ln_c.b"), eps)
        a = O.layer_norm(h, self.W("fusion.ln_h.w"), self.W("fusion.ln_h.b"), eps)
        u = r("fusion_u", np.concatenate([s, a], axis=-1))
        wg1, bg1 = self.W("fusion.w_g1"), self.W("fusion.b_g1")
        g = O.sigmoid(O.linear(u, wg1[:d], bg1[:d]))
        hid = r("fusion_hid", O.gelu_erf(O.linear(u, wg1[d:], bg1[d:])))
        delta = O.linear(hid, self.W("fusion.w2"), self.W("fusion.b2"))
        return O.layer_norm(h + g * delta, self.W("fusion.ln_out.w"), self.W("fusion.ln_out.b"), eps)

    def lm_head(self, y):
        self._net = "head"
        n = self._r("head_in", O.rms_norm(y, self.W("final_norm"), self.m.norm_eps))
        return O.linear(n, self.W("embed") if self.m.tied_lm_head else self.W("lm_head"))


def with_exact(sites) -> type:
    """A Bf16Oracle subclass that keeps ``sites`` exact."""
    return type("Bf16OracleExact", (Bf16Oracle,), {"exact": frozenset(sites)})


def site_errors(p=PROTOCOL):
    """Logits rel-L2 against the fp64 oracle of one refresh + step on a
    partly unmasked canvas of the protocol's model (batch 2): with every site
    rounded ("all"), and with every site but one rounded ("all_but_<site>").
    The squared difference to "all" is that site's share of the error."""
    m = wl.get_workload(p["workload"]).model
    host = wl.make_weights(m, seed=p["weight_seed"], affine_std=p["affine_std"])
    B = 2
    w = wl.Workload("floor", m, batch=B, prompt_len=p["prompt_len"], gen_len=p["gen_len"],
                    steps_per_block=p["steps"], K=p["K"])
    z = wl.random_canvas(w, B, w.total_len, 0.3, seed=5, start=p["prompt_len"])
    ref = O.Oracle(m, host)
    s = ref.new_session(B)
    lr = ref.denoise_logits(s, z, ref.anchor_forward(s, z))
    out = {}
    for name, ex in [("all", ())] + [("all_but_" + t, (t,)) for t in SITES]:
        o = with_exact(ex)(m, host)
        ss = o.new_session(B)
        lg = o.denoise_logits(ss, z, o.anchor_forward(ss, z))
        out[name] = float(np.linalg.norm(lg - lr) / np.linalg.norm(lr))
    return out


def block_step_case(m, host, batch, prompt_len, block_len, seed, T, exact=()):
    """The block-mode case of the GPU's full-size tests (test_gpu_fullsize:
    prompt prefill, a refresh on an all-MASK block, one stale step on a
    partly unmasked block) for the last sequence of the batch: the logits of
    the exact oracle and of the bf16-operand path, and their rel-L2."""
    w = wl.Workload("fullsize", m, batch=batch, prompt_len=prompt_len, gen_len=4 * block_len,
                    steps_per_block=T, K=4, block_len=block_len, seed=seed)
    prompts = wl.make_prompts(w)
    b = batch - 1
    z0 = np.full((1, block_len), m.mask_id, np.int32)
    z1 = wl.random_canvas(w, batch, block_len, 0.6, seed=seed + 1)[b:b + 1]
    out = {}
    for name, cls in (("oracle", O.Oracle), ("bf16", with_exact(exact))):
        o = cls(m, host)
        sess = o.new_session(1)
        o.prefill(sess, prompts[b:b + 1])
        cache = o.anchor_forward(sess, z0)
        out[name] = o.denoise_logits(sess, z1, cache)[0]
    out["rel_l2"] = float(np.linalg.norm(out["bf16"] - out["oracle"]) / np.linalg.norm(out["oracle"]))
    return out


def run(p=PROTOCOL, log=print, exact=()):
    m = wl.get_workload(p["workload"]).model
    assert m.fusion == "gated_mlp"
    host = wl.make_weights(m, seed=p["weight_seed"], affine_std=p["affine_std"])
    emu, ref = with_exact(exact)(m, host), O.Oracle(m, host)
    B, Tn, K, G = p["batch"], p["steps"], p["K"], p["gen_len"]
    w = wl.Workload("floor", m, batch=B, prompt_len=p["prompt_len"], gen_len=G, steps_per_block=Tn, K=K)
    z = wl.initial_canvas(w, wl.make_prompts(w, batch=B, seed=p["prompt_seed"]))
    s_emu, s_ref = emu.new_session(B), ref.new_session(B)
    n_sel = ok_sel = n_forced = ok_forced = n_masked = ok_masked = 0
    for n in range(Tn):
        if n % K == 0:
            c_emu, c_ref = emu.anchor_forward(s_emu, z), ref.anchor_forward(s_ref, z)
        g = emu.denoise_step(s_emu, z, c_emu, n, Tn, G)       # the bf16 path drives the canvas
        r = ref.denoise_step(s_ref, z, c_ref, n, Tn, G)       # the teacher sees the same canvas
        masked = z == m.mask_id
        committed = masked & (g["z"] != m.mask_id)
        ok = int((g["z"][committed] == r["tok"][committed]).sum())
        if O.unmask_count(n, Tn, G) >= int(masked.sum(axis=1).max()):
            n_forced += int(committed.sum())
            ok_forced += ok
        else:
            n_sel += int(committed.sum())
            ok_sel += ok
        n_masked += int(masked.sum())
        ok_masked += int((g["tok"][masked] == r["tok"][masked]).sum())
        log(f"step {n}: confidence-selected {ok_sel}/{n_sel}, all masked {ok_masked}/{n_masked}")
        z = g["z"]
    return dict(protocol=p, selected_ok=ok_sel, selected=n_sel, forced_ok=ok_forced, forced=n_forced,
                masked_ok=ok_masked, masked=n_masked)


def depth_golden(path=os.path.join(HERE, "golden", "bf16_posttrain_depth62.json")):
    """The bf16-operand path's own logits error at the post-train model's full
    depth (2 + 54 + 6 layers), in the case test_posttrain_full_depth_one_sequence
    runs on the GPU (batch 1, 32-token prompt, block 32, seed 11, T = 32), with
    the QKV input carried exactly as the GPU's split operand carries it.
    Needs about 60 GB of host memory (the bf16 weights plus one widened
    layer); the GPU machine's host runs it."""
    w = wl.WORKLOADS["posttrain"]
    m = w.model
    host = wl.make_weights(m, seed=11)
    res = block_step_case(m, host, 1, 32, 32, seed=11, T=32, exact=("qkv_in",))
    out = {"case": dict(workload="posttrain", batch=1, prompt_len=32, block_len=32, seed=11, T=32,
                        layers=[m.n_shared, m.n_anchor, m.n_denoise], exact=["qkv_in"]),
           "bf16_path_logits_rel_l2": res["rel_l2"],
           "_source": "written by tests/bf16_floor.py --depth: the oracle with bf16 rounding at every "
                      "tensor-core operand (QKV input exact), against the fp64 oracle"}
    with open(path, "w") as f:
        json.dump(out, f, indent=1)
        f.write("\n")
    return out


if __name__ == "__main__" and "--depth" in sys.argv:
    print(json.dumps(depth_golden()))
elif __name__ == "__main__":
    res = run()
    res["_source"] = ("written by tests/bf16_floor.py: the oracle with bf16 rounding at every tensor-core operand, "
                      "teacher-forced against the fp64 oracle")
    # where the flips come from: each site's share of the logits error, and the
    # agreement of the same protocol with the dominant site (the QKV
    # projections' input) kept exact, everywhere and in one network at a time
    res["site_logits_rel_l2"] = site_errors()
    for ex in (("qkv_in",), ("qkv_in@denoise",), ("qkv_in@anchor",)):
        r = run(log=lambda _: None, exact=ex)
        res["exact_" + "_".join(ex).replace("@", "_in_")] = {k: r[k] for k in
                                                             ("selected_ok", "selected", "forced_ok", "forced",
                                                              "masked_ok", "masked")}
    with open(os.path.join(HERE, "golden", "bf16_floor_small.json"), "w") as f:
        json.dump(res, f, indent=1)
        f.write("\n")
    print(json.dumps(res))
