"""GPU parity of the consumer (Sec. 3.2): text queries attend causally to the visual K/V the
build wrote into the cache, plus text K/V around them, through the C ABI's dv_text_attention.

The sequence of every batch element is: n_sys text slots (a system prompt), the N_v visual
slots written by dv_build_visual_memory (slot0 = n_sys), then N_t text slots whose tokens are
the queries (query t sits at slot n_sys + N_v + t). The oracle computes the same attention in
fp64 from its own visual K/V (oracle.build_tokens) and the same synthetic text K/V and queries,
so nothing it uses comes from the GPU.

Tolerances. With K/V written directly as bf16 (no build), the oracle sees exactly the kernel's
inputs; the kernel's own error is the bf16 rounding of the probabilities P (relative <= 2^-8,
averaging over the keys) and of the output (<= 2^-8): the build's bar applies, max scaled error
<= 2e-2 and cosine >= 0.9999 per query row. End to end, the visual K/V also carry the build's
own error (<= 2e-2 per element, ~1.5e-3 rms), which moves scores and the weighted values: the
bar is 4e-2 per element with the same cosine.
"""
import numpy as np
import pytest

import oracle
import synth
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu
E2E_REL_TOL = 4e-2


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34972_gb300.build import build_library
    build_library()


def _run_case(cfg, n_sys, n_text, n_q_heads, layer, capacity=None, batch_cache=None,
              q_slot_edit=None, label="", rel_tol=E2E_REL_TOL):
    import torch
    import paper_2609_34972_gb300 as dv
    B, Nv, H, D = cfg.batch, cfg.n_vis, cfg.n_kv_heads, cfg.head_dim
    S_used = n_sys + Nv + n_text
    S = capacity or S_used
    inp = synth.make_inputs(cfg)
    # text keys/values (already rotated, as a backbone would store them) and queries
    tk = synth.normal_bf16(cfg.seed + 100, 20, (B, n_sys + n_text, H, D), 0.0, 1.0)
    tv = synth.normal_bf16(cfg.seed + 100, 21, (B, n_sys + n_text, H, D), 0.0, 1.0)
    qb = synth.normal_bf16(cfg.seed + 100, 22, (B, n_q_heads, n_text, D), 0.0, 1.0)
    q_slot = np.broadcast_to(n_sys + Nv + np.arange(n_text, dtype=np.int32), (B, n_text)).copy()
    if q_slot_edit is not None:
        q_slot_edit(q_slot)
    n_keys = np.full(B, S_used, dtype=np.int32)
    scale = 1.0 / np.sqrt(D)

    # GPU: text K/V into their slots (plumbing), the build writes the visual slots
    k, v, plan = gu.run_build(inp, seq_len=S, batch_cache=batch_cache, slot0=n_sys)
    Bc = k.shape[1]
    for l in range(cfg.n_layers):
        k[l, :B, :n_sys] = gu.torch_bf16(tk[:, :n_sys], "cuda")
        v[l, :B, :n_sys] = gu.torch_bf16(tv[:, :n_sys], "cuda")
        k[l, :B, n_sys + Nv:S_used] = gu.torch_bf16(tk[:, n_sys:], "cuda")
        v[l, :B, n_sys + Nv:S_used] = gu.torch_bf16(tv[:, n_sys:], "cuda")
    q = gu.torch_bf16(qb, "cuda")
    nk = torch.from_numpy(n_keys).cuda()
    qs = torch.from_numpy(q_slot).cuda()
    kb = k[:, :B] if Bc > B else k
    vb = v[:, :B] if Bc > B else v
    out = dv.text_attention(q, kb, vb, layer, nk, qs, scale)
    torch.cuda.synchronize()
    assert dv.text_attention_status() == dv.DV_OK

    # oracle: its own visual K/V of this layer + the same text K/V and queries, in fp64
    ref = oracle.build_tokens(inp, np.arange(cfg.tokens), layers=[layer])
    kvis = ref["k"][:, 0].reshape(B, Nv, H, D)
    vvis = ref["v"][:, 0].reshape(B, Nv, H, D)
    tkf = synth.bf16_to_f32(tk).astype(np.float64)
    tvf = synth.bf16_to_f32(tv).astype(np.float64)
    kf = np.concatenate([tkf[:, :n_sys], kvis, tkf[:, n_sys:]], axis=1)
    vf = np.concatenate([tvf[:, :n_sys], vvis, tvf[:, n_sys:]], axis=1)
    qf = synth.bf16_to_f32(qb).astype(np.float64)
    want = oracle.text_attention(qf, kf, vf, n_keys, q_slot, scale)

    got = out.double().cpu().numpy()
    g = got.reshape(-1, 1, D)
    o = want.reshape(-1, 1, D)
    live = np.abs(o).sum(axis=-1)[:, 0] > 0
    assert np.all(g[~live] == 0.0), "a query that sees no key must get zeros"
    gu.assert_parity(g[live], g[live], o[live], o[live], D, "attention " + label, rel_tol=rel_tol)
    return out


def test_attention_tiny_mha_head64():
    cfg = synth.config("tiny", n_vis=64, batch=2)
    _run_case(cfg, n_sys=5, n_text=20, n_q_heads=8, layer=2, label="tiny head 64")


def test_attention_gqa_head128_multi_block_split():
    # 15 + 300 + 37 = 352 keys: three 128-key blocks (ragged), split over the cluster; grouped
    # queries (4 per kv head) make 148 query rows per kv head: two 128-row blocks.
    cfg = gu.small_config("attn_gqa", d=1024, n_layers=2, n_kv_heads=2, n_heads=8, head_dim=128,
                          rank=64, n_vis=300, batch=2, x0_sigma=0.5, seed=81, pos_start=15)
    _run_case(cfg, n_sys=15, n_text=37, n_q_heads=8, layer=1, capacity=400,
              label="gqa head 128")


def test_attention_queries_without_keys_and_early_slots():
    # Query 0 sits at slot -1 (sees nothing: zeros); query 1 at slot 3 (inside the system
    # prompt: sees 4 text keys); query 2 at slot 40 (part of the visual keys).
    cfg = synth.config("tiny", n_vis=64, batch=1)

    def edit(q_slot):
        q_slot[0, 0], q_slot[0, 1], q_slot[0, 2] = -1, 3, 40

    _run_case(cfg, n_sys=5, n_text=8, n_q_heads=8, layer=0, q_slot_edit=edit, label="early slots")


def test_attention_strided_cache_with_spare_batch_rows():
    # The cache holds more batch rows and slots than the sequence uses.
    cfg = synth.config("tiny", n_vis=100, batch=2)
    _run_case(cfg, n_sys=7, n_text=30, n_q_heads=16, layer=3, capacity=300, batch_cache=3,
              label="strided cache")


def test_attention_llava15_full_layer():
    # LLaVA-1.5-7B-shaped layer: 35 system slots, 576 visual, 64 text queries, 32 heads of 128.
    cfg = synth.CONFIGS["llava15_7b"]
    _run_case(cfg, n_sys=35, n_text=64, n_q_heads=32, layer=5, label="llava15 layer")


def _exact_case(hd, B, hq, hkv, nt, n_keys, S, seed, label, k_gain=None):
    # Every slot holds synthetic bf16 K/V (no build): the oracle reads the same values.
    # k_gain (per slot) scales the keys before their bf16 rounding.
    import torch
    import paper_2609_34972_gb300 as dv
    L = 2
    kb = synth.normal_bf16(seed, 30, (L, B, S, hkv, hd), 0.0, 1.0)
    if k_gain is not None:
        kb = synth.f64_to_bf16(synth.bf16_to_f32(kb).astype(np.float64) *
                               np.asarray(k_gain, dtype=np.float64)[None, None, :, None, None])
    vb = synth.normal_bf16(seed, 31, (L, B, S, hkv, hd), 0.0, 1.0)
    qb = synth.normal_bf16(seed, 32, (B, hq, nt, hd), 0.0, 1.0)
    n_keys = np.asarray(n_keys, dtype=np.int32)
    # even batch rows: the last nt slots; odd rows: strided slots (some past n_keys)
    q_slot = np.stack([n_keys[b] - nt + np.arange(nt) if b % 2 == 0 else 300 + 7 * np.arange(nt)
                       for b in range(B)]).astype(np.int32)
    scale = 1.0 / np.sqrt(hd)
    k = gu.torch_bf16(kb, "cuda")
    v = gu.torch_bf16(vb, "cuda")
    out = dv.text_attention(gu.torch_bf16(qb, "cuda"), k, v, 1, torch.from_numpy(n_keys).cuda(),
                            torch.from_numpy(q_slot).cuda(), scale)
    torch.cuda.synchronize()
    assert dv.text_attention_status() == dv.DV_OK
    f = lambda a: synth.bf16_to_f32(a).astype(np.float64)
    want = oracle.text_attention(f(qb), f(kb[1]), f(vb[1]), n_keys, q_slot, scale)
    g = out.double().cpu().numpy().reshape(-1, 1, hd)
    o = want.reshape(-1, 1, hd)
    gu.assert_parity(g, g, o, o, hd, label)


@pytest.mark.parametrize("hd,hq,hkv,nt", [(128, 32, 32, 64), (128, 28, 4, 50), (64, 8, 2, 33)])
def test_attention_kernel_on_exact_inputs(hd, hq, hkv, nt):
    _exact_case(hd, 2, hq, hkv, nt, [700, 650], 768, 90 + hd, f"attention kernel hd{hd} hq{hq}/{hkv}")


# Launch shapes that reach every kernel variant and cluster size the launcher picks (clusters =
# batch x kv heads x 128-row query blocks; cluster size S = the largest of 2, 4, 8 within the key
# blocks with one CTA per SM (two stages); where that is 1, one stage with two CTAs per SM in
# clusters of 2 if those fit, on 152 SMs):
#   two stages, S = 8: 2 clusters, 9 key blocks; two stages, S = 4: 24 clusters; two stages,
#   S = 2: 64 clusters (64 of 128 query rows valid) and 48 clusters (tiles of 128, 128 and 94
#   query rows); one stage, S = 2: 80 clusters of 16 query rows and 120 clusters (tiles of 128
#   and 72 rows), 3 key blocks.
@pytest.mark.parametrize("hd,B,hq,hkv,nt,n_keys,S", [
    (128, 1, 8, 2, 30, [1100], 1152),
    (64, 1, 8, 2, 30, [1100], 1152),
    (128, 2, 12, 12, 20, [1000, 977], 1024),
    (64, 2, 12, 12, 20, [1000, 977], 1024),
    (128, 4, 20, 20, 16, [300, 290, 300, 257], 320),
    (64, 4, 20, 20, 16, [300, 290, 300, 257], 320),
    (64, 2, 32, 32, 64, [700, 650], 768),
    (128, 4, 28, 4, 50, [700, 650, 700, 690], 768),
    (128, 3, 40, 20, 100, [300, 290, 277], 320),
    # many query blocks per kv head: 28 / 4 GQA, 200 text queries = 1400 rows (11 blocks of
    # 128, the last ragged), 88 clusters: one stage, S = 2
    (128, 2, 28, 4, 200, [700, 650], 768),
])
def test_attention_every_cluster_shape(hd, B, hq, hkv, nt, n_keys, S):
    _exact_case(hd, B, hq, hkv, nt, n_keys, S, 500 + hd + B + hq,
                f"attention hd{hd} B{B} hq{hq}/{hkv} nt{nt}")


@pytest.mark.parametrize("hd,B,hq,hkv,nt,n_keys,S,gain", [
    # two stages, 8-CTA clusters, 2 key blocks per CTA; keys growing with the slot
    (128, 1, 8, 2, 30, [2000], 2048, "rise"),
    # one stage, 2-CTA clusters, 8 key blocks per CTA; two stages, 4-CTA clusters, 8 blocks
    (128, 4, 20, 20, 16, [2000, 1900, 2000, 1950], 2048, "rise"),
    (64, 2, 12, 12, 20, [4000, 3900], 4096, "fall"),
])
def test_attention_running_maximum_grows_across_blocks(hd, B, hq, hkv, nt, n_keys, S, gain):
    # Key magnitudes that change along the slots make each row's running maximum jump by more
    # than 2^8 between key blocks (so O in TMEM is rescaled) or stay put (no rescale), with
    # softmax weights far from uniform.
    slots = np.arange(S, dtype=np.float64)
    g = 1.0 + slots / 96.0 if gain == "rise" else 1.0 + (S - slots) / 96.0
    _exact_case(hd, B, hq, hkv, nt, n_keys, S, 700 + hd + B, f"attention max growth hd{hd} {gain}",
                k_gain=g)
