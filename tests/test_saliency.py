"""Compress-stage L1 saliency (Section 4.1): the oracle pinned by planted
weights and closed forms (CPU), elasto_topk against the oracle's top-k (CPU,
host-only C call), and elasto_saliency on the GPU against the oracle, with a
model built from the tables it induces."""
import dataclasses

import numpy as np
import pytest

from oracle import resnet as orr
from oracle import vit as ov
from oracle.saliency import resnet_saliency, top_k, vit_embed_saliency, vit_saliency
from paper_2609_10018_gb300 import binding, synth

TINY_BF16 = synth.vit_small_variant(synth.TINY, dtype=synth.BF16)


def test_oracle_finds_planted_head_and_channel():
    cfg = synth.TINY
    w = ov.widen_all(synth.make_vit_weights(cfg))
    d = cfg.dim
    w["l1.qkv_w"][d + 2 * 64: d + 3 * 64] *= 10.0     # head 2's key rows
    w["l3.fc2_w"][:, 77] *= 50.0                      # channel 77's W2 column
    hs, fs = vit_saliency(w, cfg)
    assert int(np.argmax(hs[1])) == 2
    assert int(np.argmax(fs[3])) == 77
    # closed form: a head's score is the mean of the row averages it owns
    j, l = 1, 4
    qkv, proj = np.abs(w[f"l{l}.qkv_w"]), np.abs(w[f"l{l}.proj_w"])
    rows = [qkv[b * d + j * 64 + r].mean() for b in range(3) for r in range(64)] + \
           [proj[:, j * 64 + r].mean() for r in range(64)]
    assert abs(hs[l, j] - np.mean(rows)) < 1e-15


def test_oracle_embedding_saliency_planted_and_closed_form():
    cfg = synth.TINY
    w = ov.widen_all(synth.make_vit_weights(cfg))
    w["l2.fc2_w"][41] *= 30.0                         # channel 41: its W2 row (an output of the block)
    w["l4.qkv_w"][:, 99] *= 30.0                      # channel 99: its W_qkv column (an input)
    e = vit_embed_saliency(w, cfg)
    assert set(top_k(e, 2).tolist()) == {41, 99}
    # closed form for one channel: mean of its 2 + 4L row / column averages
    c, d = 7, cfg.dim
    parts = [np.abs(w["patch_w"][c]).mean(), np.abs(w["head_w"][:, c]).mean()]
    for l in range(cfg.layers):
        parts += [np.abs(w[f"l{l}.qkv_w"][:, c]).mean(), np.abs(w[f"l{l}.proj_w"][c]).mean(),
                  np.abs(w[f"l{l}.fc1_w"][:, c]).mean(), np.abs(w[f"l{l}.fc2_w"][c]).mean()]
    assert len(parts) == 2 + 4 * cfg.layers
    assert abs(e[c] - np.mean(parts)) < 1e-15
    assert e.shape == (d,)


def test_oracle_top_k_rules():
    s = np.array([3.0, 1.0, 3.0, 5.0, 0.5])
    assert top_k(s, 2).tolist() == [0, 3]          # 5.0, then the first of the tied 3.0s
    assert top_k(s, 3).tolist() == [0, 2, 3]
    assert top_k(s, 0).tolist() == []
    # one ranking gives nested tables (Eq. 8)
    r = np.random.default_rng(0).random(50)
    for k in range(1, 50):
        assert set(top_k(r, k)) <= set(top_k(r, k + 1))


def test_resnet_oracle_planted_channels():
    cfg = dataclasses.replace(synth.RESNET50, img=32, classes=10)
    w = ov.widen_all(synth.make_resnet_weights(cfg))
    w["b4.conv1_w"][9] *= 20.0                      # S_a channel 9 of block 4 (conv1 output row)
    w["b7.conv3_w"][:, 3] *= 20.0                   # S_b channel 3 of block 7 (conv3 input column)
    sa, sb = resnet_saliency(w, orr.block_list(cfg))
    assert int(np.argmax(sa[4])) == 9
    assert int(np.argmax(sb[7])) == 3


def test_topk_c_abi_matches_oracle():
    rng = np.random.default_rng(2)
    for _ in range(200):
        n = int(rng.integers(1, 40))
        s = rng.integers(0, 6, n).astype(np.float32)  # many ties
        k = int(rng.integers(0, n + 1))
        assert binding.elasto_topk(s, k).tolist() == top_k(s, k).tolist()


@pytest.mark.gpu
@pytest.mark.parametrize("cfg", [synth.TINY, TINY_BF16, synth.VIT_S], ids=lambda c: f"{c.name}-{c.dtype}")
def test_gpu_vit_saliency_matches_oracle(cfg):
    w = synth.make_vit_weights(cfg)
    a, b = binding.elasto_saliency(binding.vit_desc(cfg, 1), [w[k] for k in synth.vit_weight_names(cfg)],
                                   cfg.layers * cfg.heads, cfg.layers * cfg.mlp)
    hs, fs = vit_saliency(ov.widen_all(w), cfg)
    assert np.allclose(a.reshape(hs.shape), hs, rtol=2e-5, atol=0)
    assert np.allclose(b.reshape(fs.shape), fs, rtol=2e-5, atol=0)
    tables = binding.saliency_tables_vit(cfg, w)
    for m, (kh, kf) in enumerate(zip(cfg.mode_heads, cfg.mode_mlp)):
        for l in range(cfg.layers):
            # compare as sets of the oracle's top-k unless two scores straddle the cut within float error
            assert tables[m]["heads"][l].tolist() == top_k(hs[l], kh).tolist()
            got, ref = set(tables[m]["mlp"][l].tolist()), set(top_k(fs[l], kf).tolist())
            if got != ref:
                cut = np.sort(fs[l])[::-1][kf - 1: kf + 1]
                assert abs(cut[0] - cut[1]) <= 1e-5 * abs(cut[0])


@pytest.mark.gpu
@pytest.mark.parametrize("cfg", [synth.TINY, synth.VIT_S], ids=lambda c: c.name)
def test_gpu_embedding_saliency_matches_oracle(cfg):
    w = synth.make_vit_weights(cfg)
    e = binding.elasto_saliency_embed(binding.vit_desc(cfg, 1), [w[k] for k in synth.vit_weight_names(cfg)])
    ref = vit_embed_saliency(ov.widen_all(w), cfg)
    assert np.allclose(e, ref, rtol=2e-5, atol=0)


@pytest.mark.gpu
def test_gpu_model_from_embedding_saliency_tables():
    """Heads, MLP channels and embedding channels all chosen by the GPU
    saliency; every mode matches the oracle."""
    from helpers import dev, empty_dev, rel_err, stream_handle
    import torch
    cfg = synth.TINY
    w = synth.make_vit_weights(cfg)
    tables = binding.saliency_tables_vit(cfg, w, embed_widths=[None, 120])
    assert len(tables[1]["embed"]) == 120
    wide = ov.widen_all(w)
    img = synth.make_images(cfg, 16)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=16) as model:
        x = dev(img)
        out = empty_dev((16, cfg.classes), torch.float32)
        for m, t in enumerate(tables):
            model.set_mode(m)
            model.forward(stream_handle(), x.data_ptr(), 16, out.data_ptr())
            model.sync_status(stream_handle())
            ref = ov.vit_forward_sliced(wide, cfg, t["heads"], t["mlp"], img, embed_kept=t.get("embed"))
            assert rel_err(out.cpu().numpy().astype(np.float64), ref) <= 1e-2


@pytest.mark.gpu
def test_gpu_model_from_saliency_tables():
    """Tables from the GPU saliency are nested, so the modes share one packed
    copy; every mode matches the oracle."""
    from helpers import dev, empty_dev, rel_err, stream_handle
    import torch
    cfg = synth.TINY
    w = synth.make_vit_weights(cfg)
    tables = binding.saliency_tables_vit(cfg, w)
    wide = ov.widen_all(w)
    img = synth.make_images(cfg, 8)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=8) as model:
        assert model.query(binding.Q_PREFIX_SHARED) == 1
        x = dev(img)
        out = empty_dev((8, cfg.classes), torch.float32)
        for m, t in enumerate(tables):
            model.set_mode(m)
            model.forward(stream_handle(), x.data_ptr(), 8, out.data_ptr())
            model.sync_status(stream_handle())
            ref = ov.vit_forward_sliced(wide, cfg, t["heads"], t["mlp"], img)
            assert rel_err(out.cpu().numpy().astype(np.float64), ref) <= 1e-2


@pytest.mark.gpu
def test_gpu_resnet_saliency_matches_oracle():
    cfg = dataclasses.replace(synth.RESNET50, img=32, classes=10)
    w = synth.make_resnet_weights(cfg)
    blocks = orr.block_list(cfg)
    n = sum(wd for (_, wd, _, _) in blocks)
    a, b = binding.elasto_saliency(binding.resnet_desc(cfg, 1), [w[k] for k in synth.resnet_weight_names(cfg)], n, n)
    sa, sb = resnet_saliency(ov.widen_all(w), blocks)
    assert np.allclose(a, np.concatenate(sa), rtol=2e-5, atol=0)
    assert np.allclose(b, np.concatenate(sb), rtol=2e-5, atol=0)
