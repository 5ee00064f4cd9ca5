"""Embedding-width pruning (Section 4.1: the compress stage also shrinks the
hidden size of the LayerNorm and patch-embedding layers) through the C-ABI
against the fp64 oracle: DNs that keep a subset of the d residual-stream
channels (widths that are and are not multiples of 64), mixed with unpruned
modes in one model, fp32-stored and bf16-stored weights, the no-allocation
entry point, exact packed layouts and the cost queries.

Acceptance as for every DN: max|dlogit| <= 1e-2 * max|logit_oracle|."""
import numpy as np
import pytest

from helpers import dev, empty_dev, rel_err, stream_handle, top1_agreement
from oracle import vit as ov
from paper_2609_10018_gb300 import binding, synth

pytestmark = pytest.mark.gpu

TOL = 1e-2


def _run(model, images_dev, batch, classes, mode):
    import torch
    logits = empty_dev((batch, classes), torch.float32)
    model.set_mode(mode)
    model.forward(stream_handle(), images_dev.data_ptr(), batch, logits.data_ptr())
    model.sync_status(stream_handle())
    return logits.cpu().numpy().astype(np.float64)


def _ref(wide, cfg, t, img):
    return ov.vit_forward_sliced(wide, cfg, t["heads"], t["mlp"], img, embed_kept=t.get("embed"))


def _tiny_tables():
    cfg = synth.TINY
    base = synth.make_vit_tables(cfg)
    tables = [base[0], base[0], base[1], base[1], base[1]]
    return cfg, synth.with_embedding(cfg, tables, [None, 128, 150, 100, 37])


def test_tiny_embedding_pruned_modes_fp32_weights():
    cfg, tables = _tiny_tables()
    w = synth.make_vit_weights(cfg)
    wide = ov.widen_all(w)
    img = synth.make_images(cfg, 256, seed=4)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=256) as model:
        assert model.query(binding.Q_PREFIX_SHARED) == 0
        x = dev(img)
        for m, t in enumerate(tables):
            got, ref = _run(model, x, 256, cfg.classes, m), _ref(wide, cfg, t, img)
            err, agree = rel_err(got, ref), top1_agreement(got, ref)
            print(f"tiny mode {m} (d = {cfg.dim if t['embed'] is None else len(t['embed'])}): err {err:.2e} "
                  f"top-1 {agree:.4f}")
            assert err <= TOL
            assert agree >= 0.99
        # switching back and forth reproduces each mode bit for bit
        first = [_run(model, x[:8], 8, cfg.classes, m) for m in range(len(tables))]
        for m in (4, 0, 3, 1, 2, 4):
            assert np.array_equal(_run(model, x[:8], 8, cfg.classes, m), first[m])


def test_vit_s_embedding_pruned_modes_bf16_weights():
    cfg = synth.VIT_S
    w = synth.make_vit_weights(cfg)
    wide = ov.widen_all(w)
    tables = synth.with_embedding(cfg, synth.make_vit_tables(cfg), [None, 320, 200, 96])
    img = synth.make_images(cfg, 16, seed=6)
    sample = np.arange(0, 16, 3)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=16) as model:
        x = dev(img)
        macs = [model.query(binding.Q_MODE_MACS, m) for m in range(len(tables))]
        assert macs[0] > macs[1] > macs[2] > macs[3]
        for m, t in enumerate(tables):
            got, ref = _run(model, x, 16, cfg.classes, m), _ref(wide, cfg, t, img[sample])
            err = rel_err(got[sample], ref)
            print(f"vit_s mode {m}: err {err:.2e}")
            assert err <= TOL
            assert np.all(np.isfinite(got))


def test_vit_b_embedding_pruned_mode_sampled():
    cfg = synth.VIT_B
    w = synth.make_vit_weights(cfg)
    wide = ov.widen_all(w)
    base = synth.make_vit_tables(cfg)
    tables = synth.with_embedding(cfg, [base[0], base[2]], [None, 448])
    img = synth.make_images(cfg, 64, seed=8)
    sample = np.array([0, 31, 63])
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=64) as model:
        x = dev(img)
        got = _run(model, x, 64, cfg.classes, 1)
        err = rel_err(got[sample], _ref(wide, cfg, tables[1], img[sample]))
        print(f"vit_b d = 448 mode: err {err:.2e}")
        assert err <= TOL


def test_one_image_embedding_pruned_modes():
    """One image on a larger handle (split-K out-projection and FC2 whose
    partial-sum launches also compute the LayerNorms over the kept channels)
    for pruned widths that are and are not multiples of 64."""
    cfg = synth.VIT_S
    w = synth.make_vit_weights(cfg)
    wide = ov.widen_all(w)
    tables = synth.with_embedding(cfg, synth.make_vit_tables(cfg), [None, 320, 200, 96])
    img = synth.make_images(cfg, 2, seed=8)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=16) as model:
        for i in range(2):
            x = dev(img[i:i + 1])
            for m, t in enumerate(tables):
                err = rel_err(_run(model, x, 1, cfg.classes, m), _ref(wide, cfg, t, img[i:i + 1]))
                print(f"vit_s one image {i} mode {m}: err {err:.2e}")
                assert err <= TOL


def test_embedding_pruned_packed_layouts_exact():
    """Packed buffers of a pruned mode are the stored weights' kept rows and
    columns, bit for bit (bf16-stored ViT-S)."""
    cfg = synth.VIT_S
    w = synth.make_vit_weights(cfg)
    tables = synth.with_embedding(cfg, synth.make_vit_tables(cfg), [None, 200, None, 96])
    D = cfg.dim
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=1) as model:
        for m in (1, 3):
            t = tables[m]
            E = t["embed"]
            for l in (0, cfg.layers - 1):
                p = f"l{l}."
                heads, F = t["heads"][l], t["mlp"][l]
                rows = np.concatenate([blk * D + j * 64 + np.arange(64) for blk in range(3) for j in heads])
                cols = np.concatenate([j * 64 + np.arange(64) for j in heads])
                want = {0: w[p + "qkv_w"][rows][:, E], 2: w[p + "proj_w"][E][:, cols],
                        3: w[p + "fc1_w"][F][:, E], 5: w[p + "fc2_w"][E][:, F]}
                for which, ref in want.items():
                    ref = np.ascontiguousarray(ref)
                    out = model.export_packed(m, l, which, np.empty(ref.shape, np.uint16))
                    assert out.tobytes() == ref.tobytes(), (m, l, which)


def test_noalloc_embedding_pruned_modes():
    import torch
    cfg, tables = _tiny_tables()
    w = synth.make_vit_weights(cfg)
    img = synth.make_images(cfg, 32, seed=11)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=32) as model:
        x = dev(img)
        s = stream_handle()
        for m in range(len(tables)):
            want = _run(model, x, 32, cfg.classes, m)
            o = torch.empty((32, cfg.classes), dtype=torch.float32, device="cuda")
            binding.elasto_forward_noalloc(model.handle, s, x.data_ptr(), 32, o.data_ptr())
            model.sync_status(s)
            # the two entry points round the patch-embedding sums in different
            # orders (fp32), which the bf16 activations carry to ~1e-3
            assert rel_err(o.cpu().numpy().astype(np.float64), want) <= TOL, m
