"""End-to-end DN forward of the elastic ViTs through the C-ABI against the
fp64 oracle: every mode of the tiny, ViT-S/16 and ViT-B/16 configurations,
bit-exact packed layouts, mode switching, degenerate tables.

Acceptance (per mode): max|dlogit| <= 1e-2 * max|logit_oracle|, and top-1
agreement >= 99.9 % (2000 tiny images per mode, 256 ViT-S/16 images per mode,
all 256 images of a ViT-B/16 batch in every mode). With
random weights the ViTs give almost every image the same top class, so the
image-dependent part of the logits (centred over the batch) is checked as
well: within 2e-2, and its top class equal to the oracle's wherever the
oracle's margin decides it."""
import numpy as np
import pytest

from helpers import check_image_dependent_part, dev, empty_dev, margin, rel_err, stream_handle, top1_agreement
from oracle_pool import vit_logits
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


@pytest.fixture(scope="module")
def tiny():
    cfg = synth.TINY
    w = synth.make_vit_weights(cfg)
    tables = synth.make_vit_tables(cfg)
    return cfg, w, ov.widen_all(w), tables


def test_tiny_all_modes_2000_images(tiny):
    cfg, w, wide, tables = tiny
    n_img = 2000
    img = synth.make_images(cfg, n_img)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=n_img) as model:
        x = dev(img)
        for m, t in enumerate(tables):
            got = _run(model, x, n_img, cfg.classes, m)
            ref = ov.vit_forward_sliced(wide, cfg, t["heads"], t["mlp"], img)
            err, agree = rel_err(got, ref), top1_agreement(got, ref)
            mg = margin(ref)
            print(f"tiny mode {m}: err {err:.2e} top1 {agree:.4f} margin p1/p50 {np.percentile(mg, 1):.3e}/"
                  f"{np.median(mg):.3e}")
            assert err <= TOL
            assert agree >= 0.999
            check_image_dependent_part(f"tiny mode {m} ({n_img} images)", got, ref, cfg.layers)


def test_tiny_batch_8_matches_oracle(tiny):
    cfg, w, wide, tables = tiny
    img = synth.make_images(cfg, cfg.batch)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=cfg.batch) as model:
        x = dev(img)
        for m, t in enumerate(tables):
            assert rel_err(_run(model, x, cfg.batch, cfg.classes, m),
                           ov.vit_forward_sliced(wide, cfg, t["heads"], t["mlp"], img)) <= TOL


@pytest.mark.parametrize("cfg", [synth.TINY, synth.VIT_S, synth.VIT_B], ids=lambda c: c.name)
def test_packed_layouts_bit_exact(cfg):
    w = synth.make_vit_weights(cfg)
    tables = synth.make_vit_tables(cfg)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=1) as model:
        for m, t in enumerate(tables):
            for l in range(cfg.layers):
                ref = ov.vit_pack_layer(w, cfg, l, t["heads"][l], t["mlp"][l])
                for which, name in enumerate(ov.PACK_ORDER):
                    out = np.empty_like(ref[name])
                    model.export_packed(m, l, which, out)
                    assert out.tobytes() == ref[name].tobytes(), (m, l, name)


def _check_top1(tag, got, ref):
    """Top-1 agreement >= 99.9 %, where a disagreement only counts if the
    oracle's own top-1/top-2 margin exceeds twice the largest logit error
    (below that either class is a valid answer)."""
    agree = got.argmax(axis=1) == ref.argmax(axis=1)
    decided = margin(ref) > 2.0 * float(np.max(np.abs(got - ref)))
    assert np.mean(agree | ~decided) >= 0.999, (tag, np.flatnonzero(decided & ~agree))


def _parity_rows(cfg, tag, got, ref):
    out = check_image_dependent_part(tag, got, ref, cfg.layers)
    assert out["err"] <= TOL, (tag, out["err"])
    _check_top1(tag, got, ref)
    assert np.all(np.isfinite(got))


def _sampled_parity(cfg, batch, sample, modes=None):
    w = synth.make_vit_weights(cfg)
    tables = synth.make_vit_tables(cfg)
    img = synth.make_images(cfg, batch)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=batch) as model:
        x = dev(img)
        for m in (modes if modes is not None else range(len(tables))):
            rows = sample(m) if callable(sample) else sample
            got = _run(model, x, batch, cfg.classes, m)
            ref = vit_logits(cfg, tables, m, img[rows])
            _parity_rows(cfg, f"{cfg.name} B={batch} mode {m} ({len(rows)} images)", got[rows], ref)


def test_vit_s_256_images_all_modes():
    """ViT-S/16 at its batch of 64: four batches, 256 images per mode, every
    one against the oracle."""
    cfg = synth.VIT_S
    w = synth.make_vit_weights(cfg)
    tables = synth.make_vit_tables(cfg)
    n_img, B = 256, cfg.batch
    img = synth.make_images(cfg, n_img)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=B) as model:
        for m in range(len(tables)):
            got = np.concatenate([_run(model, dev(img[i:i + B]), B, cfg.classes, m) for i in range(0, n_img, B)])
            ref = vit_logits(cfg, tables, m, img)
            _parity_rows(cfg, f"{cfg.name} mode {m} ({n_img} images)", got, ref)


def test_vit_b_batch_256_all_modes():
    """ViT-B/16 at batch 256: all 256 images of every mode."""
    _sampled_parity(synth.VIT_B, 256, np.arange(256))


@pytest.mark.parametrize("batch", [1, 32])
def test_vit_b_small_batches(batch):
    _sampled_parity(synth.VIT_B, batch, np.arange(batch), modes=[0, 4])


def test_one_image_on_larger_handles_all_modes(tiny):
    """A one-image forward on handles built for more images takes the
    one-image plans (FC2's reduction split over idle SMs, the partial sums
    added in a second launch): every mode against the oracle, and within the
    same bound of that image's logits inside a larger batch (the split sums
    FC2 in another order, and a last-bit change of the fp32 residual can move
    a later bf16 rounding)."""
    for cfg, w, wide, tables, big in [(*tiny, 8), _vit_s_setup() + (64,)]:
        img = synth.make_images(cfg, big)
        with binding.ElasticModel.vit(cfg, w, tables, max_batch=big) as model:
            x1, xb = dev(img[:1]), dev(img)
            for m, t in enumerate(tables):
                one = _run(model, x1, 1, cfg.classes, m)
                ref = ov.vit_forward_sliced(wide, cfg, t["heads"], t["mlp"], img[:1])
                assert rel_err(one, ref) <= TOL, (cfg.name, m)
                many = _run(model, xb, big, cfg.classes, m)[:1]
                assert rel_err(one, many) <= TOL, (cfg.name, m)
                # repeatable bit for bit (the split sums in a fixed order)
                assert np.array_equal(_run(model, x1, 1, cfg.classes, m), one)
                # eight images: the 8-image plans split the residual GEMMs too
                eight = _run(model, dev(img[:8]), 8, cfg.classes, m)
                ref8 = ov.vit_forward_sliced(wide, cfg, t["heads"], t["mlp"], img[[0, 7]])
                assert rel_err(eight[[0, 7]], ref8) <= TOL, (cfg.name, m)


def _vit_s_setup():
    cfg = synth.VIT_S
    w = synth.make_vit_weights(cfg)
    return cfg, w, ov.widen_all(w), synth.make_vit_tables(cfg)


def test_mode_switch_between_enqueued_forwards(tiny):
    """set_mode only affects forwards enqueued after it; no sync in between."""
    import torch
    cfg, w, wide, tables = tiny
    img = synth.make_images(cfg, cfg.batch)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=cfg.batch) as model:
        x = dev(img)
        outs = [empty_dev((cfg.batch, cfg.classes), torch.float32) for _ in range(4)]
        seq = [1, 0, 1, 1]
        s = stream_handle()
        for o, m in zip(outs, seq):
            model.set_mode(m)
            model.forward(s, x.data_ptr(), cfg.batch, o.data_ptr())
        model.sync_status(s)
        for o, m in zip(outs, seq):
            t = tables[m]
            assert rel_err(o.cpu().numpy().astype(np.float64),
                           ov.vit_forward_sliced(wide, cfg, t["heads"], t["mlp"], img)) <= TOL
        assert model.mode == 1


def test_forward_host_equals_device_forward(tiny):
    cfg, w, wide, tables = tiny
    img = synth.make_images(cfg, 5)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=8) as model:
        dev_out = _run(model, dev(img), 5, cfg.classes, 1)
        host_out = np.zeros((5, cfg.classes), np.float32)
        model.forward_host(img, host_out)
        assert np.array_equal(host_out.astype(np.float64), dev_out)


def test_forward_host_batches_equals_device_forward(tiny):
    """Batches streamed from (pinned) host memory with the copies overlapped:
    every batch's logits equal the device forward of the same images bit for
    bit, in both modes, with batches alternating between the two staging
    buffers."""
    import torch
    cfg, w, wide, tables = tiny
    nb, B = 5, 3
    imgs = [torch.from_numpy(synth.make_images(cfg, B, seed=100 + i)).pin_memory().numpy() for i in range(nb)]
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=4) as model:
        for m in range(len(tables)):
            model.set_mode(m)
            outs = [torch.zeros((B, cfg.classes), dtype=torch.float32).pin_memory().numpy() for _ in range(nb)]
            model.forward_host_batches(imgs, outs)
            for i in range(nb):
                assert np.array_equal(outs[i].astype(np.float64), _run(model, dev(imgs[i]), B, cfg.classes, m)), (m, i)
        with pytest.raises(binding.ElastoError) as e:
            model.forward_host_batches([np.zeros((5,) + imgs[0].shape[1:], imgs[0].dtype)],
                                       [np.zeros((5, cfg.classes), np.float32)])
        assert e.value.status == binding.ERR_INVALID_ARG


def test_degenerate_and_non_nested_tables():
    """Layers keeping no head and/or no MLP channel, a channel count that is
    not a multiple of 8, and tables that are not nested across modes."""
    cfg = synth.vit_small_variant(synth.TINY, dtype=synth.BF16)
    w = synth.make_vit_weights(cfg)
    wide = ov.widen_all(w)
    t0 = synth.make_vit_tables(cfg)[0]
    rng = np.random.default_rng(3)
    odd = {"heads": [np.sort(rng.choice(3, k, replace=False)).astype(np.int32) for k in (0, 1, 3, 2, 0, 1)],
           "mlp": [np.sort(rng.choice(768, k, replace=False)).astype(np.int32) for k in (100, 0, 768, 1, 0, 37)]}
    tables = [t0, odd] + synth.make_vit_tables(cfg, nested=False)[1:]
    img = synth.make_images(cfg, 6)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=6) as model:
        assert model.query(binding.Q_PREFIX_SHARED) == 0  # not nested: one packed copy per mode
        x = dev(img)
        for m, t in enumerate(tables):
            got = _run(model, x, 6, cfg.classes, m)
            ref = ov.vit_forward_sliced(wide, cfg, t["heads"], t["mlp"], img)
            assert rel_err(got, ref) <= TOL, m


@pytest.mark.parametrize("cfg", [synth.TINY, synth.VIT_S, synth.VIT_B], ids=lambda c: c.name)
def test_nested_modes_share_one_packed_copy(cfg):
    """Nested kept sets (Eq. 8): one prefix-ordered copy per layer serves every
    mode, so the packed weights take the largest mode's memory, not the sum
    over modes; mode 0 and the smallest mode still match the oracle."""
    w = synth.make_vit_weights(cfg)
    wide = ov.widen_all(w)
    tables = synth.make_vit_tables(cfg)
    img = synth.make_images(cfg, 4)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=4) as model:
        assert model.query(binding.Q_PREFIX_SHARED) == 1
        total = model.query(binding.Q_PACKED_TOTAL)
        views = [model.query(binding.Q_PACKED_BYTES, m) for m in range(len(tables))]
        assert views[0] == max(views)
        assert total <= views[0] + 2048 * 10 * cfg.layers  # alignment and guard zones only (<= 2 KiB a buffer)
        assert total < sum(views)
        x = dev(img)
        for m in (0, len(tables) - 1):
            t = tables[m]
            ref = ov.vit_forward_sliced(wide, cfg, t["heads"], t["mlp"], img)
            assert rel_err(_run(model, x, 4, cfg.classes, m), ref) <= TOL, m


def test_batch_limits_and_bad_mode(tiny):
    cfg, w, wide, tables = tiny
    import torch
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=4) as model:
        x = dev(synth.make_images(cfg, 5))
        y = empty_dev((5, cfg.classes), torch.float32)
        with pytest.raises(binding.ElastoError) as e:
            model.forward(stream_handle(), x.data_ptr(), 5, y.data_ptr())
        assert e.value.status == binding.ERR_INVALID_ARG
        with pytest.raises(binding.ElastoError) as e:
            model.set_mode(2)
        assert e.value.status == binding.ERR_BAD_MODE
        assert model.mode == 0
        assert model.query(binding.Q_N_MODES) == 2
        assert model.query(binding.Q_PACKED_BYTES, 1) < model.query(binding.Q_PACKED_BYTES, 0)


def test_profile_dns_and_select(tiny):
    """elasto_profile_dns measures each mode on this GPU; Eq. 10 over the
    measured table picks the cheapest mode meeting the budgets."""
    cfg, w, wide, tables = tiny
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=8) as model:
        model.set_mode(1)
        lut = model.profile_dns(stream_handle(), batch=8, trials=10)
        assert model.mode == 1  # restored
        assert len(lut) == 2 and all(e["latency_ms"] > 0 for e in lut)
        assert all(np.isnan(e["accuracy"]) for e in lut)
        assert lut[1]["gflops"] < lut[0]["gflops"] and lut[1]["memory_bytes"] < lut[0]["memory_bytes"]
        assert np.isclose(lut[0]["gflops"], 2 * model.query(binding.Q_MODE_MACS, 0) * 8 / 1e9)
        nan = float("nan")
        assert binding.elasto_select_dn(lut, nan, nan, nan) == 1
        lut[0]["accuracy"], lut[1]["accuracy"] = 80.0, 60.0   # the caller's validation accuracies
        assert binding.elasto_select_dn(lut, nan, nan, 70.0) == 0
        assert binding.elasto_select_dn(lut, nan, lut[1]["memory_bytes"], 70.0) is None
