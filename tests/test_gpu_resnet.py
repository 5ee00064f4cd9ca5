"""End-to-end ResNet-50 DN forward (Eq. 7) through the C-ABI against the fp64
oracle: every mode of the 224x224 configuration, 2000 images per mode of a
32x32, 10-class variant of the same network (CIFAR-10 shaped input), packed
weights against the oracle's BN folding, ragged batches, kept counts that are
not multiples of 8, mode switching and the launch records.

Acceptance (per mode): max|dlogit| <= 1e-2 * max|logit_oracle| and top-1
agreement >= 99.9 % over 2000 images."""
import dataclasses

import numpy as np
import pytest

from helpers import dev, empty_dev, margin, rel_err, stream_handle, top1_agreement
from oracle import resnet as orr
from oracle.vit import widen_all
from oracle_pool import resnet_logits
from paper_2609_10018_gb300 import binding, synth

pytestmark = pytest.mark.gpu

TOL = 1e-2
CENTERED_TOL = 2e-2  # on the image-dependent part alone (a far smaller quantity)
SMALL = dataclasses.replace(synth.RESNET50, name="resnet50_32px", img=32, classes=10)


def _run(model, images_dev, batch, classes, mode):
    import torch
    logits = empty_dev((batch, classes), torch.float32)
    model.set_mode(mode)
    model.forward(stream_handle(), images_dev.data_ptr(), batch, logits.data_ptr())
    model.sync_status(stream_handle())
    return logits.cpu().numpy().astype(np.float64)


def _centered(x):
    return x - x.mean(axis=0, keepdims=True)


def _report(tag, got, ref):
    """Besides the logit metric: the part of the logits that varies from image
    to image (logits minus their mean over the batch). With random weights
    most of a ResNet logit is the same for every image, so this is what shows
    that the images themselves went through the network correctly."""
    err, agree, mg = rel_err(got, ref), top1_agreement(got, ref), margin(ref)
    cerr = rel_err(_centered(got), _centered(ref))
    spread = float(np.max(np.abs(_centered(ref))) / np.max(np.abs(ref)))
    print(f"{tag}: err {err:.2e} top1 {agree:.4f} margin p1/p50 {np.percentile(mg, 1):.3e}/{np.median(mg):.3e} "
          f"image-dependent part: {spread:.2e} of max|logit|, its err {cerr:.2e}")
    assert cerr <= CENTERED_TOL
    return err, agree


def test_resnet50_small_all_modes_2000_images():
    cfg = SMALL
    w, tables = synth.make_resnet_weights(cfg), synth.make_resnet_tables(cfg)
    n_img, chunk = 2000, 500
    img = synth.make_images(cfg, n_img)
    with binding.ElasticModel.resnet(cfg, w, tables, max_batch=chunk) as model:
        for m in range(cfg.n_modes):
            got = np.concatenate([_run(model, dev(img[i:i + chunk]), chunk, cfg.classes, m)
                                  for i in range(0, n_img, chunk)])
            ref = resnet_logits(cfg, tables, m, img)
            err, agree = _report(f"resnet50 32px mode {m}", got, ref)
            assert err <= TOL
            assert agree >= 0.999


def test_resnet50_224_all_modes():
    """224x224 (ImageNet-shaped), 128 images per mode (the bench's batch)."""
    cfg = synth.RESNET50
    w, tables = synth.make_resnet_weights(cfg), synth.make_resnet_tables(cfg)
    n_img = 128
    img = synth.make_images(cfg, n_img)
    with binding.ElasticModel.resnet(cfg, w, tables, max_batch=n_img) as model:
        x = dev(img)
        for m in range(cfg.n_modes):
            got = _run(model, x, n_img, cfg.classes, m)
            ref = resnet_logits(cfg, tables, m, img, chunk=2)
            err, agree = _report(f"resnet50 224px mode {m}", got, ref)
            assert err <= TOL
            decided = margin(ref) > 2.0 * float(np.max(np.abs(got - ref)))
            assert np.all((got.argmax(axis=1) == ref.argmax(axis=1)) | ~decided)


def test_resnet_packed_weights_match_oracle_folding():
    """Export of the packed (gathered, BN-folded) buffers against the oracle's
    fold_bn of the kept channels, rounded to f16: within one f16 step."""
    cfg = synth.RESNET50
    w, tables = synth.make_resnet_weights(cfg), synth.make_resnet_tables(cfg)
    wide = widen_all(w)
    blocks = synth.resnet_blocks(cfg)
    with binding.ElasticModel.resnet(cfg, w, tables, max_batch=1) as model:
        for m in (0, 3):
            for i in (0, 3, 15):
                cin, wd, _, _ = blocks[i]
                A, B = tables[m]["a"][i].astype(np.int64), tables[m]["b"][i].astype(np.int64)
                p = f"b{i}."

                def bn(name, idx):
                    return [wide[f"{p}{name}.{s}"][idx] for s in ("g", "b", "mean", "var")]

                W1, b1 = orr.fold_bn(wide[p + "conv1_w"][A], *bn("bn1", A))
                W2, b2 = orr.fold_bn(wide[p + "conv2_w"][B][:, A], *bn("bn2", B))
                W3, b3 = orr.fold_bn(wide[p + "conv3_w"][:, B], *bn("bn3", slice(None)))
                want = {0: W1[:, :, 0, 0], 1: b1, 2: W2.transpose(0, 2, 3, 1), 3: b2, 4: W3[:, :, 0, 0], 5: b3}
                for which, ref in want.items():
                    ref = np.ascontiguousarray(ref)
                    if which % 2 == 0:
                        got = model.export_packed(m, i, which, np.empty(ref.shape, np.uint16))
                        rb = ref.astype(np.float16).view(np.uint16).astype(np.int32)
                        assert np.max(np.abs(got.astype(np.int32) - rb)) <= 1, (m, i, which)
                    else:
                        got = model.export_packed(m, i, which, np.empty(ref.shape, np.float32))
                        assert np.allclose(got, ref, rtol=1e-6, atol=1e-7), (m, i, which)


def test_resnet_forward_host_batches_equals_device_forward():
    import torch
    cfg = SMALL
    w, tables = synth.make_resnet_weights(cfg), synth.make_resnet_tables(cfg)
    nb, B = 4, 2
    imgs = [torch.from_numpy(synth.make_images(cfg, B, seed=200 + i)).pin_memory().numpy() for i in range(nb)]
    with binding.ElasticModel.resnet(cfg, w, tables, max_batch=B) as model:
        model.set_mode(3)
        outs = [np.zeros((B, cfg.classes), np.float32) for _ in range(nb)]
        model.forward_host_batches(imgs, outs)
        for i in range(nb):
            assert np.array_equal(outs[i].astype(np.float64), _run(model, dev(imgs[i]), B, cfg.classes, 3)), i


def test_resnet_batch_1_and_ragged_and_switch():
    cfg = SMALL
    w, tables = synth.make_resnet_weights(cfg), synth.make_resnet_tables(cfg)
    img = synth.make_images(cfg, 7, seed=5)
    with binding.ElasticModel.resnet(cfg, w, tables, max_batch=7) as model:
        x1, x7 = dev(img[:1]), dev(img)
        refs = [resnet_logits(cfg, tables, m, img) for m in range(cfg.n_modes)]
        for m in range(cfg.n_modes):
            assert rel_err(_run(model, x1, 1, cfg.classes, m), refs[m][:1]) <= TOL
            assert rel_err(_run(model, x7, 7, cfg.classes, m), refs[m]) <= TOL
        # switching back and forth reproduces each mode's logits bit for bit
        first = [_run(model, x7, 7, cfg.classes, m) for m in range(cfg.n_modes)]
        for m in (3, 0, 2, 1, 3):
            assert np.array_equal(_run(model, x7, 7, cfg.classes, m), first[m])


@pytest.mark.parametrize("img_size", [45, 34])
def test_resnet_odd_and_even_image_sizes(img_size):
    """The stem at sizes other than 32 and 224: 45 is odd (the last 2x2 pixel
    block of the space-to-depth image is half outside the image), 34 gives a
    stem output of 17 (odd, so no pixel block tiles it evenly)."""
    cfg = dataclasses.replace(SMALL, name=f"resnet50_{img_size}px", img=img_size)
    w, tables = synth.make_resnet_weights(cfg), synth.make_resnet_tables(cfg)
    img = synth.make_images(cfg, 9, seed=11)
    with binding.ElasticModel.resnet(cfg, w, tables, max_batch=9) as model:
        x = dev(img)
        for m in (0, cfg.n_modes - 1):
            got, ref = _run(model, x, 9, cfg.classes, m), resnet_logits(cfg, tables, m, img)
            _report(f"resnet50 {img_size}px mode {m}", got, ref)
            assert rel_err(got, ref) <= TOL


def test_resnet_kept_counts_not_multiple_of_8():
    """Kept sets of 5, 13, 27 ... channels (zero-padded inside the library)."""
    cfg = SMALL
    w = synth.make_resnet_weights(cfg)
    rng = np.random.default_rng(7)
    t = {"a": [], "b": []}
    for (_, wd, _, _) in synth.resnet_blocks(cfg):
        for key in ("a", "b"):
            k = int(rng.integers(1, wd + 1))
            if k % 8 == 0:
                k -= 1 if k > 1 else 0
            t[key].append(np.sort(rng.choice(wd, size=max(k, 1), replace=False)).astype(np.int32))
    tables = [t]
    img = synth.make_images(cfg, 32, seed=9)
    with binding.ElasticModel.resnet(cfg, w, tables, max_batch=32) as model:
        got = _run(model, dev(img), 32, cfg.classes, 0)
    ref = resnet_logits(cfg, tables, 0, img)
    assert rel_err(got, ref) <= TOL


def test_resnet_profile_records_and_queries():
    cfg = SMALL
    w, tables = synth.make_resnet_weights(cfg), synth.make_resnet_tables(cfg)
    img = synth.make_images(cfg, 4)
    with binding.ElasticModel.resnet(cfg, w, tables, max_batch=4) as model:
        x = dev(img)
        model.profile(True)
        _run(model, x, 4, cfg.classes, 1)
        recs = model.profile_read()
        assert len(recs) == model.query(binding.Q_LAUNCHES, 1)
        kinds = {r["kind"] for r in recs}
        assert {"gemm", "im2col", "pool", "head"} <= kinds
        assert all(r["ms"] >= 0 for r in recs)
        # MACs per image of each mode, counted from the kept widths
        full = model.query(binding.Q_MODE_MACS, 0)
        assert model.query(binding.Q_MODE_MACS, 3) < model.query(binding.Q_MODE_MACS, 1) < full
        assert model.query(binding.Q_PACKED_BYTES, 3) < model.query(binding.Q_PACKED_BYTES, 0)


def test_resnet_fp32_stored_weights_and_images():
    """weight_dtype ELASTO_F32: fp32 images through the stem gather, fp32
    weights rounded to f16 after BN folding."""
    cfg = dataclasses.replace(SMALL, dtype=synth.F32)
    w, tables = synth.make_resnet_weights(cfg), synth.make_resnet_tables(cfg)
    img = synth.make_images(cfg, 16, seed=3)
    assert img.dtype == np.float32
    with binding.ElasticModel.resnet(cfg, w, tables, max_batch=16) as model:
        x = dev(img)
        for m in (0, 3):
            got = _run(model, x, 16, cfg.classes, m)
            _report(f"resnet50 32px fp32-stored mode {m}", got, resnet_logits(cfg, tables, m, img))
            assert rel_err(got, resnet_logits(cfg, tables, m, img)) <= TOL
