"""One-image forwards as one persistent launch (csrc/persistent.cu): every
mode of the tiny (bf16), ViT-S/16 and ViT-B/16 models against the fp64
oracle, degenerate layers (no head, no MLP channel, channel counts that are
not multiples of 8), embedding-pruned modes, the agreement with the
kernel-by-kernel forward, repeatability, CUDA-graph replay, and the cases
that keep the kernel-by-kernel path."""
import numpy as np
import pytest

from helpers import dev, empty_dev, rel_err, stream_handle
from oracle import vit as ov
from oracle_pool import vit_logits
from paper_2609_10018_gb300 import binding, synth

pytestmark = pytest.mark.gpu

TOL = 1e-2  # max |logit error| / max |logit|, as for every ViT parity test


def _one(model, x_dev, classes, mode):
    import torch
    out = empty_dev((1, classes), torch.float32)
    model.set_mode(mode)
    model.forward(stream_handle(), x_dev.data_ptr(), 1, out.data_ptr())
    model.sync_status(stream_handle())
    return out.cpu().numpy().astype(np.float64)


def _per_image(model, img, classes, mode):
    return np.concatenate([_one(model, dev(img[i:i + 1]), classes, mode) for i in range(len(img))])


def _tiny_bf16():
    return synth.vit_small_variant(synth.TINY, dtype=synth.BF16)


def _check_modes(cfg, tables, n_img, max_batch=4, cross_tol=TOL):
    """Every mode, n_img images one at a time: one launch against the oracle
    and against the kernel-by-kernel forward of the same image."""
    w = synth.make_vit_weights(cfg)
    img = synth.make_images(cfg, n_img)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=max_batch) as model:
        assert model.query(binding.Q_ONE_LAUNCH, 0) == 0  # opt-in
        model.set_one_launch(True)
        for m in range(len(tables)):
            assert model.query(binding.Q_ONE_LAUNCH, m) == 1, (cfg.name, m)
        for m in range(len(tables)):
            model.set_one_launch(True)
            got = _per_image(model, img, cfg.classes, m)
            model.set_one_launch(False)
            kbk = _per_image(model, img, cfg.classes, m)
            model.set_one_launch(True)
            ref = vit_logits(cfg, tables, m, img, chunk=1)
            e_ref, e_kbk = rel_err(got, ref), rel_err(got, kbk)
            print(f"{cfg.name} mode {m}: one launch vs oracle {e_ref:.2e}, vs kernel by kernel {e_kbk:.2e}, "
                  f"kernel by kernel vs oracle {rel_err(kbk, ref):.2e}")
            assert e_ref <= TOL, (cfg.name, m, e_ref)
            assert e_kbk <= cross_tol, (cfg.name, m, e_kbk)
            assert np.array_equal(np.argmax(got, 1), np.argmax(kbk, 1)) or e_kbk <= 1e-3


def test_tiny_every_mode_and_degenerate_layers():
    cfg = _tiny_bf16()
    t = synth.make_vit_tables(cfg)
    rng = np.random.default_rng(7)
    odd = {"heads": [np.sort(rng.choice(3, k, replace=False)).astype(np.int32) for k in (0, 1, 3, 2, 0, 1)],
           "mlp": [np.sort(rng.choice(768, k, replace=False)).astype(np.int32) for k in (100, 0, 768, 1, 0, 37)]}
    _check_modes(cfg, t + [odd], n_img=12)


def test_tiny_nested_prefix_copy():
    cfg = _tiny_bf16()
    tables = synth.make_vit_tables(cfg)
    w = synth.make_vit_weights(cfg)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=2) as model:
        assert model.query(binding.Q_PREFIX_SHARED) == 1
    _check_modes(cfg, tables, n_img=8, max_batch=2)


def test_vit_s_every_mode():
    _check_modes(synth.VIT_S, synth.make_vit_tables(synth.VIT_S), n_img=4)


def test_vit_b_every_mode():
    _check_modes(synth.VIT_B, synth.make_vit_tables(synth.VIT_B), n_img=2, max_batch=1)


def test_embedding_pruned_modes():
    cfg = synth.VIT_S
    tables = synth.with_embedding(cfg, synth.make_vit_tables(cfg), [None, 320, 256, 200])
    _check_modes(cfg, tables, n_img=3)


def test_repeatable_and_graph_replay():
    """Bit-identical on repeat (no atomics: fixed split order), and the same
    logits when replayed from a captured CUDA graph."""
    import torch
    cfg = synth.VIT_S
    w, tables = synth.make_vit_weights(cfg), synth.make_vit_tables(cfg)
    img = synth.make_images(cfg, 3)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=1) as model:
        model.set_one_launch(True)
        model.set_mode(2)
        x = [dev(img[i:i + 1]) for i in range(3)]
        first = [_one(model, xi, cfg.classes, 2) for xi in x]
        assert all(np.array_equal(_one(model, xi, cfg.classes, 2), f) for xi, f in zip(x, first))
        stream = torch.cuda.Stream()
        src = torch.empty_like(x[0])
        out = empty_dev((1, cfg.classes), torch.float32)
        src.copy_(x[0])
        with torch.cuda.stream(stream):
            model.forward(stream.cuda_stream, src.data_ptr(), 1, out.data_ptr())  # warm-up outside capture
        stream.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            model.forward(torch.cuda.current_stream().cuda_stream, src.data_ptr(), 1, out.data_ptr())
        for i in (1, 2, 0):
            src.copy_(x[i])
            g.replay()
            torch.cuda.synchronize()
            assert np.array_equal(out.cpu().numpy().astype(np.float64), first[i]), i
        model.sync_status(stream_handle())


def test_profile_shows_one_launch():
    cfg = _tiny_bf16()
    w, tables = synth.make_vit_weights(cfg), synth.make_vit_tables(cfg)
    img = dev(synth.make_images(cfg, 1))
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=4) as model:
        model.set_one_launch(True)
        model.profile(True)
        _one(model, img, cfg.classes, 0)
        recs = model.profile_read()
        assert [r["kind"] for r in recs] == ["one_launch"]
        assert recs[0]["ms"] > 0
        model.set_one_launch(False)
        _one(model, img, cfg.classes, 0)
        kinds = [r["kind"] for r in model.profile_read()]
        assert "one_launch" not in kinds and kinds.count("attention") == cfg.layers


def test_fp32_stored_models_keep_the_kernel_by_kernel_path():
    """fp32 weights run as two bf16 planes, which the one-launch plan does
    not carry: the query says so and the forward still matches the oracle."""
    cfg = synth.TINY
    assert cfg.dtype == synth.F32
    w, tables = synth.make_vit_weights(cfg), synth.make_vit_tables(cfg)
    img = synth.make_images(cfg, 2)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=2) as model:
        model.set_one_launch(True)
        assert model.query(binding.Q_ONE_LAUNCH, 0) == 0
        got = _per_image(model, img, cfg.classes, 1)
    ref = ov.vit_forward_sliced(ov.widen_all(w), cfg, tables[1]["heads"], tables[1]["mlp"], img)
    assert rel_err(got, ref) <= TOL
