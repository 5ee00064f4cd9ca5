"""elasto_forward_noalloc: the forward for callers that may not allocate
device memory while serving (a process whose memory manager owns the whole
GPU after start-up, or a latency-critical loop that cannot take the device
synchronisation an allocation may cause). Its activations live in a fixed
64 MiB array inside the library instead of the handle's workspace.

Checked here, through the C-ABI: on two calls in a row its logits match
elasto_forward's on the same inputs within the parity tolerance the other
tests use, and the fp64 oracle's directly; the device's free memory does not
change across calls; and a batch whose scratch does not fit in the array is
rejected with a clear error. This file is collected last on purpose."""
import numpy as np
import pytest

from helpers import dev, empty_dev, rel_err, stream_handle
from oracle import vit as ov
from paper_2609_10018_gb300 import binding, synth

pytestmark = pytest.mark.gpu

TOL = 1e-2


def _logits_both_ways(model, cfg, images, batch, mode):
    import torch
    s = stream_handle()
    model.set_mode(mode)
    ref = empty_dev((batch, cfg.classes), torch.float32)
    model.forward(s, images.data_ptr(), batch, ref.data_ptr())
    outs = []
    for _ in range(2):  # two calls in a row share (and overwrite) the static scratch
        o = empty_dev((batch, cfg.classes), torch.float32)
        binding.elasto_forward_noalloc(model.handle, s, images.data_ptr(), batch, o.data_ptr())
        outs.append(o)
    model.sync_status(s)
    return ref.cpu().numpy().astype(np.float64), [o.cpu().numpy().astype(np.float64) for o in outs]


def test_noalloc_matches_forward_and_oracle_tiny_all_modes():
    cfg = synth.TINY
    w = synth.make_vit_weights(cfg)
    wide = ov.widen_all(w)
    tables = synth.make_vit_tables(cfg)
    img = synth.make_images(cfg, cfg.batch)
    images = dev(img)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=cfg.batch) as model:
        for m, t in enumerate(tables):
            ref, outs = _logits_both_ways(model, cfg, images, cfg.batch, m)
            want = ov.vit_forward_sliced(wide, cfg, t["heads"], t["mlp"], img)
            for o in outs:
                assert rel_err(o, ref) <= TOL
                assert rel_err(o, want) <= TOL


def test_noalloc_leaves_free_device_memory_unchanged():
    """After a first call (which looks up the array's address and builds the
    launch plans), further calls change the device's free memory by nothing:
    they allocate no device memory."""
    import torch
    cfg = synth.TINY
    w = synth.make_vit_weights(cfg)
    tables = synth.make_vit_tables(cfg)
    B = 32  # beyond max_batch: the handle's workspace could not hold it
    images = dev(synth.make_images(cfg, B))
    out = empty_dev((B, cfg.classes), torch.float32)
    s = stream_handle()
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=1) as model:
        for m in range(len(tables)):
            model.set_mode(m)
            binding.elasto_forward_noalloc(model.handle, s, images.data_ptr(), B, out.data_ptr())
        model.sync_status(s)
        free0, _ = torch.cuda.mem_get_info()
        for _ in range(3):
            for m in range(len(tables)):
                model.set_mode(m)
                binding.elasto_forward_noalloc(model.handle, s, images.data_ptr(), B, out.data_ptr())
        model.sync_status(s)
        free1, _ = torch.cuda.mem_get_info()
        assert free1 == free0


def test_noalloc_vit_b_largest_batch_and_limit():
    import torch
    cfg = synth.VIT_B
    w = synth.make_vit_weights(cfg)
    tables = synth.make_vit_tables(cfg)
    cap = 18  # 64 MiB / about 3.6 MB of activations per image in the full mode
    images = dev(synth.make_images(cfg, cap + 1))
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=cap) as model:
        ref, outs = _logits_both_ways(model, cfg, images, cap, 0)
        for o in outs:
            assert rel_err(o, ref) <= TOL
        too_big = empty_dev((cap + 1, cfg.classes), torch.float32)
        with pytest.raises(binding.ElastoError) as e:
            binding.elasto_forward_noalloc(model.handle, stream_handle(), images.data_ptr(), cap + 1,
                                           too_big.data_ptr())
        assert e.value.status == binding.ERR_INVALID_ARG
        assert "64 MiB" in str(e.value) and str(cap) in str(e.value)
