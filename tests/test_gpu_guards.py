"""Out-of-bounds write detection without a device memory checker: every buffer
of a handle's arena is followed by a guard zone filled with 0xA5 at create
time. Every `with ElasticModel(...)` block of the GPU tests checks the zones
when it ends; here the forwards most likely to write past an end (ragged
batches, one image, the largest batch, every mode) are checked explicitly,
and the checker itself is shown to find a damaged zone and name its buffer."""
import dataclasses

import pytest

from helpers import dev, empty_dev, stream_handle
from paper_2609_10018_gb300 import binding, synth

pytestmark = pytest.mark.gpu


def _forward_all(model, cfg, n_modes, batches):
    import torch
    img = dev(synth.make_images(cfg, max(batches)))
    out = empty_dev((max(batches), cfg.classes), torch.float32)
    for m in range(n_modes):
        model.set_mode(m)
        for b in batches:
            model.forward(stream_handle(), img.data_ptr(), b, out.data_ptr())
    model.sync_status(stream_handle())


@pytest.mark.parametrize("cfg,max_batch,batches", [
    (synth.TINY, 13, (1, 7, 8, 13)),
    (synth.VIT_B, 9, (1, 8, 9)),
], ids=["tiny", "vit_b16"])
def test_vit_forwards_leave_guards_intact(cfg, max_batch, batches):
    w, tables = synth.make_vit_weights(cfg), synth.make_vit_tables(cfg)
    with binding.ElasticModel.vit(cfg, w, tables, max_batch=max_batch) as model:
        assert model.query(binding.Q_GUARD_ZONES) > 10
        _forward_all(model, cfg, len(tables), batches)
        assert binding.elasto_check_guards(model.handle, stream_handle()) == 0


def test_resnet_forwards_leave_guards_intact():
    cfg = dataclasses.replace(synth.RESNET50, name="resnet50_40px", img=40, classes=10)
    w, tables = synth.make_resnet_weights(cfg), synth.make_resnet_tables(cfg)
    with binding.ElasticModel.resnet(cfg, w, tables, max_batch=5) as model:
        assert model.query(binding.Q_GUARD_ZONES) > 10
        _forward_all(model, cfg, cfg.n_modes, (1, 3, 5))
        assert binding.elasto_check_guards(model.handle, stream_handle()) == 0


@pytest.mark.parametrize("which", ["first", "middle", "last"])
def test_checker_finds_a_damaged_zone(which):
    cfg = synth.TINY
    w, tables = synth.make_vit_weights(cfg), synth.make_vit_tables(cfg)
    model = binding.ElasticModel.vit(cfg, w, tables, max_batch=2)
    try:
        nz = model.query(binding.Q_GUARD_ZONES)
        zone = {"first": 0, "middle": nz // 2, "last": nz - 1}[which]
        assert binding.elasto_check_guards(model.handle, stream_handle()) == 0
        binding.elasto_debug_damage_guard(model.handle, zone)
        with pytest.raises(binding.ElastoError) as e:
            binding.elasto_check_guards(model.handle, stream_handle())
        assert e.value.status == binding.ERR_GUARD
        assert "1 guard zone(s) overwritten" in str(e.value)
        with pytest.raises(binding.ElastoError):
            binding.elasto_debug_damage_guard(model.handle, nz)
    finally:
        model.close()
