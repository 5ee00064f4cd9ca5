"""Each CUDA kernel on its own, through the C-ABI op entry points, against
the fp64 oracle's matching sub-step, at odd and ragged shapes."""
import numpy as np
import pytest

from helpers import bf16_to_f64, dev, empty_dev, stream_handle
from oracle import vit as ov
from paper_2609_10018_gb300 import binding, synth

pytestmark = pytest.mark.gpu


def _bf16(rng, shape, scale=1.0):
    return synth.f32_to_bf16_bits(rng.standard_normal(shape, dtype=np.float32) * np.float32(scale))


def _status():
    import torch
    return torch.zeros(1, dtype=torch.int32, device="cuda")


GEMM_CASES = [
    # M, N, K, epilogue
    (128, 256, 64, binding.EPI_BIAS_BF16),            # one tile
    (200, 576, 384, binding.EPI_BIAS_BF16),           # ragged M, 3-head QKV width
    (1000, 192, 48, binding.EPI_BIAS_BF16),           # K below one k-block (tiny patch projection)
    (333, 1000, 768, binding.EPI_BIAS_F32),           # N not a multiple of 32 (classifier width)
    (1537, 3072, 768, binding.EPI_BIAS_GELU_BF16),    # FC1
    (1537, 768, 3072, binding.EPI_BIAS_RESID_F32),    # FC2 with residual
    (257, 768, 0, binding.EPI_BIAS_RESID_F32),        # no kept channel: residual += bias
    (6304, 2304, 768, binding.EPI_BIAS_BF16),         # ViT-B QKV at batch 32
    (130, 200, 136, binding.EPI_BIAS_RELU_BF16),      # conv-like K
    (130, 64, 72, binding.EPI_BIAS_RESID_RELU_BF16),
    (64, 1152, 384, binding.EPI_BIAS_GELU_BF16),      # ViT-S 75 % MLP, M below one tile
    # f16 operands (ResNet-50 path)
    (200, 48, 576, binding.EPI_BIAS_RELU_F16),        # 3x3 conv of 64 kept channels into 48
    (130, 16, 72, binding.EPI_BIAS_F16),              # N below one 64-column chunk
    (1537, 256, 2048, binding.EPI_BIAS_RELU_F16),     # K >= 1536: CTA-pair kernel with f16
    (333, 1024, 136, binding.EPI_BIAS_RESID_RELU_F16),
    (6272, 2048, 512, binding.EPI_BIAS_RESID_RELU_F16),  # last conv3 of ResNet-50 at batch 128
]

F16_EPIS = (binding.EPI_BIAS_RELU_F16, binding.EPI_BIAS_F16, binding.EPI_BIAS_RESID_RELU_F16)


def _f16(rng, shape, scale=1.0):
    return (rng.standard_normal(shape, dtype=np.float32) * np.float32(scale)).astype(np.float16).view(np.uint16)


def _f16_to_f64(bits):
    a = bits.cpu().numpy() if hasattr(bits, "cpu") else np.asarray(bits)
    return a.view(np.float16).astype(np.float64)


@pytest.mark.parametrize("M,N,K,epi", GEMM_CASES)
def test_gemm_epilogues_match_fp64(M, N, K, epi):
    import torch
    rng = np.random.default_rng(M * 7 + N * 3 + K)
    half = epi in F16_EPIS
    gen, dec = (_f16, _f16_to_f64) if half else (_bf16, bf16_to_f64)
    A = gen(rng, (M, max(K, 8)))[:, :K].copy() if K else np.zeros((M, 0), np.uint16)
    W = gen(rng, (N, max(K, 8)), 0.05)[:, :K].copy() if K else np.zeros((N, 0), np.uint16)
    bias = rng.standard_normal(N).astype(np.float32)
    ref = dec(A) @ dec(W).T + bias
    f32_out = epi in (binding.EPI_BIAS_F32, binding.EPI_BIAS_RESID_F32)
    resid = None
    if epi == binding.EPI_BIAS_RESID_F32:
        x0 = rng.standard_normal((M, N)).astype(np.float32)
        out = dev(x0)
        ref = ref + x0
    else:
        out = empty_dev((M, N), torch.float32 if f32_out else torch.uint16)
    if epi == binding.EPI_BIAS_GELU_BF16:
        ref = ov.gelu(ref)
    elif epi == binding.EPI_BIAS_RELU_BF16:
        ref = np.maximum(ref, 0)
    elif epi == binding.EPI_BIAS_RELU_F16:
        ref = np.maximum(ref, 0)
    elif epi in (binding.EPI_BIAS_RESID_RELU_BF16, binding.EPI_BIAS_RESID_RELU_F16):
        r = gen(rng, (M, N))
        resid = dev(r)
        ref = np.maximum(ref + dec(r), 0)
    st = _status()
    dA = dev(A) if K else None
    dW = dev(W) if K else None
    db = dev(bias)
    binding.elasto_op_gemm(stream_handle(), dA.data_ptr() if K else None, dW.data_ptr() if K else None,
                           db.data_ptr(), out.data_ptr(), resid.data_ptr() if resid is not None else None,
                           M, N, K, epi, st.data_ptr())
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    got = out.cpu().numpy().astype(np.float64) if f32_out else dec(out)
    scale = float(np.max(np.abs(ref)))
    if f32_out:
        assert np.all(np.abs(got - ref) <= 1e-5 * scale + 1e-6 * np.abs(ref)), float(np.max(np.abs(got - ref)))
    elif half:  # one f16 rounding of the fp32 result
        assert np.all(np.abs(got - ref) <= 2.0 ** -11 * np.abs(ref) + 1e-5 * scale), float(np.max(np.abs(got - ref)))
    else:  # one bf16 rounding of the fp32 result
        assert np.all(np.abs(got - ref) <= 2.0 ** -8 * np.abs(ref) + 1e-5 * scale), float(np.max(np.abs(got - ref)))


def test_gemm_full_size_outproj_sampled_rows():
    """ViT-B out-projection at batch 256 (M = 50432 = 394 tiles), sampled rows."""
    import torch
    M, N, K = 256 * 197, 768, 768
    rng = np.random.default_rng(11)
    A = _bf16(rng, (M, K))
    W = _bf16(rng, (N, K), 0.03)
    bias = rng.standard_normal(N).astype(np.float32)
    x0 = rng.standard_normal((M, N)).astype(np.float32)
    out = dev(x0)
    dA, dW, db = dev(A), dev(W), dev(bias)
    binding.elasto_op_gemm(stream_handle(), dA.data_ptr(), dW.data_ptr(), db.data_ptr(),
                           out.data_ptr(), None, M, N, K, binding.EPI_BIAS_RESID_F32, 0)
    torch.cuda.synchronize()
    rows = np.concatenate([np.arange(0, 130), rng.choice(M, 300, replace=False), np.arange(M - 130, M)])
    got = out.cpu().numpy()[rows].astype(np.float64)
    ref = bf16_to_f64(A[rows]) @ bf16_to_f64(W).T + bias + x0[rows]
    assert np.max(np.abs(got - ref)) <= 1e-5 * np.max(np.abs(ref))


@pytest.mark.parametrize("rows,d", [(1000, 192), (333, 384), (2051, 768), (7, 1024)])
def test_layernorm_matches_fp64(rows, d):
    import torch
    rng = np.random.default_rng(rows + d)
    x = (rng.standard_normal((rows, d)) * 2.0 + 0.7).astype(np.float32)
    g = (1 + 0.1 * rng.standard_normal(d)).astype(np.float32)
    b = (0.1 * rng.standard_normal(d)).astype(np.float32)
    y = empty_dev((rows, d), torch.uint16)
    dx, dg, db = dev(x), dev(g), dev(b)
    binding.elasto_op_layernorm(stream_handle(), dx.data_ptr(), dg.data_ptr(), db.data_ptr(), y.data_ptr(), rows, d)
    torch.cuda.synchronize()
    ref = ov.layer_norm(x.astype(np.float64), g, b)
    got = bf16_to_f64(y)
    assert np.all(np.abs(got - ref) <= 2.0 ** -8 * np.abs(ref) + 1e-5 * np.max(np.abs(ref)))


@pytest.mark.parametrize("rows,cols", [(100, 1), (64, 10), (300, 197), (17, 1000)])
def test_softmax_matches_fp64(rows, cols):
    import torch
    rng = np.random.default_rng(rows * cols)
    x = (rng.standard_normal((rows, cols)) * 4).astype(np.float32)
    y = empty_dev((rows, cols), torch.float32)
    dx = dev(x)
    binding.elasto_op_softmax(stream_handle(), dx.data_ptr(), y.data_ptr(), rows, cols)
    torch.cuda.synchronize()
    ref = ov.softmax_rows(x.astype(np.float64))
    got = y.cpu().numpy().astype(np.float64)
    assert np.max(np.abs(got - ref)) <= 1e-6
    assert np.allclose(got.sum(1), 1.0, atol=1e-5)


# the last three give each of the 152 persistent CTAs four or more items, so
# every K/V slot and Q buffer is reused (2 slots at n = 256, 3 below 209 keys)
ATTN_CASES = [(2, 197, 3), (3, 65, 2), (1, 256, 1), (2, 1, 1), (2, 17, 4), (1, 129, 12),
              (160, 256, 4), (120, 65, 6), (100, 129, 7), (64, 197, 12)]


@pytest.mark.parametrize("B,n,h", ATTN_CASES)
def test_attention_matches_fp64(B, n, h):
    import torch
    rng = np.random.default_rng(B * 1000 + n * 10 + h)
    qkv = _bf16(rng, (B, n, 3, h, 64))
    out = empty_dev((B, n, h * 64), torch.uint16)
    st = _status()
    dq = dev(qkv)
    binding.elasto_op_attention(stream_handle(), dq.data_ptr(), out.data_ptr(), B, n, h, st.data_ptr())
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    q = bf16_to_f64(qkv)
    ref = np.concatenate([ov.attention(q[:, :, 0, j], q[:, :, 1, j], q[:, :, 2, j], 64) for j in range(h)], axis=-1)
    got = bf16_to_f64(out)
    # P is rounded to bf16 before P.V and O to bf16 at the end
    assert np.max(np.abs(got - ref)) <= 1e-2 * np.max(np.abs(ref)), float(np.max(np.abs(got - ref)))


def test_attention_reference_raised_by_a_late_large_score():
    """Rows whose largest score lies far beyond the first 32 keys (and far
    above their scores): the one-pass softmax must raise its reference and
    rescale the P it already wrote. Rows 0-5 and 130-135 attend almost
    entirely to key 150 (q . k = 768 there, |q . k| ~ 20 elsewhere)."""
    import torch
    B, n, h = 2, 197, 3
    rng = np.random.default_rng(77)
    qkv = (rng.standard_normal((B, n, 3, h, 64)) * 0.3).astype(np.float32)
    rows = np.r_[0:6, 130:136]
    qkv[:, rows, 0, :, :] = 3.5
    qkv[:, 150, 1, :, :] = 3.5
    qkv = synth.f32_to_bf16_bits(qkv)
    out = empty_dev((B, n, h * 64), torch.uint16)
    st = _status()
    dq = dev(qkv)
    binding.elasto_op_attention(stream_handle(), dq.data_ptr(), out.data_ptr(), B, n, h, st.data_ptr())
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    q = bf16_to_f64(qkv)
    ref = np.concatenate([ov.attention(q[:, :, 0, j], q[:, :, 1, j], q[:, :, 2, j], 64) for j in range(h)], axis=-1)
    got = bf16_to_f64(out)
    assert np.all(np.isfinite(got))
    assert np.max(np.abs(got - ref)) <= 1e-2 * np.max(np.abs(ref)), float(np.max(np.abs(got - ref)))
    # those rows are (almost) the value row of key 150
    assert np.allclose(got[:, rows], np.concatenate([q[:, 150:151, 2, j] for j in range(h)], axis=-1)
                       .repeat(len(rows), axis=1), atol=2e-2)


def test_attention_full_size_sampled():
    """ViT-B shape at batch 256: 256 x 12 heads x 197 tokens; sampled images."""
    import torch
    B, n, h = 256, 197, 12
    rng = np.random.default_rng(5)
    qkv = _bf16(rng, (B, n, 3, h, 64))
    out = empty_dev((B, n, h * 64), torch.uint16)
    dq = dev(qkv)
    binding.elasto_op_attention(stream_handle(), dq.data_ptr(), out.data_ptr(), B, n, h, 0)
    torch.cuda.synchronize()
    got = bf16_to_f64(out)
    for b in (0, 1, 128, 255):
        q = bf16_to_f64(qkv[b])
        ref = np.concatenate([ov.attention(q[:, 0, j], q[:, 1, j], q[:, 2, j], 64) for j in range(h)], axis=-1)
        assert np.max(np.abs(got[b] - ref)) <= 1e-2 * np.max(np.abs(ref))


CONV_CASES = [
    # B, H, W, C, N, k, stride, pad, relu
    (3, 13, 11, 24, 40, 3, 1, 1, True),      # ragged image, channels below one 64-group
    (2, 15, 15, 64, 128, 3, 2, 1, True),     # stride 2, odd size
    (5, 7, 7, 136, 48, 1, 2, 0, False),      # strided 1x1 projection, 3 channel groups (ragged)
    (1, 56, 56, 64, 64, 3, 1, 1, True),      # ResNet-50 stage 1 conv2 at batch 1
    (40, 2, 2, 512, 512, 3, 1, 1, True),     # whole images per tile (nb > 1)
    (4, 9, 9, 16, 24, 3, 2, 1, False),       # N below one 64-column chunk, stride 2 (16-channel k-blocks)
    (3, 11, 13, 8, 40, 3, 1, 1, True),       # 8 channels: 16-wide k-blocks, half of each zero
    (2, 20, 20, 16, 64, 4, 1, 2, True),      # 4 x 4 taps on 16 channels (the space-to-depth stem's shape)
    # stride 1 on 64-channel groups runs as halo tiles (taps = shifted windows of one load per group):
    (2, 28, 28, 128, 128, 3, 1, 1, True),    # ResNet-50 stage 2 shape: two groups, W streamed per tap
    (3, 14, 14, 256, 320, 3, 1, 1, False),   # four groups, two N tiles (the second ragged)
    (2, 9, 30, 72, 64, 5, 1, 2, True),       # 5 x 5, ragged second group, 3 row blocks of 3 rows
    (2, 10, 12, 64, 64, 3, 1, 0, True),      # no padding
]


@pytest.mark.parametrize("B,H,W,C,N,k,stride,pad,relu", CONV_CASES)
def test_conv2d_implicit_gemm_matches_fp64(B, H, W, C, N, k, stride, pad, relu):
    import torch
    from oracle import resnet as orr
    rng = np.random.default_rng(B * 1000 + H * 10 + C)
    x = _f16(rng, (B, H, W, C))
    wt = (rng.standard_normal((N, C, k, k)) * np.sqrt(2.0 / (C * k * k))).astype(np.float16)
    bias = rng.standard_normal(N).astype(np.float32) * 0.1
    cp = 16 if C <= 16 else (C + 63) // 64 * 64
    packed = np.zeros((N, k, k, cp), np.float16)
    packed[..., :C] = wt.transpose(0, 2, 3, 1)
    ref = orr.conv2d(_f16_to_f64(x), wt.astype(np.float64), stride, pad) + bias
    if relu:
        ref = np.maximum(ref, 0)
    Ho, Wo = ref.shape[1], ref.shape[2]
    out = empty_dev((B, Ho, Wo, N), torch.uint16)
    out.fill_(0x7E00)  # f16 NaN: every output must be written
    st = _status()
    dx, dw, db = dev(x), dev(packed.view(np.uint16)), dev(bias)
    binding.elasto_op_conv2d(stream_handle(), dx.data_ptr(), B, H, W, C, dw.data_ptr(), N, k, stride, pad,
                             db.data_ptr(), relu, out.data_ptr(), st.data_ptr())
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    got = _f16_to_f64(out)
    assert np.all(np.isfinite(got))
    scale = float(np.max(np.abs(ref)))
    assert np.all(np.abs(got - ref) <= 2.0 ** -10 * np.abs(ref) + 1e-4 * scale), float(np.max(np.abs(got - ref)))


def test_bounded_wait_gives_up_and_leaves_the_context_usable():
    """A device-side wait that nothing satisfies ends after its limit with
    ELASTO_ERR_TIMEOUT in the status word (no trap, no hang); the next launch
    on the same context works. An armed wait returns at once."""
    import time
    import torch
    st = _status()
    el = torch.zeros(1, dtype=torch.int64, device="cuda")
    binding.elasto_op_bounded_wait(stream_handle(), True, st.data_ptr(), el.data_ptr())
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert int(el.item()) < 10_000_000                     # well under 10 ms
    t0 = time.perf_counter()
    binding.elasto_op_bounded_wait(stream_handle(), False, st.data_ptr(), el.data_ptr())
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    assert int(st.item()) == binding.ERR_TIMEOUT
    assert 0.9e9 <= int(el.item()) <= 3e9 and wall < 10.0
    # the context is still usable: an attention launch right after matches the oracle
    test_attention_matches_fp64(2, 65, 2)


def test_grid_barrier_gives_up_and_leaves_the_context_usable():
    """The grid-wide barrier of the one-launch forward: two barriers over one
    block per SM pass at once; a barrier waiting for arrivals that never come
    ends after its limit with ELASTO_ERR_TIMEOUT (every block leaves through
    the abort flag, no hang), and the context stays usable."""
    import time
    import torch
    st = _status()
    el = torch.zeros(1, dtype=torch.int64, device="cuda")
    sync = torch.zeros(2, dtype=torch.int32, device="cuda")
    binding.elasto_op_grid_barrier(stream_handle(), False, sync.data_ptr(), st.data_ptr(), el.data_ptr())
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert int(el.item()) < 10_000_000
    assert int(sync[0].item()) == 2 * torch.cuda.get_device_properties(0).multi_processor_count
    t0 = time.perf_counter()
    binding.elasto_op_grid_barrier(stream_handle(), True, sync.data_ptr(), st.data_ptr(), el.data_ptr())
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    assert int(st.item()) == binding.ERR_TIMEOUT
    assert int(sync[1].item()) == 1  # the abort flag
    assert 0.9e9 <= int(el.item()) <= 3e9 and wall < 10.0
    test_attention_matches_fp64(2, 65, 2)
