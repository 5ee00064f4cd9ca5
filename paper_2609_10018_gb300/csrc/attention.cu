// Fused multi-head attention over the kept heads only (Eq. 2-3 restricted to
// the DN's head set H; heads outside H were removed from W^Q, W^K, W^V at
// pack time, so this kernel never sees them).
//
// Input: qkv [B, n, 3, h_m, 64] bf16 exactly as the QKV GEMM writes it (q | k |
// v blocks, kept heads in ascending order). Output: [B, n, h_m * 64] bf16,
// the heads concatenated in the same order (the K axis of the sliced W^O).
//
// One CTA per (image, kept head); for each 128-query tile:
//   TMA: Q tile (128 x 64), K and V (n_pad x 64, once), 3-D maps so that rows
//        past n read as zero;
//   tcgen05.mma  S = Q K^T  (M=128, N=n_pad, K=64) into TMEM;
//   4 warps, one query row per thread (TMEM lane = row): row max and
//        exp2-based softmax numerators over the n valid keys in fp32, written
//        as bf16 P into shared memory in the 128B-swizzled K-major layout;
//   tcgen05.mma  O = P V  (M=128, N=64, K=n_pad; V is read MN-major);
//   epilogue: O row * (1 / row sum) -> bf16, 128 contiguous bytes per thread.
// Scale 1/sqrt(64) (the base model's head width; it does not change with the
// number of kept heads). n <= 256.
#include "common.h"
#include "ptx.cuh"

namespace elasto {

namespace {

constexpr int THREADS = 192;
constexpr int HD = 64;                      // head width d_i
constexpr int QT = 128;                     // queries per tile
constexpr int MAXK = 256;                   // max keys
constexpr int Q_BYTES = QT * HD * 2;        // 16 KB
constexpr int KV_BYTES = MAXK * HD * 2;     // 32 KB each
constexpr int P_ATOM = QT * 128;            // 64 keys x 128 rows, 16 KB
constexpr int P_BYTES = 4 * P_ATOM;         // 64 KB
constexpr size_t SMEM_BYTES = 1024 + Q_BYTES + 2 * KV_BYTES + P_BYTES + 128;
constexpr int TMEM_COLS = 256;

__global__ void __launch_bounds__(THREADS, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmKV,
                   bf16* __restrict__ out, int n, int n_pad, int heads, int* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sK = sQ + Q_BYTES;
  uint8_t* sV = sK + KV_BYTES;
  uint8_t* sP = sV + KV_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sP + P_BYTES);
  uint64_t* bar_q = bars + 0;   // Q tile landed
  uint64_t* bar_kv = bars + 1;  // K, V landed
  uint64_t* bar_s = bars + 2;   // S in TMEM
  uint64_t* bar_p = bars + 3;   // P in smem (128 arrivals)
  uint64_t* bar_o = bars + 4;   // O in TMEM
  uint64_t* bar_e = bars + 5;   // O read out (128 arrivals)
  uint64_t* drain = bars + 6;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 7);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int jj = blockIdx.x;  // kept-head index
  const int b = blockIdx.y;   // image
  const int w = heads * HD;
  const int n_tiles = (n + QT - 1) / QT;

  if (threadIdx.x == 0) {
    mbar_init(bar_q, 1);
    mbar_init(bar_kv, 1);
    mbar_init(bar_s, 1);
    mbar_init(bar_p, 128);
    mbar_init(bar_o, 1);
    mbar_init(bar_e, 128);
    mbar_init(drain, 1);
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      bool ok = true;
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmKV);
      mbar_expect_tx(bar_kv, 2 * n_pad * HD * 2);
      tma_load_3d(sK, &tmKV, bar_kv, w + jj * HD, 0, b);
      tma_load_3d(sV, &tmKV, bar_kv, 2 * w + jj * HD, 0, b);
      const uint32_t idesc_s = idesc_bf16_f32(QT, n_pad);
      const uint32_t idesc_o = idesc_bf16_f32(QT, HD, false, true);
      for (int qt = 0; qt < n_tiles && ok; ++qt) {
        const uint32_t ph = qt & 1;
        if (qt > 0) {  // previous tile's O must be read out before S overwrites TMEM
          if (!mbar_wait(bar_e, ph ^ 1)) { ok = false; break; }
        }
        mbar_expect_tx(bar_q, Q_BYTES);
        tma_load_3d(sQ, &tmQ, bar_q, jj * HD, qt * QT, b);
        if (!mbar_wait(bar_q, ph) || !mbar_wait(bar_kv, 0)) { ok = false; break; }
        tc_fence_after();
        const uint32_t q0 = smem_addr(sQ), k0 = smem_addr(sK);
#pragma unroll
        for (int k = 0; k < HD / 16; ++k)
          tc_mma(tmem, sdesc_sw128(q0 + k * 32, 16, 1024), sdesc_sw128(k0 + k * 32, 16, 1024), idesc_s, k != 0);
        tc_commit(bar_s);
        if (!mbar_wait(bar_p, ph)) { ok = false; break; }
        tc_fence_after();
        const uint32_t p0 = smem_addr(sP), v0 = smem_addr(sV);
        for (int s = 0; s < n_pad / 16; ++s) {
          const uint64_t ad = sdesc_sw128(p0 + (s >> 2) * P_ATOM + (s & 3) * 32, 16, 1024);
          const uint64_t bd = sdesc_sw128(v0 + s * 16 * 128, 16384, 1024);
          tc_mma(tmem, ad, bd, idesc_o, s != 0);
        }
        tc_commit(bar_o);
      }
      if (!ok) record_status(status, ELASTO_ERR_TIMEOUT);
      tc_commit(drain);
      mbar_wait(drain, 0);
      mbar_wait(bar_kv, 0);
    }
  } else if (warp >= 2) {
    const int qq = warp & 3;                 // TMEM lane quarter
    const int r = qq * 32 + lane;            // row within the query tile
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(qq * 32) << 16);
    const float kscale = 0.125f * 1.4426950408889634f;  // 1/sqrt(64) * log2(e)
    for (int qt = 0; qt < n_tiles; ++qt) {
      const uint32_t ph = qt & 1;
      if (!mbar_wait(bar_s, ph)) {
        if (lane == 0) record_status(status, ELASTO_ERR_TIMEOUT);
        break;
      }
      tc_fence_after();
      // pass 1: row max over the valid keys
      float mx = -INFINITY;
      for (int c = 0; c < n_pad; c += 16) {
        uint32_t v[16];
        tmem_ld_16(lane_base + c, v);
        tmem_ld_wait();
#pragma unroll
        for (int j = 0; j < 16; ++j)
          if (c + j < n) mx = fmaxf(mx, __uint_as_float(v[j]));
      }
      // pass 2: numerators, row sum, P (bf16, swizzled K-major rows)
      float sum = 0.0f;
      const float mxs = mx * kscale;
      uint8_t* prow = sP + r * 128;
      for (int c = 0; c < n_pad; c += 16) {
        uint32_t v[16];
        tmem_ld_16(lane_base + c, v);
        tmem_ld_wait();
        uint32_t pk[8];
#pragma unroll
        for (int j = 0; j < 16; j += 2) {
          const float p0 = (c + j < n) ? exp2f(fmaf(__uint_as_float(v[j]), kscale, -mxs)) : 0.0f;
          const float p1 = (c + j + 1 < n) ? exp2f(fmaf(__uint_as_float(v[j + 1]), kscale, -mxs)) : 0.0f;
          sum += p0 + p1;
          pk[j >> 1] = pack_bf16x2(p0, p1);
        }
        const int atom = c >> 6;
        const int chunk = (c & 63) >> 3;  // 16-byte chunk index within the 128-byte row
        uint8_t* base = prow + atom * P_ATOM;
        *reinterpret_cast<uint4*>(base + ((chunk ^ (r & 7)) << 4)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
        *reinterpret_cast<uint4*>(base + (((chunk + 1) ^ (r & 7)) << 4)) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
      }
      fence_async_smem();
      tc_fence_before();
      mbar_arrive(bar_p);
      // epilogue
      if (!mbar_wait(bar_o, ph)) {
        if (lane == 0) record_status(status, ELASTO_ERR_TIMEOUT);
        break;
      }
      tc_fence_after();
      const float inv = 1.0f / sum;
      const int i = qt * QT + r;
      uint32_t o[32];
      uint4 pk4[8];
      tmem_ld_32x32b_x32(lane_base, o);
      tmem_ld_wait();
#pragma unroll
      for (int j = 0; j < 4; ++j)
        pk4[j] = make_uint4(pack_bf16x2(__uint_as_float(o[8 * j + 0]) * inv, __uint_as_float(o[8 * j + 1]) * inv),
                            pack_bf16x2(__uint_as_float(o[8 * j + 2]) * inv, __uint_as_float(o[8 * j + 3]) * inv),
                            pack_bf16x2(__uint_as_float(o[8 * j + 4]) * inv, __uint_as_float(o[8 * j + 5]) * inv),
                            pack_bf16x2(__uint_as_float(o[8 * j + 6]) * inv, __uint_as_float(o[8 * j + 7]) * inv));
      tmem_ld_32x32b_x32(lane_base + 32, o);
      tmem_ld_wait();
#pragma unroll
      for (int j = 0; j < 4; ++j)
        pk4[4 + j] =
            make_uint4(pack_bf16x2(__uint_as_float(o[8 * j + 0]) * inv, __uint_as_float(o[8 * j + 1]) * inv),
                       pack_bf16x2(__uint_as_float(o[8 * j + 2]) * inv, __uint_as_float(o[8 * j + 3]) * inv),
                       pack_bf16x2(__uint_as_float(o[8 * j + 4]) * inv, __uint_as_float(o[8 * j + 5]) * inv),
                       pack_bf16x2(__uint_as_float(o[8 * j + 6]) * inv, __uint_as_float(o[8 * j + 7]) * inv));
      tc_fence_before();
      mbar_arrive(bar_e);
      if (i < n) {
        uint4* dst = reinterpret_cast<uint4*>(out + (static_cast<size_t>(b) * n + i) * w + jj * HD);
#pragma unroll
        for (int j = 0; j < 8; ++j) dst[j] = pk4[j];
      }
    }
  }
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

}  // namespace

cudaError_t attn_init_attributes() {
  return cudaFuncSetAttribute(attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(SMEM_BYTES));
}

elasto_status attn_plan(AttnPlan* p, const bf16* qkv, bf16* out, int batch_cap, int n, int heads, int* status) {
  if (!p || !qkv || !out || batch_cap <= 0 || n <= 0 || heads <= 0) {
    set_error("attention: invalid arguments");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (n > MAXK) {
    set_error("attention: at most 256 tokens are supported");
    return ELASTO_ERR_UNSUPPORTED;
  }
  *p = AttnPlan{};
  p->qkv = qkv;
  p->out = out;
  p->n = n;
  p->n_pad = (n + 15) / 16 * 16;
  p->heads = heads;
  p->batch_cap = batch_cap;
  p->status = status;
  const uint64_t cols = static_cast<uint64_t>(3) * heads * HD;
  if (!encode_tmap_3d(&p->tmQ, qkv, cols, n, batch_cap, cols * 2, cols * 2 * n, HD, QT, 1) ||
      !encode_tmap_3d(&p->tmKV, qkv, cols, n, batch_cap, cols * 2, cols * 2 * n, HD, p->n_pad, 1)) {
    set_error("attention: cuTensorMapEncodeTiled failed");
    return ELASTO_ERR_UNSUPPORTED;
  }
  p->valid = true;
  return ELASTO_OK;
}

cudaError_t attn_launch(const AttnPlan& p, int batch, cudaStream_t s) {
  if (batch <= 0) return cudaSuccess;
  dim3 grid(p.heads, batch);
  attn_tc_kernel<<<grid, THREADS, SMEM_BYTES, s>>>(p.tmQ, p.tmKV, p.out, p.n, p.n_pad, p.heads, p.status);
  return cudaGetLastError();
}

}  // namespace elasto
