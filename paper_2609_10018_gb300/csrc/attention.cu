// Fused multi-head attention over the kept heads only (Eq. 2-3 restricted to
// the DN's head set H; heads outside H were removed from W^Q, W^K, W^V at
// pack time, so this kernel never sees them).
//
// Input: qkv [B, n, 3, h_m, 64] bf16 exactly as the QKV GEMM writes it (q | k |
// v blocks, kept heads in packing order), or [B, n, h_m, 3, 64] when the modes
// share one prefix-ordered packed copy (each head's q, k, v adjacent, so a
// prefix of heads is a prefix of columns). Output: [B, n, h_m * 64] bf16, the
// heads concatenated in the same order (the K axis of the packed W^O).
//
// Persistent kernel; a work item is one (image, kept head) and needs at most
// two 128-query tiles (n <= 256). Items run from the last image to the first:
// the QKV GEMM wrote its rows in increasing order, so the most recent (still
// in L2) are read first. Roles:
//   warp 0      TMA producer: K and V of an item into one of `kv_slots`
//               shared-memory slots, its query tiles into one of two Q
//               buffers per tile (3-D maps: rows past n read as zero);
//   warp 1      tcgen05.mma issuer: S_t = Q_t K^T (M=128, N=n_pad, K=64) into
//               the 256-column TMEM region of query tile t, then O_t = P_t V
//               with P_t read from TMEM (M=128, N=64, K=n_pad; V MN-major);
//   warps 2-9   two groups of four, one per query tile: one query row per
//               thread (TMEM lane = row). Row max and exp2 numerators over the
//               n valid keys in fp32; P_t stored back into TMEM as bf16 pairs
//               over the S columns already consumed; then O row * (1 / row
//               sum) -> bf16, 128 contiguous bytes per thread. Warps whose 32
//               rows are all padding (past n) skip the TMEM work.
// The two query tiles run half an item apart: the issue order is
//   S(0,0); then per item k: S(k,1), PV(k,0), S(k+1,0), PV(k,1)
// so the tensor pipe computes one tile's MMAs while the other tile's group
// runs its softmax (both softmaxes at once would share the exp units while
// the tensor pipe idles). An item's K/V slot is released after PV(k,1), its
// Q buffers after S(k,1).
// TMEM per tile region: S in [0, n_pad), P in [0, n_pad / 2), O in [128, 192)
// (O overwrites S columns the softmax has consumed, so S(k+1,t) waits until
// O(k,t) is read out).
// Scale 1/sqrt(64) (the base model's head width; it does not change with the
// number of kept heads). Every mbarrier wait is bounded.
#include "common.h"
#include "ptx.cuh"

namespace elasto {

namespace {

constexpr int THREADS = 320;
constexpr int HD = 64;                      // head width d_i
constexpr int QT = 128;                     // queries per tile
constexpr int MAXK = 256;                   // max keys
constexpr int Q_BYTES = QT * HD * 2;        // 16 KB
constexpr int QBUF_BYTES = 4 * Q_BYTES;     // two buffers per query tile
constexpr int BAR_BYTES = 256;
constexpr int SMEM_LIMIT = 232448;          // dynamic shared memory per block on sm_103
constexpr int TMEM_COLS = 512;
constexpr int O_COL = 128;

// Shared memory: [Q buffers][KV slots][barriers], 1024-byte aligned.
__host__ __device__ constexpr int kv_slot_bytes(int n_pad) { return 2 * n_pad * HD * 2; }
__host__ __device__ constexpr int kv_slots_for(int n_pad) {
  return 1024 + QBUF_BYTES + 3 * kv_slot_bytes(n_pad) + BAR_BYTES <= SMEM_LIMIT ? 3 : 2;
}
__host__ __device__ constexpr int smem_bytes_for(int n_pad) {
  return 1024 + QBUF_BYTES + kv_slots_for(n_pad) * kv_slot_bytes(n_pad) + BAR_BYTES;
}
__host__ __device__ constexpr int max_smem_bytes() {
  int m = 0;
  for (int n_pad = 16; n_pad <= MAXK; n_pad += 16) m = smem_bytes_for(n_pad) > m ? smem_bytes_for(n_pad) : m;
  return m;
}
static_assert(max_smem_bytes() <= SMEM_LIMIT, "attention shared memory");

__global__ void __launch_bounds__(THREADS, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmKV,
                   bf16* __restrict__ out, int n, int n_pad, int heads, int items, int blk_stride,
                   int head_stride, int* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int ns = kv_slots_for(n_pad);
  const int slot_bytes = kv_slot_bytes(n_pad);
  uint8_t* qbuf = smem;                                    // [tile][parity] Q_BYTES each
  uint8_t* kvbuf = smem + QBUF_BYTES;                      // [slot] K then V, n_pad rows of 128 B
  uint64_t* bars = reinterpret_cast<uint64_t*>(kvbuf + ns * slot_bytes);
  uint64_t* full = bars + 0;        // [3] item k's Q, K, V landed (slot k % ns)
  uint64_t* kv_empty = bars + 3;    // [3] slot's PV MMAs finished
  uint64_t* q_empty = bars + 6;     // [2] Q buffers of parity k & 1 consumed by S(k, *)
  uint64_t* s_full = bars + 8;      // [2] S_t in TMEM
  uint64_t* p_full = bars + 10;     // [2] P_t in TMEM (128 arrivals)
  uint64_t* o_full = bars + 12;     // [2] O_t in TMEM
  uint64_t* o_empty = bars + 14;    // [2] O_t read out (128 arrivals)
  uint64_t* drain = bars + 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 17);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int w = heads * HD;
  const int tiles = n > QT ? 2 : 1;
  // items of this CTA: blockIdx.x, blockIdx.x + gridDim.x, ...
  const int nk = items > static_cast<int>(blockIdx.x) ? (items - 1 - blockIdx.x) / gridDim.x + 1 : 0;

  if (threadIdx.x == 0) {
    for (int k = 0; k < 3; ++k) {
      mbar_init(&full[k], 1);
      mbar_init(&kv_empty[k], 1);
    }
    for (int k = 0; k < 2; ++k) {
      mbar_init(&q_empty[k], 1);
      mbar_init(&s_full[k], 1);
      mbar_init(&p_full[k], 128);
      mbar_init(&o_full[k], 1);
      mbar_init(&o_empty[k], 128);
    }
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
  pdl_wait();  // the set-up above overlapped the previous kernel's tail
  pdl_trigger();

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmKV);
      const uint32_t bytes = tiles * Q_BYTES + 2 * n_pad * HD * 2;
      bool ok = true;
      int k = 0;
      for (; k < nk; ++k) {
        const int item = blockIdx.x + k * gridDim.x;
        const int slot = k % ns, b = (items - 1 - item) / heads, jj = (items - 1 - item) - b * heads;
        if (!mbar_wait(&kv_empty[slot], ((k / ns) & 1) ^ 1) || !mbar_wait(&q_empty[k & 1], ((k >> 1) & 1) ^ 1)) {
          ok = false;
          break;
        }
        uint8_t* kb = kvbuf + slot * slot_bytes;
        mbar_expect_tx(&full[slot], bytes);
        const int qx = jj * head_stride;
        tma_load_3d(kb, &tmKV, &full[slot], qx + blk_stride, 0, b);
        tma_load_3d(kb + slot_bytes / 2, &tmKV, &full[slot], qx + 2 * blk_stride, 0, b);
        for (int t = 0; t < tiles; ++t)
          tma_load_3d(qbuf + (2 * t + (k & 1)) * Q_BYTES, &tmQ, &full[slot], qx, t * QT, b);
      }
      if (!ok) record_status(status, ELASTO_ERR_TIMEOUT);
      // the loads of the last items have landed before the CTA exits
      for (int j = (k > ns ? k - ns : 0); j < k; ++j) mbar_wait(&full[j % ns], (j / ns) & 1);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && nk > 0) {
      const uint32_t idesc_s = idesc_bf16_f32(QT, n_pad);
      const uint32_t idesc_o = idesc_bf16_f32(QT, HD, false, true);
      bool ok = true;
      // S(k, t): needs item k landed (waited once, at t = 0) and O(k-1, t)
      // read out (S overwrites the O columns of its tile region)
      auto issue_s = [&](int k, int t) -> bool {
        const int slot = k % ns;
        if (t == 0 && !mbar_wait(&full[slot], (k / ns) & 1)) return false;
        if (!mbar_wait(&o_empty[t], (k & 1) ^ 1)) return false;
        tc_fence_after();
        const uint32_t q0 = smem_addr(qbuf + (2 * t + (k & 1)) * Q_BYTES);
        const uint32_t k0 = smem_addr(kvbuf + slot * slot_bytes);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          tc_mma(tmem + t * 256, sdesc_sw128(q0 + kk * 32, 16, 1024), sdesc_sw128(k0 + kk * 32, 16, 1024), idesc_s,
                 kk != 0);
        tc_commit(&s_full[t]);
        if (t == tiles - 1) tc_commit(&q_empty[k & 1]);
        return true;
      };
      // PV(k, t): needs P(k, t) in TMEM
      auto issue_pv = [&](int k, int t) -> bool {
        if (!mbar_wait(&p_full[t], k & 1)) return false;
        tc_fence_after();
        const uint32_t v0 = smem_addr(kvbuf + (k % ns) * slot_bytes + slot_bytes / 2);
        for (int s = 0; s < n_pad / 16; ++s)
          tc_mma_tmem_a(tmem + t * 256 + O_COL, tmem + t * 256 + 8 * s, sdesc_sw128(v0 + s * 16 * 128, 16384, 1024),
                        idesc_o, s != 0);
        tc_commit(&o_full[t]);
        if (t == tiles - 1) tc_commit(&kv_empty[k % ns]);
        return true;
      };
      ok = issue_s(0, 0);
      const bool issued = ok;
      for (int k = 0; k < nk && ok; ++k) {
        if (tiles == 2) ok = issue_s(k, 1);
        if (ok) ok = issue_pv(k, 0);
        if (ok && k + 1 < nk) ok = issue_s(k + 1, 0);
        if (ok && tiles == 2) ok = issue_pv(k, 1);
      }
      if (!ok) record_status(status, ELASTO_ERR_TIMEOUT);
      if (issued) {  // every MMA this thread issued has finished once `drain` completes
        tc_commit(drain);
        mbar_wait(drain, 0);
      }
    }
  } else {
    // ------------------------------------------------------------ softmax + epilogue
    const int t = (warp - 2) >> 2;           // query tile of this group
    const int qq = warp & 3;                 // TMEM lane quarter
    const int r = qq * 32 + lane;            // row within the query tile
    // a warp whose 32 rows are all past n has no softmax or read-out work
    const bool active = t * QT + qq * 32 < n;
    if (t < tiles) {
      const uint32_t lane_base = tmem + (static_cast<uint32_t>(qq * 32) << 16) + t * 256;
      const float kscale = 0.125f * 1.4426950408889634f;  // 1/sqrt(64) * log2(e)
      const int n_read = (n + 63) & ~63;                  // columns read in 64-column steps
      for (int k = 0; k < nk; ++k) {
        const int item = blockIdx.x + k * gridDim.x;
        const uint32_t ph = k & 1;
        const int b = (items - 1 - item) / heads, jj = (items - 1 - item) - b * heads;
        if (!mbar_wait(&s_full[t], ph)) {
          if (lane == 0) record_status(status, ELASTO_ERR_TIMEOUT);
          break;
        }
        tc_fence_after();
        float sum = 1.0f;
        if (active) {
          // pass 1: row max over the valid keys (four independent partial maxima)
          float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
          for (int c = 0; c < n_read; c += 64) {
            uint32_t v[32], u[32];
            tmem_ld_32x32b_x32(lane_base + c, v);
            tmem_ld_32x32b_x32(lane_base + c + 32, u);
            tmem_ld_wait();
            if (c + 64 <= n) {
#pragma unroll
              for (int j = 0; j < 32; ++j) {
                m4[j & 3] = fmaxf(m4[j & 3], __uint_as_float(v[j]));
                m4[j & 3] = fmaxf(m4[j & 3], __uint_as_float(u[j]));
              }
            } else {
#pragma unroll
              for (int j = 0; j < 32; ++j) {
                if (c + j < n) m4[j & 3] = fmaxf(m4[j & 3], __uint_as_float(v[j]));
                if (c + 32 + j < n) m4[j & 3] = fmaxf(m4[j & 3], __uint_as_float(u[j]));
              }
            }
          }
          const float mx = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
          // pass 2: numerators and row sum; P as bf16 pairs into TMEM columns
          // [c/2, c/2 + 32), all of which this pass has already read
          const float mxs = mx * kscale;
          float s4[4] = {0.0f, 0.0f, 0.0f, 0.0f};
          for (int c = 0; c < n_read; c += 64) {
            uint32_t v[64], pk[32];
            tmem_ld_32x32b_x32(lane_base + c, *reinterpret_cast<uint32_t(*)[32]>(v));
            tmem_ld_32x32b_x32(lane_base + c + 32, *reinterpret_cast<uint32_t(*)[32]>(v + 32));
            tmem_ld_wait();
            if (c + 64 <= n) {
#pragma unroll
              for (int j = 0; j < 64; j += 2) {
                const float p0 = ex2_approx(fmaf(__uint_as_float(v[j]), kscale, -mxs));
                const float p1 = ex2_approx(fmaf(__uint_as_float(v[j + 1]), kscale, -mxs));
                s4[(j >> 1) & 3] += p0 + p1;
                pk[j >> 1] = pack_bf16x2(p0, p1);
              }
            } else {
#pragma unroll
              for (int j = 0; j < 64; j += 2) {
                const float p0 = (c + j < n) ? ex2_approx(fmaf(__uint_as_float(v[j]), kscale, -mxs)) : 0.0f;
                const float p1 = (c + j + 1 < n) ? ex2_approx(fmaf(__uint_as_float(v[j + 1]), kscale, -mxs)) : 0.0f;
                s4[(j >> 1) & 3] += p0 + p1;
                pk[j >> 1] = pack_bf16x2(p0, p1);
              }
            }
            tmem_st_16(lane_base + (c >> 1), *reinterpret_cast<const uint32_t(*)[16]>(pk));
            tmem_st_16(lane_base + (c >> 1) + 16, *reinterpret_cast<const uint32_t(*)[16]>(pk + 16));
          }
          sum = (s4[0] + s4[1]) + (s4[2] + s4[3]);
          tmem_st_wait();
        }
        tc_fence_before();
        mbar_arrive(&p_full[t]);
        // epilogue
        if (!mbar_wait(&o_full[t], ph)) {
          if (lane == 0) record_status(status, ELASTO_ERR_TIMEOUT);
          break;
        }
        tc_fence_after();
        uint32_t o[64];
        if (active) {
          tmem_ld_32x32b_x32(lane_base + O_COL, *reinterpret_cast<uint32_t(*)[32]>(o));
          tmem_ld_32x32b_x32(lane_base + O_COL + 32, *reinterpret_cast<uint32_t(*)[32]>(o + 32));
          tmem_ld_wait();
        }
        tc_fence_before();
        mbar_arrive(&o_empty[t]);
        const int row = t * QT + r;
        if (active && row < n) {
          const float inv = 1.0f / sum;
          uint4* dst = reinterpret_cast<uint4*>(out + (static_cast<size_t>(b) * n + row) * w + jj * HD);
#pragma unroll
          for (int j = 0; j < 8; ++j)
            dst[j] = make_uint4(pack_bf16x2(__uint_as_float(o[8 * j + 0]) * inv, __uint_as_float(o[8 * j + 1]) * inv),
                                pack_bf16x2(__uint_as_float(o[8 * j + 2]) * inv, __uint_as_float(o[8 * j + 3]) * inv),
                                pack_bf16x2(__uint_as_float(o[8 * j + 4]) * inv, __uint_as_float(o[8 * j + 5]) * inv),
                                pack_bf16x2(__uint_as_float(o[8 * j + 6]) * inv, __uint_as_float(o[8 * j + 7]) * inv));
        }
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
  return cudaFuncSetAttribute(attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, max_smem_bytes());
}

elasto_status attn_plan(AttnPlan* p, const bf16* qkv, bf16* out, int batch_cap, int n, int heads, int* status,
                        bool interleaved) {
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
  p->blk_stride = interleaved ? HD : heads * HD;
  p->head_stride = interleaved ? 3 * HD : HD;
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
  const int items = batch * p.heads;
  const int grid = items < num_sms() ? items : num_sms();
  return launch_pdl(attn_tc_kernel, dim3(grid), dim3(THREADS), smem_bytes_for(p.n_pad), s, p.tmQ, p.tmKV, p.out, p.n,
                    p.n_pad,
                    p.heads, items, p.blk_stride, p.head_stride, p.status);
}

}  // namespace elasto
