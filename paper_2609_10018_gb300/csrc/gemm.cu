// Tensor-core GEMM with fused epilogues: out = epi(A[M,K] . W[N,K]^T).
//
// This is every dense contraction of the DN forward (Section 4.1): the patch
// projection, the sliced QKV projection of the kept heads (Eq. 2, 4), the
// sliced output projection W^O (Eq. 2, 4) and the sliced MLP W1 / W2
// (Eq. 5, 6). Slicing happened at create time, so here the kept widths are
// just the problem's N or K.
//
// Design (sm_103a):
//  - persistent grid, one CTA per SM (or one CTA pair per two SMs), static
//    round-robin over 128 x bn tiles (N tile index fastest so the CTAs
//    running together share A rows in L2; m_reverse runs the rows backwards);
//  - warp 0 lane 0: TMA producer, ring of 128x64 (A) and bn x 64 (B) bf16 or
//    f16 tiles with the 128-byte swizzle, one mbarrier pair per stage. W may
//    instead be loaded once per CTA and kept (b_resident: one N tile);
//  - warp 1 lane 0: issues tcgen05.mma (M=128, N=bn, K=16) into one of two
//    TMEM accumulators (2 x 256 fp32 columns), commits stages back to the
//    producer and finished accumulators to the epilogue. K >= 1536 on
//    256-row tiles: CTA pairs (cta_group::2, M = 256, each CTA holds half of
//    B);
//  - warps 2-17: epilogue, four warps per 32-lane quarter of TMEM (= 32 rows
//    of the tile), each taking a quarter of every 64-column chunk.
//    * bf16 outputs (QKV, FC1+GELU, conv+ReLU) and the fp32 residual stream
//      (out-proj, FC2): each thread writes its row piece of a 128-row x
//      128-byte chunk into a 128B-swizzled staging buffer in shared memory
//      (bank conflict free 16-byte stores) and one thread stores the chunk
//      with a TMA tensor store. For the residual, the old rows of X are
//      brought into the same staging buffer by TMA loads issued several
//      chunks ahead, so the read-modify-write of X runs at full memory
//      parallelism. The 16-bit residual + ReLU of the CNN block outputs works
//      the same way.
//    * the remaining epilogue (fp32 out) transposes through padded shared
//      memory for row-contiguous stores (warps 2-5); it also writes the
//      partial sums of a split-K plan, whose k-block range is
//      tile / (mt * nt).
//  - implicit-GEMM convolution: A tiles are 4-D TMA boxes of the NHWC input
//    (one tap and channel group per k-block, padding read as zeros), and the
//    output is stored by 4-D boxes of the tile's pixel block.
//  Every mbarrier wait is bounded; a timeout records ELASTO_ERR_TIMEOUT.
#include <algorithm>

#include "act.cuh"
#include "common.h"
#include "ptx.cuh"

namespace elasto {

namespace {

constexpr int BM = 128, BK = 64, MAX_STAGES = 8, MAX_BN = 256;
constexpr int EPI_THREADS = 512;                 // 16 epilogue warps, four per TMEM lane quarter
constexpr int THREADS = 64 + EPI_THREADS;
constexpr int THREADS_CONV = THREADS + 32;  // implicit convolutions: warp 18 is a second TMA producer
constexpr int A_STAGE = BM * BK * 2;        // 16 KB
constexpr int CBUF = BM * 128;              // 16 KB staging chunk (128 rows x 128 B)
constexpr int POOL = 224 * 1024;            // operand ring + staging buffers
constexpr int MAX_CBUFS = 8;
constexpr int EPI_LD = 33;                  // padded row of the transpose tile
constexpr int EPI_TILE = 32 * EPI_LD;       // floats per epilogue warp
constexpr int TMEM_COLS = 512;
constexpr size_t SMEM_BYTES = 1024 + POOL + 512;

template <int EPI>
struct EpiTraits {
  static constexpr bool half = EPI == EPI_BIAS_RELU_F16 || EPI == EPI_BIAS_F16 || EPI == EPI_BIAS_RESID_RELU_F16;
  // 16-bit residual + ReLU (block outputs of the CNN): the residual chunk is
  // brought into the staging buffer by TMA like the fp32 residual stream
  static constexpr bool resid16 = EPI == EPI_BIAS_RESID_RELU_BF16 || EPI == EPI_BIAS_RESID_RELU_F16;
  static constexpr bool tma = EPI == EPI_BIAS_BF16 || EPI == EPI_BIAS_GELU_BF16 || EPI == EPI_BIAS_RELU_BF16 ||
                              EPI == EPI_BIAS_RESID_F32 || EPI == EPI_BIAS_RELU_F16 || EPI == EPI_BIAS_F16 ||
                              resid16;
  static constexpr bool f32 = EPI == EPI_BIAS_RESID_F32;
  static constexpr bool resid = EPI == EPI_BIAS_RESID_F32 || resid16;
  static constexpr int cw = f32 ? 32 : 64;  // columns per 128-byte staging chunk
};

// M-tile of the q-th tile row in the schedule: q, or mt - 1 - q when the plan
// runs its rows last to first (m_reverse: the GEMM then reads first the rows
// of its A operand that the previous kernel wrote last, still in L2).
__device__ __forceinline__ int m_tile(const GemmArgs& a, int q, int mt) { return a.m_reverse ? mt - 1 - q : q; }

// Row of the residual source that a tile starting at output row m0 reads: the
// same row, or for a periodic source (resid_row_mod rows per period, stored
// for enough periods that any 128 consecutive rows from a start below the
// period are present) the row m0 mod period.
__device__ __forceinline__ int resid_row(const GemmArgs& a, int m0) {
  return a.resid_row_mod > 0 ? m0 % a.resid_row_mod : m0;
}

template <int EPI>
__device__ __forceinline__ float epi_act(float v) {
  if constexpr (EPI == EPI_BIAS_GELU_BF16) return gelu(v);
  if constexpr (EPI == EPI_BIAS_RELU_BF16 || EPI == EPI_BIAS_RELU_F16 || EpiTraits<EPI>::resid16)
    return fmaxf(v, 0.0f);
  return v;
}

// One 32-bit word of the epilogue's 16-bit type -> two fp32 values.
template <int EPI>
__device__ __forceinline__ float2 unpack_in(uint32_t w) {
  if constexpr (EpiTraits<EPI>::half)
    return __half22float2(*reinterpret_cast<const __half2*>(&w));
  else
    return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}

// Two fp32 values -> one 32-bit word of the epilogue's 16-bit output type.
template <int EPI>
__device__ __forceinline__ uint32_t pack_out(float lo, float hi) {
  if constexpr (EpiTraits<EPI>::half)
    return pack_f16x2(lo, hi);
  else
    return pack_bf16x2(lo, hi);
}

// W consecutive bias values starting at column col (zero past N or if null).
template <int W>
__device__ __forceinline__ void load_bias(const float* bias, int col, int N, float (&b)[W]) {
  if (bias && col + W <= N) {
    const float4* p = reinterpret_cast<const float4*>(bias + col);
#pragma unroll
    for (int j = 0; j < W / 4; ++j) {
      const float4 v = __ldg(p + j);
      b[4 * j] = v.x;
      b[4 * j + 1] = v.y;
      b[4 * j + 2] = v.z;
      b[4 * j + 3] = v.w;
    }
  } else {
#pragma unroll
    for (int j = 0; j < W; ++j) b[j] = (bias && col + j < N) ? __ldg(bias + col + j) : 0.0f;
  }
}

// Implicit-GEMM convolution: number of M tiles and the pixel block of one.
__host__ __device__ __forceinline__ int conv_mtiles(const GemmArgs& a) {
  return ((a.cv_wo + a.cv_bw - 1) / a.cv_bw) * ((a.cv_ho + a.cv_bh - 1) / a.cv_bh) *
         ((a.cv_batch + a.cv_nb - 1) / a.cv_nb);
}
__device__ __forceinline__ void conv_tile(const GemmArgs& a, int mtile, int& b0, int& oy0, int& ox0) {
  const int tx = (a.cv_wo + a.cv_bw - 1) / a.cv_bw, ty = (a.cv_ho + a.cv_bh - 1) / a.cv_bh;
  const int r = mtile / tx;
  ox0 = (mtile - r * tx) * a.cv_bw;
  oy0 = (r % ty) * a.cv_bh;
  b0 = (r / ty) * a.cv_nb;
}

// Walks this CTA's sequence of (tile, chunk) pairs, skipping chunks past N.
struct ChunkIter {
  int t, c;
  bool valid;
  int stride;
  __device__ __forceinline__ void init(int tiles, int start, int step) {
    t = start;
    stride = step;
    c = 0;
    valid = t < tiles;
  }
  __device__ __forceinline__ void advance(int tiles, int nt, int bn, int cw, int N) {
    const int n0 = (t % nt) * bn;
    ++c;
    if (c * cw >= bn || n0 + c * cw >= N) {
      c = 0;
      t += stride;
      valid = t < tiles;
    }
  }
};

// PAIR: the kernel runs as clusters of two CTAs on neighbouring SMs that
// share 256-row tiles: each CTA loads its 128 rows of A and half of the B
// tile; the even CTA issues tcgen05.mma.cta_group::2 (M = 256) for both and
// signals both CTAs' barriers with multicast commits; each CTA's epilogue
// reads its own half of the accumulator from its own TMEM.
template <int EPI, int NB, bool PAIR>
__global__ void __launch_bounds__(THREADS_CONV, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmB2,
                   const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmR,
                   const GemmArgs args) {
  using TR = EpiTraits<EPI>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int S = args.stages, E = args.cbufs;
  // NB: 1, or 2 when W is held as a bf16 (hi, lo) pair
  const int BSTG = args.b_stage;  // NB planes of bn rows (bn / 2 rows per CTA of a pair)
  const bool bres = !PAIR && NB == 1 && args.b_resident;
  uint8_t* sA = smem;
  uint8_t* sB = smem + S * A_STAGE;  // the B ring, or (bres) every k-block of B
  const int bke = args.k16 ? 16 : BK;  // K values per k-block
  const int nk = (args.K + bke - 1) / bke;
  uint8_t* sC = sB + (bres ? nk : S) * BSTG;  // E staging chunks, or the transpose tiles
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + POOL);
  uint64_t* full = bars;
  uint64_t* empty = bars + MAX_STAGES;
  uint64_t* tfull = bars + 2 * MAX_STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint64_t* rfull = drain + 1;  // MAX_CBUFS residual-landed barriers
  uint64_t* bfull = rfull + MAX_CBUFS;  // resident B landed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bfull + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int M = args.M, N = args.N, bn = args.bn;
  constexpr int TM = PAIR ? 2 * BM : BM;  // rows per tile
  const int mt = args.conv ? conv_mtiles(args) : (M + TM - 1) / TM, nt = (N + bn - 1) / bn;
  // split-K (fp32 partial outputs only): tile t covers output tile
  // t % (mt * nt) and k-block range t / (mt * nt) of ks. Every other
  // epilogue has ks = 1 at compile time and no division on its tile path.
  constexpr bool kSplit = EPI == EPI_BIAS_F32;
  const int ks = kSplit && args.ksplit > 1 ? args.ksplit : 1;
  const int mn_tiles = mt * nt;
  const int tiles = mn_tiles * ks;
  const int rank = PAIR ? static_cast<int>(cluster_ctarank()) : 0;  // this CTA's row half of a pair tile
  const int t_start = PAIR ? static_cast<int>(cluster_id_x()) : static_cast<int>(blockIdx.x);
  const int t_stride = PAIR ? static_cast<int>(cluster_count_x()) : static_cast<int>(gridDim.x);
  const bool leader = rank == 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < MAX_STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], (PAIR ? 2 : 1) * (TR::tma ? EPI_THREADS / 32 : 4));
    }
    mbar_init(drain, 1);
    for (int e = 0; e < MAX_CBUFS; ++e) mbar_init(&rfull[e], 1);
    mbar_init(bfull, 1);
    tmem_slot[1] = 0;  // the epilogue's fail flag
    fence_barrier_init();
  }
  if (warp == 0) {
    if constexpr (PAIR) {
      tmem_alloc_pair(tmem_slot, TMEM_COLS);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(tmem_slot, TMEM_COLS);
      tmem_relinquish();
    }
  }
  if (warp == 1 && lane == 0) {
    if (nk > 0) {
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmB);
      if constexpr (NB == 2) tma_prefetch_desc(&tmB2);
    }
    if constexpr (TR::tma) tma_prefetch_desc(&tmC);
    if constexpr (TR::resid) tma_prefetch_desc(&tmR);
  }
  tc_fence_before();
  if constexpr (PAIR)
    cluster_sync_all();  // both CTAs' barriers initialised before any remote arrive
  else
    __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // Everything above overlapped the previous kernel's tail. Every thread
  // waits for that kernel (pdl_wait) before its first access to data it may
  // write; the weights are not such data, so the producer thread starts
  // loading them first and waits after that.
  if (!(warp == 0 && lane == 0 && nk > 0)) {
    pdl_wait();
    pdl_trigger();
  }

  // Implicit convolutions run two producer threads (warp 0 and warp 18,
  // lane 0 of each) that take alternate k-blocks: issuing one 4-D box load
  // occupies its warp for ~0.26 us, longer than the tensor core spends on a
  // narrow k-block.
  const int nprod = (!PAIR && args.conv && static_cast<int>(blockDim.x) == THREADS_CONV) ? 2 : 1;
  if (warp == 0 || warp == THREADS / 32) {
    // ------------------------------------------------------------ producer
    const int pid = warp == 0 ? 0 : 1;
    if (lane == 0 && pid < nprod && nk > 0) {
      int stage = 0;
      uint32_t phase = 0;
      long seq = 0;         // k-block sequence index over this CTA's tiles
      long last_mine = -1;  // the last k-block this thread issued
      bool ok = true;
      // pair: the even CTA's full barrier counts both CTAs' bytes
      const uint32_t bytes = PAIR ? 2 * (A_STAGE + (bn / 2) * BK * 2)
                                  : (args.conv ? args.cv_a_bytes : A_STAGE) + (bres ? 0 : NB * bn * bke * 2);
      const bool b_loaded = bres && t_start < tiles && pid == 0;
      if (b_loaded) {  // all of W, once: nk k-blocks of the single N tile
        mbar_expect_tx(bfull, static_cast<uint32_t>(nk) * bn * bke * 2);
        for (int kb = 0; kb < nk; ++kb) tma_load_2d(sB + kb * BSTG, &tmB, bfull, kb * bke, 0);
      }
      // the first tile's first S stages: armed and their weights requested
      // before the wait (fresh stages: no empty-slot wait needed); thread 0
      // issues these k-blocks
      int pre = 0;
      if (!PAIR && !bres && t_start < tiles) {
        const int tq = kSplit ? t_start % mn_tiles : t_start;
        const int kb0 = kSplit ? (t_start / mn_tiles) * nk / ks : 0;
        const int kb1 = kSplit ? (t_start / mn_tiles + 1) * nk / ks : nk;
        const int n0 = (tq % nt) * bn;
        pre = kb1 - kb0 < S ? kb1 - kb0 : S;
        if (pid == 0)
          for (int i = 0; i < pre; ++i) {
            mbar_expect_tx(&full[i], bytes);
            tma_load_2d(sB + i * BSTG, &tmB, &full[i], (kb0 + i) * bke, n0);
            if constexpr (NB == 2) tma_load_2d(sB + i * BSTG + BSTG / 2, &tmB2, &full[i], (kb0 + i) * BK, n0);
          }
      }
      auto mine = [&](long q) { return nprod == 1 || (q < pre ? pid == 0 : static_cast<int>(q & 1) == pid); };
      pdl_wait();
      pdl_trigger();
      for (int t = t_start; t < tiles && ok; t += t_stride) {
        const int tq = kSplit ? t % mn_tiles : t;
        const int kb0 = kSplit ? (t / mn_tiles) * nk / ks : 0, kb1 = kSplit ? (t / mn_tiles + 1) * nk / ks : nk;
        const int m0 = m_tile(args, tq / nt, mt) * TM + rank * BM, n0 = (tq % nt) * bn;
        int cb0 = 0, cy0 = 0, cx0 = 0;  // implicit conv: first image, output row and column of the tile
        int cg = 0, kx = 0, ky = 0;     // implicit conv: the k-block's channel group and tap, advanced in step
        if (args.conv) {
          conv_tile(args, m_tile(args, tq / nt, mt), cb0, cy0, cx0);
          const int tap = kb0 / args.cv_cgroups;
          cg = kb0 - tap * args.cv_cgroups;
          ky = tap / args.cv_ks;
          kx = tap - ky * args.cv_ks;
        }
        for (int kb = kb0; kb < kb1; ++kb, ++seq) {
          if (mine(seq)) {
            if (!(PAIR ? mbar_wait_cluster(&empty[stage], phase ^ 1) : mbar_wait(&empty[stage], phase ^ 1))) {
              ok = false;
              break;
            }
            if constexpr (PAIR) {
              const uint32_t full_lead = cluster_map(smem_addr(&full[stage]), 0);
              if (leader) mbar_expect_tx(&full[stage], bytes);
              tma_load_2d_pair(sA + stage * A_STAGE, &tmA, full_lead, kb * BK, m0);
              tma_load_2d_pair(sB + stage * BSTG, &tmB, full_lead, kb * BK, n0 + rank * (bn / 2));
            } else {
              const bool armed = seq < pre;  // this stage's weights were requested before the wait
              if (!armed) mbar_expect_tx(&full[stage], bytes);
              if (args.conv) {
                tma_load_4d(sA + stage * A_STAGE, &tmA, &full[stage], cg * bke,
                            cx0 * args.cv_stride - args.cv_pad + kx, cy0 * args.cv_stride - args.cv_pad + ky, cb0);
              } else {
                tma_load_2d(sA + stage * A_STAGE, &tmA, &full[stage], kb * BK, m0);
              }
              if (!bres && !armed) tma_load_2d(sB + stage * BSTG, &tmB, &full[stage], kb * bke, n0);
              if constexpr (NB == 2)
                if (!armed) tma_load_2d(sB + stage * BSTG + BSTG / 2, &tmB2, &full[stage], kb * BK, n0);
            }
            last_mine = seq;
          }
          if (++stage == S) {
            stage = 0;
            phase ^= 1;
          }
          if (++cg == args.cv_cgroups) {  // (meaningful for convolutions only)
            cg = 0;
            if (++kx == args.cv_ks) {
              kx = 0;
              ++ky;
            }
          }
        }
      }
      if (!ok) record_status(args.status, ELASTO_ERR_TIMEOUT);
      // Drain: no copy this thread issued may still be landing in shared
      // memory when the CTA exits (returns at once on the normal path): the
      // stages of the sequence's last S k-blocks (no later k-block reuses
      // them) that this thread issued. In a pair only the even CTA's
      // barriers see the copies; the cluster barrier before exit orders the
      // odd CTA behind this drain.
      for (long q = seq - 1; leader && q >= 0 && q > seq - 1 - S; --q) {
        if (!mine(q) || q > last_mine) continue;
        const int st = static_cast<int>(q % S);
        const uint32_t ph = static_cast<uint32_t>((q / S) & 1);
        PAIR ? mbar_wait_cluster(&full[st], ph) : mbar_wait(&full[st], ph);
      }
      if (b_loaded) mbar_wait(bfull, 0);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && leader) {
      const uint32_t idesc = idesc_16_f32(TM, bn, args.f16 != 0);
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true, issued = false;
      // resident B: every tile's MMAs read it; wait for it once
      if (bres && t_start < tiles && !mbar_wait(bfull, 0)) ok = false;
      int local = 0;
      for (int t = t_start; t < tiles && ok; t += t_stride, ++local) {
        const int acc = local & 1;
        const uint32_t use = static_cast<uint32_t>(local >> 1);
        if (!(PAIR ? mbar_wait_cluster(&tempty[acc], (use & 1) ^ 1) : mbar_wait(&tempty[acc], (use & 1) ^ 1))) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t dtm = tmem_base + acc * MAX_BN;
        if (nk == 0) {
          mbar_arrive(&tfull[acc]);
          if constexpr (PAIR) mbar_arrive_cluster(cluster_map(smem_addr(&tfull[acc]), 1));
          continue;
        }
        const int kb0 = kSplit ? (t / mn_tiles) * nk / ks : 0, kb1 = kSplit ? (t / mn_tiles + 1) * nk / ks : nk;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!(PAIR ? mbar_wait_cluster(&full[stage], phase) : mbar_wait(&full[stage], phase))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_addr(sA + stage * A_STAGE), b0 = smem_addr(sB + (bres ? kb : stage) * BSTG);
          if (args.k16) {
            // one K=16 step per k-block: rows of 32 bytes in the 32-byte swizzle,
            // 8-row groups 256 bytes apart
            if constexpr (!PAIR && NB == 1)
              tc_mma(dtm, sdesc_sw32(a0, 16, 256), sdesc_sw32(b0, 16, 256), idesc, kb != kb0);
          } else {
            // the stage's descriptors once; a K = 16 step is +32 bytes = +2 in
            // the start-address field (the tiles are 1024-byte aligned, so it
            // never carries out of the field)
            const uint64_t da = sdesc_sw128(a0, 16, 1024), db = sdesc_sw128(b0, 16, 1024);
#pragma unroll
            for (int k = 0; k < BK / 16; ++k) {
              if constexpr (PAIR) {
                tc_mma_pair(dtm, da + 2 * k, db + 2 * k, idesc, kb != kb0 || k != 0);
              } else {
                tc_mma(dtm, da + 2 * k, db + 2 * k, idesc, kb != kb0 || k != 0);
                if constexpr (NB == 2)  // low half of the weights: acc += A . W_lo^T
                  tc_mma(dtm, da + 2 * k, sdesc_sw128(b0 + BSTG / 2, 16, 1024) + 2 * k, idesc, 1u);
              }
            }
          }
          issued = true;
          if constexpr (PAIR)
            tc_commit_pair_multicast(&empty[stage], 0x3);
          else
            tc_commit(&empty[stage]);
          if (++stage == S) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (ok) {
          if constexpr (PAIR)
            tc_commit_pair_multicast(&tfull[acc], 0x3);
          else
            tc_commit(&tfull[acc]);
        }
      }
      if (!ok) record_status(args.status, ELASTO_ERR_TIMEOUT);
      // All MMAs this thread issued have finished once `drain` completes.
      if (issued) {
        if constexpr (PAIR)
          tc_commit_pair(drain);
        else
          tc_commit(drain);
        mbar_wait(drain, 0);
      }
    }
  } else if constexpr (TR::tma) {
    // ------------------------------------------------------------ TMA-store epilogue
    constexpr int CW = TR::cw;
    constexpr int NG = EPI_THREADS / 128;   // warp groups sharing each chunk
    constexpr int HW = CW / NG;             // columns of a chunk handled by one thread
    constexpr int NC = HW * (TR::f32 ? 4 : 2) / 16;  // 16-byte pieces per thread
    const int q = warp & 3;                 // TMEM lane quarter
    const int g = (warp - 2) >> 2;          // warp group: which part of each chunk
    const int r = q * 32 + lane;            // row within the tile
    const bool elected = threadIdx.x == 64;
    const int cpt = bn / CW;
    const uint32_t row_tm = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
    // Every epilogue thread waits on the accumulator and residual barriers
    // itself (no barrier round just to share one thread's wait); a wait that
    // gives up raises `fail`. The flag is read only right after the chunk's
    // named barrier, where all threads see the same value, so the 512
    // threads leave together and the barrier is never left one arrival short.
    volatile int* fail = reinterpret_cast<volatile int*>(tmem_slot + 1);
    ChunkIter pf;  // residual prefetch iterator (elected thread only)
    pf.init(tiles, t_start, t_stride);
    long loads = 0, consumed = 0, stored = 0;
    if constexpr (TR::resid) {
      if (elected) {
        for (int e = 0; e < E && pf.valid; ++e) {
          mbar_expect_tx(&rfull[e], CBUF);
          tma_load_2d(sC + e * CBUF, &tmR, &rfull[e], (pf.t % nt) * bn + pf.c * CW,
                      resid_row(args, m_tile(args, pf.t / nt, mt) * TM + rank * BM));
          pf.advance(tiles, nt, bn, CW, N);
          ++loads;
        }
      }
    }
    int e = 0;
    uint32_t rph = 0;
    bool ok = true;
    int local = 0;
    for (int t = t_start; t < tiles && ok; t += t_stride, ++local) {
      const int acc = local & 1;
      const uint32_t use = static_cast<uint32_t>(local >> 1);
      if (!(PAIR ? mbar_wait_cluster(&tfull[acc], use & 1) : mbar_wait(&tfull[acc], use & 1))) *fail = 1;
      tc_fence_after();
      const int m0 = m_tile(args, t / nt, mt) * TM + rank * BM, n0 = (t % nt) * bn;
      const uint32_t acc_tm = row_tm + acc * MAX_BN;
      int nvalid = 0;
      while (nvalid < cpt && n0 + nvalid * CW < N) ++nvalid;
      for (int c = 0; c < nvalid; ++c) {
        uint8_t* buf = sC + e * CBUF;
        uint8_t* rowp = buf + r * 128;
        if constexpr (TR::resid) {
          if (!mbar_wait(&rfull[e], rph)) *fail = 1;
          ++consumed;
        }
        {
          // this thread: row r, columns [g*HW, g*HW + HW) of the chunk = the
          // 16-byte pieces NC*g .. NC*g + NC-1 of the 128-byte staging row
          uint32_t v[HW];
          if (nk > 0) {
            if constexpr (HW == 32)
              tmem_ld_32x32b_x32(acc_tm + c * CW + g * HW, v);
            else if constexpr (HW == 16)
              tmem_ld_16(acc_tm + c * CW + g * HW, v);
            else
              tmem_ld_8(acc_tm + c * CW + g * HW, v);
            tmem_ld_wait();
          } else {
#pragma unroll
            for (int j = 0; j < HW; ++j) v[j] = 0u;
          }
          if (c == nvalid - 1) {  // last TMEM read of this tile
            tc_fence_before();
            if (lane == 0) {
              if constexpr (PAIR)
                mbar_arrive_cluster(cluster_map(smem_addr(&tempty[acc]), 0));  // the even CTA issues the MMAs
              else
                mbar_arrive(&tempty[acc]);
            }
          }
          float bb[HW];
          load_bias<HW>(args.bias, n0 + c * CW + g * HW, N, bb);
          if constexpr (TR::f32) {
            // X_old arrived by TMA into the same swizzled row
#pragma unroll
            for (int j = 0; j < NC; ++j) {
              float4* p = reinterpret_cast<float4*>(rowp + (((NC * g + j) ^ (r & 7)) << 4));
              float4 o = *p;
              o.x += __uint_as_float(v[4 * j]) + bb[4 * j];
              o.y += __uint_as_float(v[4 * j + 1]) + bb[4 * j + 1];
              o.z += __uint_as_float(v[4 * j + 2]) + bb[4 * j + 2];
              o.w += __uint_as_float(v[4 * j + 3]) + bb[4 * j + 3];
              *p = o;
            }
          } else if constexpr (TR::resid16) {
            // the residual's 8 values arrived by TMA into this 16-byte piece
#pragma unroll
            for (int j = 0; j < NC; ++j) {
              uint4* p = reinterpret_cast<uint4*>(rowp + (((NC * g + j) ^ (r & 7)) << 4));
              const uint4 rv = *p;
              const uint32_t rw[4] = {rv.x, rv.y, rv.z, rv.w};
              uint32_t ow[4];
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                const float2 rf = unpack_in<EPI>(rw[i]);
                ow[i] = pack_out<EPI>(epi_act<EPI>(__uint_as_float(v[8 * j + 2 * i]) + bb[8 * j + 2 * i] + rf.x),
                                      epi_act<EPI>(__uint_as_float(v[8 * j + 2 * i + 1]) + bb[8 * j + 2 * i + 1] +
                                                   rf.y));
              }
              *p = make_uint4(ow[0], ow[1], ow[2], ow[3]);
            }
          } else {
#pragma unroll
            for (int j = 0; j < NC; ++j) {
              uint4 pk;
              pk.x = pack_out<EPI>(epi_act<EPI>(__uint_as_float(v[8 * j + 0]) + bb[8 * j + 0]),
                                 epi_act<EPI>(__uint_as_float(v[8 * j + 1]) + bb[8 * j + 1]));
              pk.y = pack_out<EPI>(epi_act<EPI>(__uint_as_float(v[8 * j + 2]) + bb[8 * j + 2]),
                                 epi_act<EPI>(__uint_as_float(v[8 * j + 3]) + bb[8 * j + 3]));
              pk.z = pack_out<EPI>(epi_act<EPI>(__uint_as_float(v[8 * j + 4]) + bb[8 * j + 4]),
                                 epi_act<EPI>(__uint_as_float(v[8 * j + 5]) + bb[8 * j + 5]));
              pk.w = pack_out<EPI>(epi_act<EPI>(__uint_as_float(v[8 * j + 6]) + bb[8 * j + 6]),
                                 epi_act<EPI>(__uint_as_float(v[8 * j + 7]) + bb[8 * j + 7]));
              *reinterpret_cast<uint4*>(rowp + (((NC * g + j) ^ (r & 7)) << 4)) = pk;
            }
          }
        }
        fence_async_smem();
        // The previous chunk's store (issued a whole chunk ago) must have read
        // its buffer before anyone passes this barrier: after it, that buffer
        // is written by the next chunk (E = 2) or refilled by the prefetch.
        if (elected) bulk_wait_read_all();
        named_bar_sync(1, EPI_THREADS);
        if (*fail) {
          ok = false;
          break;
        }
        if (elected) {
          if (args.conv) {
            int cb0, cy0, cx0;
            conv_tile(args, m_tile(args, t / nt, mt), cb0, cy0, cx0);
            tma_store_4d(&tmC, buf, n0 + c * CW, cx0, cy0, cb0);
          } else {
            tma_store_2d(&tmC, buf, n0 + c * CW, m0);
          }
          bulk_commit();  // stays in flight while the next chunk is computed
          if constexpr (TR::resid) {
            if (stored > 0 && pf.valid) {
              const int ep = e == 0 ? E - 1 : e - 1;  // buffer of the previous chunk
              mbar_expect_tx(&rfull[ep], CBUF);
              tma_load_2d(sC + ep * CBUF, &tmR, &rfull[ep], (pf.t % nt) * bn + pf.c * CW,
                          resid_row(args, m_tile(args, pf.t / nt, mt) * TM + rank * BM));
              pf.advance(tiles, nt, bn, CW, N);
              ++loads;
            }
          }
          ++stored;
        }
        if (++e == E) {
          e = 0;
          rph ^= 1;
        }
      }
    }
    if (!ok && elected) record_status(args.status, ELASTO_ERR_TIMEOUT);
    if (elected) {
      bulk_wait_all();
      if constexpr (TR::resid) {
        // Residual loads issued for chunks never consumed (only on the abort
        // path): let them land before the CTA releases its shared memory.
        for (long i = consumed; i < loads; ++i) {
          mbar_wait(&rfull[e], rph);
          if (++e == E) {
            e = 0;
            rph ^= 1;
          }
        }
      }
    }
  } else {
    // ------------------------------------------------------------ transpose epilogue
    // (warps 2-5 only; the other epilogue warps have nothing to do here)
    if (warp < 6) {
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    float* st = reinterpret_cast<float*>(sC) + (warp - 2) * EPI_TILE;
    int local = 0;
    for (int t = t_start; t < tiles; t += t_stride, ++local) {
      const int acc = local & 1;
      const uint32_t use = static_cast<uint32_t>(local >> 1);
      if (!mbar_wait(&tfull[acc], use & 1)) {
        if (lane == 0) record_status(args.status, ELASTO_ERR_TIMEOUT);
        break;
      }
      tc_fence_after();
      const int tq = t % mn_tiles;
      const int m0 = m_tile(args, tq / nt, mt) * TM + rank * BM, n0 = (tq % nt) * bn;
      const int row0 = m0 + q * 32;
      for (int c = 0; c < bn; c += 32) {
        if (n0 + c >= N) break;
        uint32_t r[32];
        if (nk > 0) {
          tmem_ld_32x32b_x32(tmem_base + (static_cast<uint32_t>(q * 32) << 16) + acc * MAX_BN + c, r);
          tmem_ld_wait();
        } else {
#pragma unroll
          for (int j = 0; j < 32; ++j) r[j] = 0u;
        }
#pragma unroll
        for (int j = 0; j < 32; ++j) st[lane * EPI_LD + j] = __uint_as_float(r[j]);
        __syncwarp();
        {  // EPI_BIAS_F32
          const int col = n0 + c + lane;
          const bool cok = col < N;
          const float bv = (cok && args.bias) ? args.bias[col] : 0.0f;
          float* out = static_cast<float*>(args.out) + (t / mn_tiles) * args.split_stride;
#pragma unroll 8
          for (int i = 0; i < 32; ++i) {
            const int row = row0 + i;
            if (cok && row < M) out[static_cast<size_t>(row) * args.ldo + col] = st[i * EPI_LD + lane] + bv;
          }
        }
        __syncwarp();
      }
      tc_fence_before();
      if (lane == 0) mbar_arrive(&tempty[acc]);
    }
    }
  }
  tc_fence_before();
  __syncthreads();
  if constexpr (PAIR) cluster_sync_all();  // the peer's TMEM and barriers are no longer in use
  if (warp == 0) {
    __syncwarp();
    tc_fence_after();
    if constexpr (PAIR)
      tmem_dealloc_pair(tmem_base, TMEM_COLS);
    else
      tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// Split-K residual: out[r, c] += (sum over splits of part[s][r, c]) + bias[c],
// the splits added in order, the sum and bias associated as in the one-pass
// RESID_F32 epilogue (x + (acc + b)). One thread per 4 columns of a row.
__global__ void splitk_reduce_kernel(const float* __restrict__ part, int ks, long long stride, int M, int N,
                                     const float* __restrict__ bias, float* __restrict__ out, int ldo) {
  pdl_wait();
  pdl_trigger();
  const int n4 = N / 4;
  const size_t total = static_cast<size_t>(M) * n4;
  for (size_t i = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
       i += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const size_t r = i / n4;
    const int c = static_cast<int>(i - r * n4) * 4;
    float4 acc = *reinterpret_cast<const float4*>(part + r * N + c);
    for (int sp = 1; sp < ks; ++sp) {
      const float4 v = *reinterpret_cast<const float4*>(part + sp * stride + r * N + c);
      acc.x += v.x;
      acc.y += v.y;
      acc.z += v.z;
      acc.w += v.w;
    }
    const float4 b = bias ? *reinterpret_cast<const float4*>(bias + c) : make_float4(0.f, 0.f, 0.f, 0.f);
    float4* o = reinterpret_cast<float4*>(out + r * ldo + c);
    float4 x = *o;
    x.x += acc.x + b.x;
    x.y += acc.y + b.y;
    x.z += acc.z + b.z;
    x.w += acc.w + b.w;
    *o = x;
  }
}

// Sum over the threads of a block of nw warps (nw <= 32); red: nw floats of
// shared memory. Every thread gets the total.
__device__ __forceinline__ float block_sum(float v, float* red, int nw) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float t = lane < nw ? red[lane] : 0.0f;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
  __syncthreads();  // red is reused by the next call
  return t;
}

// The same sum, and then the LayerNorm of each finished row: one block of
// N / 2 threads per row, two channels per thread (all the row's partial sums
// in flight at once). Statistics as layernorm_kernel takes them (mean over
// the first d_true channels, centred sum of squares less the zero padding's
// pad * mean^2, eps 1e-6), summed in another order.
__global__ void __launch_bounds__(512) splitk_reduce_ln_kernel(const float* __restrict__ part, int ks,
                                                               long long stride, int N,
                                                               const float* __restrict__ bias,
                                                               float* __restrict__ out, const float* __restrict__ g,
                                                               const float* __restrict__ b, bf16* __restrict__ y,
                                                               float inv_d, float pad) {
  __shared__ float red[32];
  pdl_wait();
  pdl_trigger();
  const size_t e = static_cast<size_t>(blockIdx.x) * N + 2 * threadIdx.x;
  float2 p2[kSplitMax];
#pragma unroll
  for (int sp = 0; sp < kSplitMax; ++sp)
    p2[sp] = sp < ks ? *reinterpret_cast<const float2*>(part + sp * stride + e) : make_float2(0.f, 0.f);
  float2 acc = p2[0];
#pragma unroll
  for (int sp = 1; sp < kSplitMax; ++sp)
    if (sp < ks) {
      acc.x += p2[sp].x;
      acc.y += p2[sp].y;
    }
  const float2 bb = bias ? reinterpret_cast<const float2*>(bias)[threadIdx.x] : make_float2(0.f, 0.f);
  float2* o = reinterpret_cast<float2*>(out + e);
  float2 x = *o;
  x.x += acc.x + bb.x;
  x.y += acc.y + bb.y;
  *o = x;
  const int nw = blockDim.x >> 5;
  const float mean = block_sum(x.x + x.y, red, nw) * inv_d;
  const float a = x.x - mean, c = x.y - mean;
  const float rstd = rsqrtf((block_sum(a * a + c * c, red, nw) - pad * mean * mean) * inv_d + 1e-6f);
  const float2 gg = reinterpret_cast<const float2*>(g)[threadIdx.x];
  const float2 be = reinterpret_cast<const float2*>(b)[threadIdx.x];
  reinterpret_cast<uint32_t*>(y)[e / 2] = pack_bf16x2(a * rstd * gg.x + be.x, c * rstd * gg.y + be.y);
}

template <int EPI, int NB, bool PAIR>
cudaError_t launch_epi(const GemmPlan& p, int M, cudaStream_t s) {
  GemmArgs a = p.args;
  a.M = M;
  a.cv_batch = M;  // implicit convolutions: M counts images
  const int nt = (a.N + a.bn - 1) / a.bn;
  if constexpr (PAIR) {
    static int max_clusters[64] = {0};
    int dev = 0;
    cudaGetDevice(&dev);
    cudaLaunchConfig_t cfg{};
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see launch_pdl
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = SMEM_BYTES;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;  // the occupancy query sees the cluster shape only
    if (dev >= 0 && dev < 64 && max_clusters[dev] == 0) {
      cfg.gridDim = dim3(2 * (num_sms() / 2));
      int n = 0;
      cudaError_t e = cudaOccupancyMaxActiveClusters(&n, gemm_tc_kernel<EPI, NB, true>, &cfg);
      if (e != cudaSuccess || n <= 0) return e != cudaSuccess ? e : cudaErrorInvalidConfiguration;
      max_clusters[dev] = n;
    }
    const int tiles = ((M + 2 * BM - 1) / (2 * BM)) * nt;
    const int clusters = tiles < max_clusters[dev] ? tiles : max_clusters[dev];
    cfg.gridDim = dim3(2 * clusters);
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, gemm_tc_kernel<EPI, NB, true>, p.tmA, p.tmB, p.tmB2, p.tmC, p.tmR, a);
  } else {
    const int tiles = (a.conv ? conv_mtiles(a) : (M + BM - 1) / BM) * nt * (a.ksplit > 1 ? a.ksplit : 1);
    const int grid = tiles < num_sms() ? tiles : num_sms();
    return launch_pdl(gemm_tc_kernel<EPI, NB, false>, dim3(grid), dim3(a.conv ? THREADS_CONV : THREADS), SMEM_BYTES, s,
                      p.tmA, p.tmB, p.tmB2,
                      p.tmC, p.tmR, a);
  }
}

}  // namespace

cudaError_t gemm_init_attributes() {
  const int bytes = static_cast<int>(SMEM_BYTES);
  cudaError_t e;
#define SET_ATTR(E)                                                                                        \
  e = cudaFuncSetAttribute(gemm_tc_kernel<E, 1, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);   \
  if (e != cudaSuccess) return e;                                                                          \
  e = cudaFuncSetAttribute(gemm_tc_kernel<E, 2, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);   \
  if (e != cudaSuccess) return e;
#define SET_ATTR_PAIR(E)                                                                                   \
  e = cudaFuncSetAttribute(gemm_tc_kernel<E, 1, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);    \
  if (e != cudaSuccess) return e;
  SET_ATTR(EPI_BIAS_BF16)
  SET_ATTR(EPI_BIAS_GELU_BF16)
  SET_ATTR(EPI_BIAS_RESID_F32)
  SET_ATTR(EPI_BIAS_F32)
  SET_ATTR(EPI_BIAS_RELU_BF16)
  SET_ATTR(EPI_BIAS_RESID_RELU_BF16)
  SET_ATTR(EPI_BIAS_RELU_F16)
  SET_ATTR(EPI_BIAS_F16)
  SET_ATTR(EPI_BIAS_RESID_RELU_F16)
  SET_ATTR_PAIR(EPI_BIAS_RELU_F16)
  SET_ATTR_PAIR(EPI_BIAS_F16)
  SET_ATTR_PAIR(EPI_BIAS_BF16)
  SET_ATTR_PAIR(EPI_BIAS_GELU_BF16)
  SET_ATTR_PAIR(EPI_BIAS_RESID_F32)
  SET_ATTR_PAIR(EPI_BIAS_RELU_BF16)
#undef SET_ATTR
#undef SET_ATTR_PAIR
  return cudaSuccess;
}

int gemm_pick_bn(int M, int N, int step, bool pair) {
  // Estimated time ~ waves x (bn + fixed per-tile overhead); ties prefer wider tiles.
  const int sms = num_sms() > 0 ? num_sms() : 148;
  const int units = pair ? sms / 2 : sms;  // concurrent tile workers
  const int mt = (M + (pair ? 2 * BM : BM) - 1) / (pair ? 2 * BM : BM);
  int best = 256;
  long best_cost = -1;
  for (int bn = 256; bn >= step; bn -= step) {
    const long tiles = static_cast<long>(mt) * ((N + bn - 1) / bn);
    const long waves = (tiles + units - 1) / units;
    const long cost = waves * (bn + 32);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = bn;
    }
  }
  return best;
}

elasto_status gemm_plan(GemmPlan* p, const bf16* A, int M_cap, const bf16* W, int N, int K, const float* bias,
                        void* out, int ldo, int epi, int* status, const bf16* W_lo, int M_hint, int ldw,
                        int bn_force) {
  if (!p || M_cap <= 0 || N <= 0 || K < 0 || !out || (K > 0 && (!A || !W))) {
    set_error("gemm_plan: invalid arguments");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (ldw <= 0) ldw = K;
  if (K % 8 != 0 || N % 2 != 0 || ldw < K || ldw % 8 != 0) {
    set_error("gemm: K and ldw must be multiples of 8 (ldw >= K) and N even");
    return ELASTO_ERR_UNSUPPORTED;
  }
  *p = GemmPlan{};
  const bool resid16 = epi == EPI_BIAS_RESID_RELU_BF16 || epi == EPI_BIAS_RESID_RELU_F16;
  const bool tma_out = epi == EPI_BIAS_BF16 || epi == EPI_BIAS_GELU_BF16 || epi == EPI_BIAS_RELU_BF16 ||
                       epi == EPI_BIAS_RESID_F32 || epi == EPI_BIAS_RELU_F16 || epi == EPI_BIAS_F16 || resid16;
  const bool f32_out = epi == EPI_BIAS_RESID_F32;
  const bool has_resid = f32_out || resid16;
  GemmArgs& a = p->args;
  a.f16 = (epi == EPI_BIAS_RELU_F16 || epi == EPI_BIAS_F16 || epi == EPI_BIAS_RESID_RELU_F16) ? 1 : 0;
  a.M = M_cap;
  a.N = N;
  a.K = K;
  // CTA pairs for the TMA-store epilogues on problems with at least one
  // 256-row tile and single-plane weights
  // (long reductions only: with K = 768 the per-tile epilogue dominates and
  // a single CTA per tile measured faster)
  const int Mt = (M_hint > 0 && M_hint < M_cap) ? M_hint : M_cap;  // rows the tiling is chosen for
  const bool pair = tma_out && !W_lo && Mt >= 2 * BM && K >= 1536;
  a.pair = pair ? 1 : 0;
  // bf16 staging chunks are 64 columns wide: their tiles are multiples of 64
  a.bn = bn_force > 0 ? bn_force : gemm_pick_bn(Mt, N, (tma_out && !f32_out) ? 64 : 32, pair);
  // one B stage holds exactly the tile's rows (both planes); the freed bytes
  // become a deeper operand ring for narrow tiles
  a.b_stage = pair ? (a.bn / 2) * BK * 2 : (W_lo ? 2 : 1) * a.bn * BK * 2;
  a.bias = bias;
  a.out = out;
  a.ldo = ldo;
  a.status = status;
  a.b_planes = W_lo ? 2 : 1;
  p->epi = epi;
  if (tma_out) {
    // residual GEMMs: 3 operand stages and 5 staging chunks fetched ahead;
    // the others: 4 stages and 2 staging chunks.
    // residual epilogues keep 5 staging chunks (residual rows fetched
    // ahead), the others 2; the rest of the pool is operand ring
    const int keep = has_resid ? 5 : 2;
    a.stages = (POOL - keep * CBUF) / (A_STAGE + a.b_stage);
    if (a.stages > MAX_STAGES) a.stages = MAX_STAGES;
    if (a.stages < 2) a.stages = 2;
    if (pair) a.stages = has_resid ? 5 : 6;  // tuned for the K >= 1536 reductions
    a.cbufs = (POOL - a.stages * (A_STAGE + a.b_stage)) / CBUF;
    if (a.cbufs > MAX_CBUFS) a.cbufs = MAX_CBUFS;
    if (ldo % 8 != 0 ||
        !encode_tmap_2d(&p->tmC, out, ldo, M_cap, static_cast<uint64_t>(ldo) * (f32_out ? 4 : 2),
                        f32_out ? 32 : 64, BM, f32_out)) {
      set_error("gemm_plan: output tensor map (alignment or size)");
      return ELASTO_ERR_UNSUPPORTED;
    }
    p->tmR = p->tmC;  // the residual is read from the output unless redirected
  } else {
    a.stages = (POOL - 4 * EPI_TILE * 4) / (A_STAGE + a.b_stage);
    if (a.stages > 4) a.stages = 4;
    a.cbufs = 0;
  }
  {
    // the operand ring, staging chunks (or transpose tiles) must fit the pool
    const int bstg = a.b_stage;
    const int tail = tma_out ? a.cbufs * CBUF : 4 * EPI_TILE * 4;
    if (a.stages < 2 || a.stages > MAX_STAGES || a.cbufs > MAX_CBUFS || (tma_out && a.cbufs < 2) ||
        a.stages * (A_STAGE + bstg) + tail > POOL) {
      set_error("gemm_plan: shared-memory layout does not fit");
      return ELASTO_ERR_UNSUPPORTED;
    }
  }
  if (K > 0) {
    if (!encode_tmap_2d(&p->tmA, A, K, M_cap, static_cast<uint64_t>(K) * 2, BK, BM) ||
        !encode_tmap_2d(&p->tmB, W, K, N, static_cast<uint64_t>(ldw) * 2, BK, pair ? a.bn / 2 : a.bn) ||
        (W_lo && !encode_tmap_2d(&p->tmB2, W_lo, K, N, static_cast<uint64_t>(ldw) * 2, BK, a.bn))) {
      set_error("gemm_plan: cuTensorMapEncodeTiled failed (alignment or size)");
      return ELASTO_ERR_UNSUPPORTED;
    }
  }
  p->valid = true;
  return ELASTO_OK;
}

elasto_status gemm_plan_split_resid(GemmPlan* p, const bf16* A, int M_cap, const bf16* W, int N, int K,
                                    const float* bias, float* out, int ldo, int* status, const bf16* W_lo, int M_rows,
                                    int ldw, float* part) {
  const int sms = num_sms() > 0 ? num_sms() : 148;
  const int rows = (M_rows > 0 && M_rows < M_cap) ? M_rows : M_cap;
  const int mt = (rows + BM - 1) / BM, nk = (K + BK - 1) / BK;
  // the N tile and split count with the fewest k-blocks per CTA, every
  // split keeping at least 4 k-blocks
  int best_bn = 0, best_ks = 1, best_kb = nk + 1;
  for (int bn : {64, 32}) {
    const int tiles = mt * ((N + bn - 1) / bn);
    const int ks = std::min({kSplitMax, sms / std::max(tiles, 1), nk / 4});
    if (ks < 2) continue;
    const int kb = (nk + ks - 1) / ks;
    if (kb < best_kb) {
      best_kb = kb;
      best_bn = bn;
      best_ks = ks;
    }
  }
  if (best_bn == 0 || !part || N % 4 != 0 || ldo % 4 != 0)
    return gemm_plan(p, A, M_cap, W, N, K, bias, out, ldo, EPI_BIAS_RESID_F32, status, W_lo, M_rows, ldw);
  elasto_status st =
      gemm_plan(p, A, M_cap, W, N, K, nullptr, part, N, EPI_BIAS_F32, status, W_lo, rows, ldw, best_bn);
  if (st != ELASTO_OK) return st;
  p->args.ksplit = best_ks;
  p->args.split_stride = static_cast<long long>(rows) * N;
  p->rbias = bias;
  p->rout = out;
  p->rldo = ldo;
  p->rcap = rows;
  return ELASTO_OK;
}

bool gemm_split_fuse_layernorm(GemmPlan* p, const float* g, const float* b, bf16* y, int d_true) {
  if (!p || p->args.ksplit <= 1 || !g || !b || !y || p->rldo != p->args.N || p->args.N % 64 != 0 ||
      p->args.N > 1024 || d_true <= 0 || d_true > p->args.N)
    return false;
  p->ln_g = g;
  p->ln_b = b;
  p->ln_y = y;
  p->ln_d = d_true;
  return true;
}

namespace {

// The part both convolution plans share. A is read through the 4D map
// {channels, x, y, image} = xd (byte strides xs) in boxes of bke channels by
// the tile's pixel block; k-block kb covers tap kb / cg (ky = tap / taps_x,
// kx = tap % taps_x) and channel group kb % cg.
elasto_status plan_conv_common(GemmPlan* p, const char* who, const void* x, const uint64_t xd[4],
                               const uint64_t xs[3], int B_cap, int Ho, int Wo, int taps, int taps_x, int cg, int bke,
                               int stride, int pad, const void* Wt, int N, const float* bias, void* out, int ldo,
                               int epi, int* status) {
  *p = GemmPlan{};
  GemmArgs& a = p->args;
  const bool k16 = bke == 16;
  a.M = B_cap;
  a.N = N;
  a.K = taps * cg * bke;
  a.k16 = k16 ? 1 : 0;
  a.conv = 1;
  a.cv_ks = taps_x;
  a.cv_stride = stride;
  a.cv_pad = pad;
  a.cv_cgroups = cg;
  a.cv_ho = Ho;
  a.cv_wo = Wo;
  // pixel block of an M tile: the fewest tiles of at most 128 pixels; whole
  // images when several fit (then nb images per tile)
  long best = -1;
  if (Ho * Wo <= BM / 2) {
    a.cv_bw = Wo;
    a.cv_bh = Ho;
    a.cv_nb = BM / (Ho * Wo);
    best = (B_cap + a.cv_nb - 1) / a.cv_nb;
  }
  for (int bw = 1; bw <= Wo && bw <= BM; ++bw)
    for (int bh = 1; bh <= Ho && bw * bh <= BM; ++bh) {
      const long tiles = long((Wo + bw - 1) / bw) * ((Ho + bh - 1) / bh) * B_cap;
      if (best < 0 || tiles < best || (tiles == best && a.cv_nb == 1 && bw > a.cv_bw)) {
        best = tiles;
        a.cv_bw = bw;
        a.cv_bh = bh;
        a.cv_nb = 1;
      }
    }
  const int rows = a.cv_bw * a.cv_bh * a.cv_nb;
  a.cv_a_bytes = rows * bke * 2;
  a.cv_batch = B_cap;
  a.bn = gemm_pick_bn(conv_mtiles(a) * BM, N, 64, false);
  a.bias = bias;
  a.out = out;
  a.ldo = ldo;
  a.status = status;
  a.b_planes = 1;
  a.f16 = 1;
  a.pair = 0;
  // one N tile whose whole W fits beside a 4-stage A ring: W is loaded once
  // per CTA and kept, instead of once per tile and k-block from L2
  const int nk = taps * cg;
  const int b_all = nk * a.bn * bke * 2;
  a.b_resident = (N <= a.bn && 4 * A_STAGE + b_all + 2 * CBUF <= POOL) ? 1 : 0;
  if (a.b_resident) {
    a.b_stage = a.bn * bke * 2;  // one k-block of W
    a.stages = (POOL - 2 * CBUF - b_all) / A_STAGE;
    if (a.stages > MAX_STAGES) a.stages = MAX_STAGES;
    a.cbufs = (POOL - a.stages * A_STAGE - b_all) / CBUF;
  } else {
    a.b_stage = a.bn * BK * 2;
    a.stages = (POOL - 2 * CBUF) / (A_STAGE + a.b_stage);
    if (a.stages > MAX_STAGES) a.stages = MAX_STAGES;
    a.cbufs = (POOL - a.stages * (A_STAGE + a.b_stage)) / CBUF;
  }
  if (a.cbufs > MAX_CBUFS) a.cbufs = MAX_CBUFS;
  if (a.cbufs < 2 || rows > BM || a.stages < 2) {
    set_error(std::string(who) + ": shared-memory layout does not fit");
    return ELASTO_ERR_UNSUPPORTED;
  }
  const uint32_t xb[4] = {uint32_t(bke), uint32_t(a.cv_bw * stride), uint32_t(a.cv_bh * stride), uint32_t(a.cv_nb)};
  const uint32_t xe[4] = {1u, uint32_t(stride), uint32_t(stride), 1u};
  const uint64_t od[4] = {uint64_t(N), uint64_t(Wo), uint64_t(Ho), uint64_t(B_cap)};
  const uint64_t os[3] = {uint64_t(ldo) * 2, uint64_t(Wo) * ldo * 2, uint64_t(Ho) * Wo * ldo * 2};
  const uint32_t ob[4] = {64u, uint32_t(a.cv_bw), uint32_t(a.cv_bh), uint32_t(a.cv_nb)};
  const uint32_t oe[4] = {1u, 1u, 1u, 1u};
  const bool wmap = k16 ? encode_tmap_2d_sw32(&p->tmB, Wt, a.K, N, uint64_t(a.K) * 2, 16, a.bn)
                        : encode_tmap_2d(&p->tmB, Wt, a.K, N, uint64_t(a.K) * 2, BK, a.bn);
  if (xb[1] > 256 || xb[2] > 256 || !encode_tmap_4d(&p->tmA, x, xd, xs, xb, xe, k16) || !wmap ||
      !encode_tmap_4d(&p->tmC, out, od, os, ob, oe)) {
    set_error(std::string(who) + ": cuTensorMapEncodeTiled failed (alignment or size)");
    return ELASTO_ERR_UNSUPPORTED;
  }
  p->tmR = p->tmC;
  p->epi = epi;
  p->valid = true;
  return ELASTO_OK;
}

bool conv_args_ok(const GemmPlan* p, const void* x, const void* Wt, void* out, int B_cap, int N, int ldo, int epi) {
  return p && x && Wt && out && B_cap > 0 && N > 0 && (epi == EPI_BIAS_RELU_F16 || epi == EPI_BIAS_F16);
}

}  // namespace

elasto_status gemm_plan_conv(GemmPlan* p, const void* x, int B_cap, int H, int W, int C, int k, int stride, int pad,
                             const void* Wt, int N, const float* bias, void* out, int ldo, int epi, int* status,
                             int Ho_out, int Wo_out) {
  if (!conv_args_ok(p, x, Wt, out, B_cap, N, ldo, epi) || H <= 0 || W <= 0 || C <= 0 || k <= 0 || stride <= 0 ||
      pad < 0) {
    set_error("gemm_plan_conv: invalid arguments");
    return ELASTO_ERR_INVALID_ARG;
  }
  const int Ho_full = (H + 2 * pad - k) / stride + 1, Wo_full = (W + 2 * pad - k) / stride + 1;
  const int Ho = Ho_out > 0 ? Ho_out : Ho_full, Wo = Wo_out > 0 ? Wo_out : Wo_full;
  if (Ho > Ho_full || Wo > Wo_full) {
    set_error("gemm_plan_conv: the output window exceeds the convolution's output");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (C % 8 != 0 || ldo % 8 != 0 || N % 2 != 0 || N > ldo || Ho <= 0 || Wo <= 0 || stride > 2) {
    set_error("gemm_plan_conv: needs C and ldo multiples of 8, N even, stride 1 or 2");
    return ELASTO_ERR_UNSUPPORTED;
  }
  // up to 16 channels: one 16-wide k-block per tap (32-byte swizzle) instead
  // of a 64-channel group that would be three quarters zeros
  const int bke = conv_tap_stride(C) == 16 ? 16 : BK;
  const uint64_t xd[4] = {uint64_t(C), uint64_t(W), uint64_t(H), uint64_t(B_cap)};
  const uint64_t xs[3] = {uint64_t(C) * 2, uint64_t(W) * C * 2, uint64_t(H) * W * C * 2};
  return plan_conv_common(p, "gemm_plan_conv", x, xd, xs, B_cap, Ho, Wo, k * k, k, conv_tap_stride(C) / bke, bke,
                          stride, pad, Wt, N, bias, out, ldo, epi, status);
}

elasto_status gemm_plan_conv_rows(GemmPlan* p, const void* x, int B_cap, int Hp, int Wp, int C, int kh, int kw,
                                  const void* Wt, int N, const float* bias, void* out, int ldo, int epi, int* status,
                                  int Ho_out, int Wo_out) {
  if (!conv_args_ok(p, x, Wt, out, B_cap, N, ldo, epi) || C <= 0 || kh <= 0 || kw <= 0 || Hp < kh || Wp < kw) {
    set_error("gemm_plan_conv_rows: invalid arguments");
    return ELASTO_ERR_INVALID_ARG;
  }
  const int Ho_full = Hp - kh + 1, Wo_full = Wp - kw + 1;
  const int Ho = Ho_out > 0 ? Ho_out : Ho_full, Wo = Wo_out > 0 ? Wo_out : Wo_full;
  if (Ho > Ho_full || Wo > Wo_full) {
    set_error("gemm_plan_conv_rows: the output window exceeds the convolution's output");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (kw * C != BK || C % 8 != 0 || ldo % 8 != 0 || N % 2 != 0 || N > ldo) {
    set_error("gemm_plan_conv_rows: needs kw * C == 64, C and ldo multiples of 8, N even");
    return ELASTO_ERR_UNSUPPORTED;
  }
  // the map's x axis steps one pixel (C channels) while each box row takes
  // kw * C = 64 values: the kw pixels that kernel row ky meets, overlapping
  // the next row's; x runs over the Wo_full window starts only, so no box row
  // reaches past the end of an input row
  const uint64_t xd[4] = {uint64_t(BK), uint64_t(Wo_full), uint64_t(Hp), uint64_t(B_cap)};
  const uint64_t xs[3] = {uint64_t(C) * 2, uint64_t(Wp) * C * 2, uint64_t(Hp) * Wp * C * 2};
  return plan_conv_common(p, "gemm_plan_conv_rows", x, xd, xs, B_cap, Ho, Wo, kh, 1, 1, BK, 1, 0, Wt, N, bias, out,
                          ldo, epi, status);
}

elasto_status gemm_set_residual_source(GemmPlan* p, const void* src, int M_cap, int row_period) {
  const bool f32 = p && p->epi == EPI_BIAS_RESID_F32;
  const bool r16 = p && (p->epi == EPI_BIAS_RESID_RELU_BF16 || p->epi == EPI_BIAS_RESID_RELU_F16);
  if (!p || !p->valid || !(f32 || r16) || !src) {
    set_error("gemm_set_residual_source: needs a residual plan and a source");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (row_period < 0 || (row_period > 0 && (p->args.conv || M_cap < row_period + BM))) {
    set_error("gemm_set_residual_source: a periodic source needs period + 128 rows and a plain GEMM");
    return ELASTO_ERR_INVALID_ARG;
  }
  p->args.resid_row_mod = row_period;
  const int ldo = p->args.ldo;
  if (!encode_tmap_2d(&p->tmR, src, ldo, M_cap, static_cast<uint64_t>(ldo) * (f32 ? 4 : 2), f32 ? 32 : 64, BM,
                      f32)) {
    set_error("gemm_set_residual_source: tensor map (alignment or size)");
    return ELASTO_ERR_UNSUPPORTED;
  }
  return ELASTO_OK;
}

namespace {

cudaError_t gemm_launch_main(const GemmPlan& p, int M, cudaStream_t s) {
  const bool two = p.args.b_planes == 2, pair = p.args.pair != 0;
#define CASE(E) \
  case E: return two ? launch_epi<E, 2, false>(p, M, s) : launch_epi<E, 1, false>(p, M, s);
#define CASE_PAIR(E)                                   \
  case E:                                              \
    if (pair) return launch_epi<E, 1, true>(p, M, s);  \
    return two ? launch_epi<E, 2, false>(p, M, s) : launch_epi<E, 1, false>(p, M, s);
  switch (p.epi) {
    CASE_PAIR(EPI_BIAS_BF16)
    CASE_PAIR(EPI_BIAS_GELU_BF16)
    CASE_PAIR(EPI_BIAS_RESID_F32)
    CASE(EPI_BIAS_F32)
    CASE_PAIR(EPI_BIAS_RELU_BF16)
    CASE(EPI_BIAS_RESID_RELU_BF16)
    CASE_PAIR(EPI_BIAS_RELU_F16)
    CASE_PAIR(EPI_BIAS_F16)
    CASE(EPI_BIAS_RESID_RELU_F16)
#undef CASE
#undef CASE_PAIR
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t gemm_launch(const GemmPlan& p, int M, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  if (p.args.ksplit <= 1) return gemm_launch_main(p, M, s);
  if (M > p.rcap) return cudaErrorInvalidValue;  // the partial buffer holds rcap rows
  cudaError_t e = gemm_launch_main(p, M, s);
  if (e != cudaSuccess) return e;
  if (p.ln_y) {
    const float inv_d = 1.0f / static_cast<float>(p.ln_d), pad = static_cast<float>(p.args.N - p.ln_d);
    return launch_pdl(splitk_reduce_ln_kernel, dim3(M), dim3(p.args.N / 2), 0, s,
                      static_cast<const float*>(p.args.out), p.args.ksplit, p.args.split_stride, p.args.N, p.rbias,
                      p.rout, p.ln_g, p.ln_b, p.ln_y, inv_d, pad);
  }
  const size_t work = static_cast<size_t>(M) * (p.args.N / 4);
  const unsigned grid = static_cast<unsigned>(std::min<size_t>((work + 255) / 256, 4096));
  return launch_pdl(splitk_reduce_kernel, dim3(grid), dim3(256), 0, s, static_cast<const float*>(p.args.out),
                    p.args.ksplit, p.args.split_stride, M, p.args.N, p.rbias, p.rout, p.rldo);
}

}  // namespace elasto
