// Tensor-core GEMM with fused epilogues: out = epi(A[M,K] . W[N,K]^T).
//
// This is every dense contraction of the DN forward (Section 4.1): the patch
// projection, the sliced QKV projection of the kept heads (Eq. 2, 4), the
// sliced output projection W^O (Eq. 2, 4) and the sliced MLP W1 / W2
// (Eq. 5, 6). Slicing happened at create time, so here the kept widths are
// just the problem's N or K.
//
// Design (sm_103a):
//  - persistent grid, one CTA per SM, static round-robin over 128 x bn tiles
//    (N tile index fastest so the CTAs running together share A rows in L2);
//  - warp 0 lane 0: TMA producer, 4-stage ring of 128x64 (A) and bn x 64 (B)
//    bf16 tiles with the 128-byte swizzle, one mbarrier pair per stage;
//  - warp 1 lane 0: issues tcgen05.mma (M=128, N=bn, K=16) into one of two
//    TMEM accumulators (2 x 256 fp32 columns), commits stages back to the
//    producer and finished accumulators to the epilogue;
//  - warps 2-5: epilogue. Each warp owns one 32-lane quarter of TMEM (= 32
//    rows of the tile), reads 32 columns at a time, transposes them through a
//    padded shared-memory tile so that global stores are row-contiguous, and
//    applies bias / GELU / residual / ReLU / position embedding.
//  Every mbarrier wait is bounded; a timeout records ELASTO_ERR_TIMEOUT.
#include "common.h"
#include "ptx.cuh"

namespace elasto {

namespace {

constexpr int BM = 128, BK = 64, STAGES = 4, MAX_BN = 256, THREADS = 192;
constexpr int A_STAGE = BM * BK * 2;        // 16 KB
constexpr int B_STAGE = MAX_BN * BK * 2;    // 32 KB
constexpr int EPI_LD = 33;                  // padded row of the transpose tile
constexpr int EPI_TILE = 32 * EPI_LD;       // floats per epilogue warp
constexpr int TMEM_COLS = 512;
constexpr size_t SMEM_BYTES = 1024 + STAGES * (A_STAGE + B_STAGE) + 4 * EPI_TILE * 4 + 256;

__device__ __forceinline__ float gelu_erf(float x) { return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f)); }

template <int EPI>
__global__ void __launch_bounds__(THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const GemmArgs args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * A_STAGE;
  float* sEpi = reinterpret_cast<float*>(sB + STAGES * B_STAGE);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sEpi + 4 * EPI_TILE);
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* tfull = bars + 2 * STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int M = args.M, N = args.N, bn = args.bn;
  const int nk = (args.K + BK - 1) / BK;
  const int mt = (M + BM - 1) / BM, nt = (N + bn - 1) / bn;
  const int tiles = mt * nt;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 4);
    }
    mbar_init(drain, 1);
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  if (warp == 1 && lane == 0 && nk > 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0 && nk > 0) {
      int stage = 0;
      uint32_t phase = 0;
      long issued = 0;
      bool ok = true;
      const uint32_t bytes = A_STAGE + bn * BK * 2;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
        const int m0 = (t / nt) * BM, n0 = (t % nt) * bn;
        for (int kb = 0; kb < nk; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1)) {
            ok = false;
            break;
          }
          mbar_expect_tx(&full[stage], bytes);
          tma_load_2d(sA + stage * A_STAGE, &tmA, &full[stage], kb * BK, m0);
          tma_load_2d(sB + stage * B_STAGE, &tmB, &full[stage], kb * BK, n0);
          ++issued;
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (!ok) record_status(args.status, ELASTO_ERR_TIMEOUT);
      // Drain: make sure no copy is still landing in shared memory when the
      // CTA exits (returns at once on the normal path).
      for (int i = 0; i < STAGES && i < issued; ++i) {
        if (stage == 0) {
          stage = STAGES;
          phase ^= 1;
        }
        --stage;
        mbar_wait(&full[stage], phase);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(BM, bn);
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true, issued = false;
      int local = 0;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++local) {
        const int acc = local & 1;
        const uint32_t use = static_cast<uint32_t>(local >> 1);
        if (!mbar_wait(&tempty[acc], (use & 1) ^ 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t dtm = tmem_base + acc * MAX_BN;
        if (nk == 0) {
          mbar_arrive(&tfull[acc]);
          continue;
        }
        for (int kb = 0; kb < nk; ++kb) {
          if (!mbar_wait(&full[stage], phase)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_addr(sA + stage * A_STAGE), b0 = smem_addr(sB + stage * B_STAGE);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            tc_mma(dtm, sdesc_sw128(a0 + k * 32, 16, 1024), sdesc_sw128(b0 + k * 32, 16, 1024), idesc,
                   (kb | k) != 0);
          }
          issued = true;
          tc_commit(&empty[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (ok) tc_commit(&tfull[acc]);
      }
      if (!ok) record_status(args.status, ELASTO_ERR_TIMEOUT);
      // All MMAs this thread issued have finished once `drain` completes.
      if (issued) {
        tc_commit(drain);
        mbar_wait(drain, 0);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    float* st = sEpi + (warp - 2) * EPI_TILE;
    int local = 0;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++local) {
      const int acc = local & 1;
      const uint32_t use = static_cast<uint32_t>(local >> 1);
      if (!mbar_wait(&tfull[acc], use & 1)) {
        if (lane == 0) record_status(args.status, ELASTO_ERR_TIMEOUT);
        break;
      }
      tc_fence_after();
      const int m0 = (t / nt) * BM, n0 = (t % nt) * bn;
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
        if constexpr (EPI == EPI_BIAS_RESID_F32 || EPI == EPI_BIAS_F32 || EPI == EPI_PATCH_POS_F32) {
          const int col = n0 + c + lane;
          const bool cok = col < N;
          const float bv = (cok && args.bias) ? args.bias[col] : 0.0f;
          float* out = static_cast<float*>(args.out);
          if constexpr (EPI == EPI_BIAS_RESID_F32) {
            float old[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int row = row0 + i;
              old[i] = (cok && row < M) ? out[static_cast<size_t>(row) * args.ldo + col] : 0.0f;
            }
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int row = row0 + i;
              if (cok && row < M) out[static_cast<size_t>(row) * args.ldo + col] = old[i] + (st[i * EPI_LD + lane] + bv);
            }
          } else if constexpr (EPI == EPI_BIAS_F32) {
#pragma unroll 8
            for (int i = 0; i < 32; ++i) {
              const int row = row0 + i;
              if (cok && row < M) out[static_cast<size_t>(row) * args.ldo + col] = st[i * EPI_LD + lane] + bv;
            }
          } else {
#pragma unroll 8
            for (int i = 0; i < 32; ++i) {
              const int row = row0 + i;
              if (cok && row < M) {
                const int img = row / args.patches, p = row - img * args.patches;
                const size_t orow = static_cast<size_t>(img) * args.tokens + 1 + p;
                out[orow * args.ldo + col] =
                    (st[i * EPI_LD + lane] + bv) + args.pos[static_cast<size_t>(1 + p) * N + col];
              }
            }
          }
        } else {
          const int cp = (lane & 15) * 2;
          const int col = n0 + c + cp;
          const bool cok = col < N;
          const float b0 = (cok && args.bias) ? args.bias[col] : 0.0f;
          const float b1 = (cok && args.bias) ? args.bias[col + 1] : 0.0f;
          uint32_t* out = static_cast<uint32_t*>(args.out);
#pragma unroll 4
          for (int i = 0; i < 16; ++i) {
            const int rr = 2 * i + (lane >> 4);
            const int row = row0 + rr;
            if (!(cok && row < M)) continue;
            float v0 = st[rr * EPI_LD + cp] + b0;
            float v1 = st[rr * EPI_LD + cp + 1] + b1;
            if constexpr (EPI == EPI_BIAS_GELU_BF16) {
              v0 = gelu_erf(v0);
              v1 = gelu_erf(v1);
            } else if constexpr (EPI == EPI_BIAS_RELU_BF16) {
              v0 = fmaxf(v0, 0.0f);
              v1 = fmaxf(v1, 0.0f);
            } else if constexpr (EPI == EPI_BIAS_RESID_RELU_BF16) {
              const __nv_bfloat162 rv =
                  *reinterpret_cast<const __nv_bfloat162*>(args.resid + static_cast<size_t>(row) * args.ldr + col);
              v0 = fmaxf(v0 + __bfloat162float(rv.x), 0.0f);
              v1 = fmaxf(v1 + __bfloat162float(rv.y), 0.0f);
            }
            out[(static_cast<size_t>(row) * args.ldo + col) >> 1] = pack_bf16x2(v0, v1);
          }
        }
        __syncwarp();
      }
      tc_fence_before();
      if (lane == 0) mbar_arrive(&tempty[acc]);
    }
  }
  __syncthreads();
  if (warp == 0) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

template <int EPI>
cudaError_t launch_epi(const GemmPlan& p, int M, cudaStream_t s) {
  GemmArgs a = p.args;
  a.M = M;
  const int tiles = ((M + BM - 1) / BM) * ((a.N + a.bn - 1) / a.bn);
  const int grid = tiles < num_sms() ? tiles : num_sms();
  gemm_tc_kernel<EPI><<<grid, THREADS, SMEM_BYTES, s>>>(p.tmA, p.tmB, a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t gemm_init_attributes() {
  const int bytes = static_cast<int>(SMEM_BYTES);
  cudaError_t e;
#define SET_ATTR(E)                                                                                     \
  e = cudaFuncSetAttribute(gemm_tc_kernel<E>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);      \
  if (e != cudaSuccess) return e;
  SET_ATTR(EPI_BIAS_BF16)
  SET_ATTR(EPI_BIAS_GELU_BF16)
  SET_ATTR(EPI_BIAS_RESID_F32)
  SET_ATTR(EPI_BIAS_F32)
  SET_ATTR(EPI_BIAS_RELU_BF16)
  SET_ATTR(EPI_BIAS_RESID_RELU_BF16)
  SET_ATTR(EPI_PATCH_POS_F32)
#undef SET_ATTR
  return cudaSuccess;
}

int gemm_pick_bn(int M, int N) {
  // Estimated time ~ waves x (bn + fixed per-tile overhead); ties prefer wider tiles.
  const int sms = num_sms() > 0 ? num_sms() : 148;
  const int mt = (M + BM - 1) / BM;
  int best = 256;
  long best_cost = -1;
  for (int bn = 256; bn >= 32; bn -= 32) {
    const long tiles = static_cast<long>(mt) * ((N + bn - 1) / bn);
    const long waves = (tiles + sms - 1) / sms;
    const long cost = waves * (bn + 32);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = bn;
    }
  }
  return best;
}

elasto_status gemm_plan(GemmPlan* p, const bf16* A, int M_cap, const bf16* W, int N, int K, const float* bias,
                        void* out, int ldo, int epi, int* status) {
  if (!p || M_cap <= 0 || N <= 0 || K < 0 || !out || (K > 0 && (!A || !W))) {
    set_error("gemm_plan: invalid arguments");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (K % 8 != 0 || N % 2 != 0) {
    set_error("gemm: K must be a multiple of 8 and N even");
    return ELASTO_ERR_UNSUPPORTED;
  }
  *p = GemmPlan{};
  GemmArgs& a = p->args;
  a.M = M_cap;
  a.N = N;
  a.K = K;
  a.bn = gemm_pick_bn(M_cap, N);
  a.bias = bias;
  a.out = out;
  a.ldo = ldo;
  a.status = status;
  p->epi = epi;
  if (K > 0) {
    if (!encode_tmap_2d(&p->tmA, A, K, M_cap, static_cast<uint64_t>(K) * 2, BK, BM) ||
        !encode_tmap_2d(&p->tmB, W, K, N, static_cast<uint64_t>(K) * 2, BK, a.bn)) {
      set_error("gemm_plan: cuTensorMapEncodeTiled failed (alignment or size)");
      return ELASTO_ERR_UNSUPPORTED;
    }
  }
  p->valid = true;
  return ELASTO_OK;
}

cudaError_t gemm_launch(const GemmPlan& p, int M, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  switch (p.epi) {
    case EPI_BIAS_BF16: return launch_epi<EPI_BIAS_BF16>(p, M, s);
    case EPI_BIAS_GELU_BF16: return launch_epi<EPI_BIAS_GELU_BF16>(p, M, s);
    case EPI_BIAS_RESID_F32: return launch_epi<EPI_BIAS_RESID_F32>(p, M, s);
    case EPI_BIAS_F32: return launch_epi<EPI_BIAS_F32>(p, M, s);
    case EPI_BIAS_RELU_BF16: return launch_epi<EPI_BIAS_RELU_BF16>(p, M, s);
    case EPI_BIAS_RESID_RELU_BF16: return launch_epi<EPI_BIAS_RESID_RELU_BF16>(p, M, s);
    case EPI_PATCH_POS_F32: return launch_epi<EPI_PATCH_POS_F32>(p, M, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace elasto
