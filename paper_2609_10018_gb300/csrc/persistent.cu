// One-launch forward of one image: the whole DN forward of Section 4.1 (patch
// projection, every layer's Eq. 2-6 over the kept heads and MLP channels,
// final norm and classifier) as the phases of a single persistent
// cooperative kernel, one CTA per SM.
//
// Why: at one image every operation is a few microseconds of work, and as
// separate kernels the forward is ~88 dependent launches whose ramp-up, first
// loads and tails dominate (Section 6.2 measures DNs at batch 1). Here a phase
// ends with a grid-wide barrier (a counter in global memory, waits bounded in
// time), and the next phase's weights are already on their way into shared
// memory while the CTA waits at it: weights never depend on the previous phase.
//
// Phases (host plan, one per mode):
//   PATCH   image -> patch rows P [n, P*P*C] bf16 (row 0: the class token slot, zeros)
//   GEMM    out = epi(A . W^T) over 128 x bn tiles and ks k-splits: bf16 with
//           bias (QKV), bf16 with bias and GELU (FC1), or fp32 partial sums
//           of a k-split (patch projection, out-projection, FC2)
//   ATTN    one (kept head, 128-query tile) per unit: S = Q K^T, softmax, O = P V
//   REDUCE  one row per warp: X = base + (sum of the partials in split
//           order + bias), then the LayerNorm that follows (or, after the
//           last layer, the final norm of the class-token row in fp32)
//   HEAD    one class per warp: logits = LN(x_cls) . W_head^T + b_head
//
// Roles (320 threads):
//   warp 0 lane 0  TMA producer: a unit's B (weight) k-blocks all at once into
//                  the B region, A k-blocks through a 7-stage ring; attention
//                  Q, K, V into buffers that alias the ring. At the end of a
//                  phase it already loads the B of its first unit of the next
//                  GEMM phase.
//   warp 1 lane 0  tcgen05.mma issuer (M = 128); warp 1 owns the TMEM (512 columns)
//   warps 2-9      two groups of four (TMEM lane quarter = warp & 3): GEMM
//                  epilogue (each group half of the tile's columns), softmax
//                  (two threads per query row, each half of the keys, row max
//                  and sum exchanged through shared memory), REDUCE / HEAD /
//                  PATCH work.
// TMEM: GEMM accumulator in columns [0, bn); attention S in [0, n_pad), P (bf16
// pairs) in [256, 256 + n_pad / 2), O in [384, 448).
// Shared memory: [A ring 7 x 16 KB | B region 72 KB | output staging 8 x 4 KB |
// barriers, exchange, the current and next phase descriptors]. Outputs
// (GEMM tiles, attention O) leave by TMA stores of 32-row boxes staged per
// warp (128-byte rows in the 128-byte swizzle).
//
// Memory ordering across phases: a phase's results are written by TMA stores
// (waited for until complete before the barrier) or ordinary stores; every
// thread fences against the async proxy (the TMA reads and writes on either
// side), the CTA synchronises, one thread releases its arrival and acquires
// everyone's; the TMA issuer fences again before its first load of the
// phase. Data written inside the kernel is never read through the
// non-coherent cache.
//
// Every wait (mbarrier or grid counter) is bounded; one that gives up records
// ELASTO_ERR_TIMEOUT in the status word and raises an abort flag that every
// other CTA sees at its next barrier, so the launch always ends.
#include <algorithm>
#include <string>
#include <vector>

#include "act.cuh"
#include "common.h"
#include "handle.h"
#include "ptx.cuh"

namespace elasto {

enum PkKind : int { PK_PATCH = 0, PK_GEMM = 1, PK_ATTN = 2, PK_REDUCE = 3, PK_HEAD = 4 };
enum PkEpi : int { PKE_BF16 = 0, PKE_GELU = 1, PKE_PART = 2 };

// One phase; the fields a kind does not use stay zero.
struct PkPhase {
  int kind = 0, units = 0;
  // GEMM: unit u -> split u / (mt * nt), tile u % (mt * nt) (M tile fastest)
  int epi = 0, mt = 0, nt = 0, ks = 1, bn = 0, nk = 0, N = 0, ldo = 0;
  int mapA = 0, mapB = 0, mapC = 0;  // mapC: the output, unswizzled, box (bn / 2) x 32 rows (x 1 split)
  const float* bias = nullptr;  // GEMM bias [N]; REDUCE bias [d]
  void* out = nullptr;          // GEMM output [rows, ldo] (bf16, or fp32 partials split_stride apart)
  long long split_stride = 0;   // elements between two splits' partial sums
  // ATTN
  int mapQ = 0, mapKV = 0, mapO = 0, n_pad = 0, heads = 0, tiles = 0, blk_stride = 0, head_stride = 0, w = 0;
  bf16* o = nullptr;  // [n, w] (mapO: unswizzled, box 32 x 32 rows)
  // REDUCE (ks and split_stride as above)
  const float* part = nullptr;  // partial sums [ks][n][d]
  const float* xsrc = nullptr;  // base rows instead of X (the patch projection's per-token addend)
  float* X = nullptr;           // residual stream [n, d]
  const float* g = nullptr;     // LayerNorm -> y (null: none)
  const float* b = nullptr;
  bf16* y = nullptr;
  const float* fg = nullptr;    // final norm of row 0 -> y32 (null: none)
  const float* fb = nullptr;
  float* y32 = nullptr;
  int d = 0, d_true = 0;        // row width (multiple of 64) and kept channels
  // PATCH
  int img_dtype = 0, img_h = 0, img_w = 0, img_c = 0, patch = 0, kpe = 0;
  bf16* prow = nullptr;         // [n, kpe]
  // HEAD (reads y32)
  const float* hw = nullptr;    // [classes, d]
  const float* hb = nullptr;
  int classes = 0;
};

namespace {

constexpr int PK_THREADS = 320;
constexpr int PK_STAGES = 7;
constexpr int PK_A_STAGE = 128 * 64 * 2;          // 16 KB
constexpr int PK_RING = PK_STAGES * PK_A_STAGE;   // 112 KB
constexpr int PK_B_BYTES = 72 * 1024;             // all B k-blocks of one GEMM unit
constexpr int PK_STG_WARP = 4096;                 // output staging of one epilogue warp (32 rows x 128 B)
constexpr int PK_STG_BYTES = 8 * PK_STG_WARP;
constexpr int PK_BAR_BYTES = 4096;                // barriers, TMEM slot, softmax exchange, phase slots
constexpr int PK_PHASE_OFF = 2304;                // two phase descriptors after the exchange arrays
constexpr int PK_SMEM = 1024 + PK_RING + PK_B_BYTES + PK_STG_BYTES + PK_BAR_BYTES;
constexpr int PK_TMEM_COLS = 512;
constexpr int PK_P_COL = 256, PK_O_COL = 384;
constexpr int PK_HD = 64;                         // head width
constexpr int PK_MAX_BN = 64;                     // epilogue: <= 32 columns per group
static_assert(PK_SMEM <= 232448, "one-launch forward shared memory");
static_assert(PK_PHASE_OFF + 2 * sizeof(PkPhase) <= PK_BAR_BYTES && sizeof(PkPhase) % 4 == 0 &&
                  PK_PHASE_OFF % alignof(PkPhase) == 0 && sizeof(PkPhase) % alignof(PkPhase) == 0,
              "phase slots");

// Copy descriptor `src` (global) into `dst` (shared) with nthr threads, thread t of them.
__device__ __forceinline__ void copy_phase(PkPhase* dst, const PkPhase* src, int t, int nthr) {
  const uint32_t* s = reinterpret_cast<const uint32_t*>(src);
  uint32_t* d = reinterpret_cast<uint32_t*>(dst);
  for (int i = t; i < static_cast<int>(sizeof(PkPhase) / 4); i += nthr) d[i] = __ldg(s + i);
}

// Attention buffers inside the ring: Q (16 KB), K and V (n_pad rows of 128 B each)
constexpr int PK_Q_OFF = 0, PK_K_OFF = 16384, PK_V_OFF = 16384 + 256 * 128;
static_assert(PK_V_OFF + 256 * 128 <= PK_RING, "attention buffers fit the ring");

__device__ __forceinline__ void tma_store_3d(const CUtensorMap* tm, const void* src, int x, int y, int z) {
  asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(tm)),
               "r"(smem_addr(src)), "r"(x), "r"(y), "r"(z)
               : "memory");
}

// One thread's row piece (nch <= 8 chunks of 16 bytes) into its warp's
// staging box of 32 such rows, the layout the TMA store reads: dense rows,
// and for 128-byte rows the 128-byte swizzle (chunk c of row r at c ^ (r % 8),
// the box 1024-byte aligned), which also keeps the 32 threads' stores on
// distinct banks.
__device__ __forceinline__ void stage_row(uint8_t* box, int lane, int nch, const uint32_t (&words)[32]) {
  uint8_t* row = box + lane * nch * 16;
  const int x = nch == 8 ? (lane & 7) : 0;
#pragma unroll
  for (int c = 0; c < 8; ++c)
    if (c < nch)
      *reinterpret_cast<uint4*>(row + ((c ^ x) * 16)) =
          make_uint4(words[4 * c], words[4 * c + 1], words[4 * c + 2], words[4 * c + 3]);
}

__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}
__device__ __forceinline__ void red_release_add(unsigned* p, unsigned v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ unsigned ld_acquire(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ unsigned ld_relaxed(const unsigned* p) {
  unsigned v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// A wait gave up: record it and make every CTA leave at its next barrier.
__device__ __forceinline__ void pk_fail(int* status, unsigned* sync) {
  record_status(status, ELASTO_ERR_TIMEOUT);
  atomicExch(sync + 1, 1u);
}

__device__ __forceinline__ float pk_warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Grid-wide barrier number `index` (0, 1, ...): sync[0] counts arrivals. False
// when a thread of this CTA failed (s_fail), the abort flag sync[1] is up or
// the wait gave up.
__device__ __forceinline__ bool grid_sync(unsigned* sync, unsigned index, int* status, int* s_ok,
                                          const int* s_fail) {
  tc_fence_before();
  fence_proxy_async_global();
  __syncthreads();
  if (threadIdx.x == 64) {
    bool ok = *s_fail == 0;
    __threadfence();
    red_release_add(sync, 1u);
    const unsigned target = (index + 1) * gridDim.x;
    if (ok && ld_acquire(sync) < target) {
      const uint64_t t0 = global_timer_ns();
      for (;;) {
        if (ld_acquire(sync) >= target) break;
        if (ld_relaxed(sync + 1) != 0u) {
          ok = false;
          break;
        }
        if (global_timer_ns() - t0 > kWaitLimitNs) {
          pk_fail(status, sync);
          ok = false;
          break;
        }
        __nanosleep(32);
      }
    }
    if (ld_relaxed(sync + 1) != 0u) ok = false;
    fence_proxy_async_global();
    *s_ok = ok ? 1 : 0;
  }
  __syncthreads();
  tc_fence_after();
  return *s_ok != 0;
}

// A GEMM unit; its k-blocks run in the order kb0 + (j + rot) % (kb1 - kb0),
// j = 0, 1, ...: units that start together read different k-blocks of the
// A operand they share (no pile-up of every SM on the same L2 lines).
struct PkUnit {
  int m0, n0, kb0, kb1, split, rot;
  __device__ __forceinline__ int kb(int j) const {
    const int nkb = kb1 - kb0, r = j + rot;
    return kb0 + (r >= nkb ? r - nkb : r);
  }
};
__device__ __forceinline__ PkUnit gemm_unit(const PkPhase& ph, int u) {
  const int tiles = ph.mt * ph.nt;
  const int split = u / tiles, t = u - split * tiles;
  PkUnit r;
  r.m0 = (t % ph.mt) * 128;
  r.n0 = (t / ph.mt) * ph.bn;
  r.kb0 = split * ph.nk / ph.ks;
  r.kb1 = (split + 1) * ph.nk / ph.ks;
  r.split = split;
  r.rot = (t / ph.mt) % (r.kb1 - r.kb0);
  return r;
}

}  // namespace

}  // namespace elasto
// ---------------------------------------------------------------- kernel
namespace elasto {
namespace {

__global__ void __launch_bounds__(PK_THREADS, 1)
    dn_one_kernel(const PkPhase* __restrict__ phases, int n_phases, const CUtensorMap* maps, int n_maps,
                  const unsigned long long* __restrict__ pf_lines, int n_pf, int n, const void* __restrict__ images,
                  float* __restrict__ logits, unsigned* sync, int* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* ring = smem;              // A stages; the attention buffers alias it
  uint8_t* bbuf = smem + PK_RING;    // the current GEMM unit's B k-blocks
  uint8_t* stg = bbuf + PK_B_BYTES;  // output staging, 4 KB per epilogue warp
  uint64_t* bars = reinterpret_cast<uint64_t*>(stg + PK_STG_BYTES);
  uint64_t* afull = bars;                  // [PK_STAGES] A stage landed
  uint64_t* aempty = bars + PK_STAGES;     // [PK_STAGES] A stage read by the MMAs
  uint64_t* bfull = bars + 2 * PK_STAGES;  // B region landed
  uint64_t* bempty = bfull + 1;            // B region's MMAs finished
  uint64_t* tfull = bfull + 2;             // accumulator complete
  uint64_t* tempty = bfull + 3;            // accumulator read out (8 warps)
  uint64_t* at_full = bfull + 4;           // Q, K, V landed
  uint64_t* at_empty = bfull + 5;          // attention buffers free again
  uint64_t* s_full = bfull + 6;            // S in TMEM
  uint64_t* p_full = bfull + 7;            // P in TMEM (8 warps)
  uint64_t* o_full = bfull + 8;            // O in TMEM
  uint64_t* o_empty = bfull + 9;           // O read out (8 warps)
  uint64_t* drain = bfull + 10;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bfull + 11);
  int* s_ok = reinterpret_cast<int*>(bfull + 12);
  int* s_fail = s_ok + 1;  // a thread of this CTA gave up a wait
  float* xmax = reinterpret_cast<float*>(bfull + 16);  // [2][128] per-group row maxima
  float* xsum = xmax + 256;                            // [2][128] per-group row sums
  // the current and the next phase's descriptor (copied from global memory
  // one phase ahead, so that no role starts a phase with a global load)
  PkPhase* sphase = reinterpret_cast<PkPhase*>(reinterpret_cast<uint8_t*>(bars) + PK_PHASE_OFF);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < PK_STAGES; ++s) {
      mbar_init(&afull[s], 1);
      mbar_init(&aempty[s], 1);
    }
    mbar_init(bfull, 1);
    mbar_init(bempty, 1);
    mbar_init(tfull, 1);
    mbar_init(tempty, 8);
    mbar_init(at_full, 1);
    mbar_init(at_empty, 1);
    mbar_init(s_full, 1);
    mbar_init(p_full, 8);
    mbar_init(o_full, 1);
    mbar_init(o_empty, 8);
    mbar_init(drain, 1);
    fence_barrier_init();
    *s_fail = 0;
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, PK_TMEM_COLS);
    tmem_relinquish();
  }
  if (warp == 0)
    for (int i = lane; i < n_maps; i += 32) tma_prefetch_desc(&maps[i]);
  if (warp >= 2 && n_phases > 0) copy_phase(&sphase[0], &phases[0], threadIdx.x - 64, PK_THREADS - 64);
  // the small parameters every CTA reads (biases, LayerNorm weights) into L2
  // now, so that no phase waits on DRAM for them
  for (int i = blockIdx.x * PK_THREADS + threadIdx.x; i < n_pf; i += gridDim.x * PK_THREADS)
    asm volatile("prefetch.global.L2::evict_last [%0];" ::"l"(pf_lines[i]) : "memory");
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // per-role pipeline state, carried across phases
  int p_ast = 0, m_ast = 0;         // A ring stage (producer, MMA issuer)
  uint32_t p_aph = 0, m_aph = 0;    // and its phase bit
  uint32_t p_nb = 0, m_nb = 0;      // B region loads / uses
  uint32_t p_na = 0, m_na = 0, e_na = 0;  // attention units
  uint32_t m_nacc = 0, e_nacc = 0;  // accumulator uses
  long p_issued = 0;                // A stages loaded
  bool m_issued = false;
  int pre_unit = -1;                // unit of this phase whose B was loaded during the last barrier
  bool ok = true;
  const int grp = (warp - 2) >> 2, quarter = warp & 3;  // warps 2-9
  const uint32_t lane_base = tmem + (static_cast<uint32_t>(quarter * 32) << 16);

  // all B k-blocks of GEMM unit `un` of phase `ph` into the B region
  auto load_b = [&](const PkPhase& ph, const PkUnit& un) -> bool {
    if (!mbar_wait(bempty, (p_nb & 1) ^ 1)) return false;
    const int nkb = un.kb1 - un.kb0, tile = ph.bn * 128;
    mbar_expect_tx(bfull, static_cast<uint32_t>(nkb * tile));
    for (int j = 0; j < nkb; ++j) tma_load_2d(bbuf + j * tile, &maps[ph.mapB], bfull, (un.kb0 + j) * 64, un.n0);
    ++p_nb;
    return true;
  };

  for (int p = 0; p < n_phases; ++p) {
    const PkPhase& ph = sphase[p & 1];
    const int kind = ph.kind;
    // lanes 1-31 of warp 0 (idle in every role) fetch the next descriptor
    if (warp == 0 && lane > 0 && p + 1 < n_phases) copy_phase(&sphase[(p + 1) & 1], &phases[p + 1], lane - 1, 31);
    if (kind == PK_GEMM) {
      if (warp == 0) {
        // ------------------------------------------------ producer
        if (lane == 0 && ok) {
          fence_proxy_async_global();
          for (int u = blockIdx.x; u < ph.units && ok; u += gridDim.x) {
            const PkUnit un = gemm_unit(ph, u);
            if (u != pre_unit && !load_b(ph, un)) {
              ok = false;
              break;
            }
            for (int j = 0; j < un.kb1 - un.kb0; ++j) {
              if (!mbar_wait(&aempty[p_ast], p_aph ^ 1)) {
                ok = false;
                break;
              }
              mbar_expect_tx(&afull[p_ast], PK_A_STAGE);
              tma_load_2d(ring + p_ast * PK_A_STAGE, &maps[ph.mapA], &afull[p_ast], un.kb(j) * 64, un.m0);
              ++p_issued;
              if (++p_ast == PK_STAGES) {
                p_ast = 0;
                p_aph ^= 1;
              }
            }
          }
        }
      } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0 && ok) {
          const uint32_t idesc = idesc_bf16_f32(128, ph.bn);
          const int tile = ph.bn * 128;
          for (int u = blockIdx.x; u < ph.units && ok; u += gridDim.x) {
            const PkUnit un = gemm_unit(ph, u);
            if (!mbar_wait(bfull, m_nb & 1) || !mbar_wait(tempty, (m_nacc & 1) ^ 1)) {
              ok = false;
              break;
            }
            tc_fence_after();
            for (int j = 0; j < un.kb1 - un.kb0; ++j) {
              if (!mbar_wait(&afull[m_ast], m_aph)) {
                ok = false;
                break;
              }
              tc_fence_after();
              const uint32_t a0 = smem_addr(ring + m_ast * PK_A_STAGE),
                             b0 = smem_addr(bbuf + (un.kb(j) - un.kb0) * tile);
#pragma unroll
              for (int k = 0; k < 4; ++k)
                tc_mma(tmem, sdesc_sw128(a0 + k * 32, 16, 1024), sdesc_sw128(b0 + k * 32, 16, 1024), idesc,
                       (j != 0 || k != 0) ? 1u : 0u);
              tc_commit(&aempty[m_ast]);
              if (++m_ast == PK_STAGES) {
                m_ast = 0;
                m_aph ^= 1;
              }
            }
            if (!ok) break;
            tc_commit(tfull);
            tc_commit(bempty);
            ++m_nb;
            ++m_nacc;
            m_issued = true;
          }
        }
      } else {
        // ------------------------------------------------ epilogue: half of the tile's columns per group
        const int half = ph.bn >> 1, c0 = grp * half;
        for (int u = blockIdx.x; u < ph.units && ok; u += gridDim.x) {
          const PkUnit un = gemm_unit(ph, u);
          // lane l holds the bias of column c0 + l of the unit (loaded while the MMAs run)
          const int bcol = un.n0 + c0 + lane;
          const float bias_l = (ph.epi != PKE_PART && lane < half && bcol < ph.N) ? __ldg(ph.bias + bcol) : 0.0f;
          const bool got = __all_sync(0xffffffffu, mbar_wait(tfull, e_nacc & 1));
          ++e_nacc;
          if (!got) {
            ok = false;
            break;
          }
          tc_fence_after();
          // all of this thread's columns (<= 32) with one TMEM wait; the
          // accumulator is free again as soon as they are in registers
          uint32_t v[32];
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (8 * j < half) tmem_ld_8(lane_base + c0 + 8 * j, *reinterpret_cast<uint32_t(*)[8]>(v + 8 * j));
          tmem_ld_wait();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(tempty);
          // bf16 outputs: bias (and GELU) and pack, two columns per word
          if (ph.epi != PKE_PART) {
#pragma unroll
            for (int e = 0; e < 16; ++e)
              if (2 * e < half) {
                float lo = __uint_as_float(v[2 * e]) + __shfl_sync(0xffffffffu, bias_l, 2 * e);
                float hi = __uint_as_float(v[2 * e + 1]) + __shfl_sync(0xffffffffu, bias_l, 2 * e + 1);
                if (ph.epi == PKE_GELU) {
                  lo = gelu(lo);
                  hi = gelu(hi);
                }
                v[e] = pack_bf16x2(lo, hi);
              }
          }
          // row pieces -> this warp's staging box -> one TMA store of 32 rows
          // (rows past n and columns past N are clipped by the map)
          uint8_t* box = stg + (warp - 2) * PK_STG_WARP;
          if (lane == 0) bulk_wait_read_all();  // the box's previous store has read it
          __syncwarp();
          stage_row(box, lane, ph.epi == PKE_PART ? half / 4 : half / 8, v);
          fence_async_smem();
          __syncwarp();
          if (lane == 0) {
            const int col = un.n0 + c0, r0 = un.m0 + quarter * 32;
            if (ph.epi == PKE_PART)
              tma_store_3d(&maps[ph.mapC], box, col, r0, un.split);
            else
              tma_store_2d(&maps[ph.mapC], box, col, r0);
            bulk_commit();
          }
        }
      }
    }
    else if (kind == PK_ATTN) {
      if (warp == 0) {
        // ------------------------------------------------ producer: K, V of the head, its query tile
        if (lane == 0 && ok) {
          fence_proxy_async_global();
          const uint32_t bytes = PK_A_STAGE + 2 * ph.n_pad * 128;
          for (int u = blockIdx.x; u < ph.units && ok; u += gridDim.x) {
            const int j = u / ph.tiles, t = u - j * ph.tiles;
            if (!mbar_wait(at_empty, (p_na & 1) ^ 1)) {
              ok = false;
              break;
            }
            mbar_expect_tx(at_full, bytes);
            const int qx = j * ph.head_stride;
            tma_load_2d(ring + PK_K_OFF, &maps[ph.mapKV], at_full, qx + ph.blk_stride, 0);
            tma_load_2d(ring + PK_V_OFF, &maps[ph.mapKV], at_full, qx + 2 * ph.blk_stride, 0);
            tma_load_2d(ring + PK_Q_OFF, &maps[ph.mapQ], at_full, qx, t * 128);
            ++p_na;
          }
        }
      } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer: S = Q K^T, then O = P V (P from TMEM)
        if (lane == 0 && ok) {
          const uint32_t idesc_s = idesc_bf16_f32(128, ph.n_pad);
          const uint32_t idesc_o = idesc_bf16_f32(128, PK_HD, false, true);
          const uint32_t q0 = smem_addr(ring + PK_Q_OFF), k0 = smem_addr(ring + PK_K_OFF),
                         v0 = smem_addr(ring + PK_V_OFF);
          for (int u = blockIdx.x; u < ph.units && ok; u += gridDim.x) {
            if (!mbar_wait(at_full, m_na & 1) || !mbar_wait(o_empty, (m_na & 1) ^ 1)) {
              ok = false;
              break;
            }
            tc_fence_after();
#pragma unroll
            for (int kk = 0; kk < PK_HD / 16; ++kk)
              tc_mma(tmem, sdesc_sw128(q0 + kk * 32, 16, 1024), sdesc_sw128(k0 + kk * 32, 16, 1024), idesc_s,
                     kk != 0 ? 1u : 0u);
            tc_commit(s_full);
            m_issued = true;
            if (!mbar_wait(p_full, m_na & 1)) {
              ok = false;
              break;
            }
            tc_fence_after();
            for (int s = 0; s < ph.n_pad / 16; ++s)
              tc_mma_tmem_a(tmem + PK_O_COL, tmem + PK_P_COL + 8 * s, sdesc_sw128(v0 + s * 16 * 128, 16384, 1024),
                            idesc_o, s != 0 ? 1u : 0u);
            tc_commit(o_full);
            tc_commit(at_empty);
            ++m_na;
          }
        }
      } else {
        // ------------------------------------------------ softmax (two threads per row) and O read-out
        const float kscale = 0.125f * 1.4426950408889634f;  // 1/sqrt(64) * log2(e)
        const int n_read = (n + 63) & ~63, half = n_read >> 1, cb = grp * half;
        const int r = quarter * 32 + lane;  // query row within the tile
        for (int u = blockIdx.x; u < ph.units; u += gridDim.x) {
          const int j = u / ph.tiles, t = u - j * ph.tiles;
          const bool active = t * 128 + quarter * 32 < n;  // some row of this warp is a real query
          bool good = ok && __all_sync(0xffffffffu, mbar_wait(s_full, e_na & 1));
          tc_fence_after();
          float mx = -INFINITY;
          if (active && good) {
            for (int c = cb; c < cb + half; c += 32) {
              uint32_t v[32];
              tmem_ld_32x32b_x32(lane_base + c, v);
              tmem_ld_wait();
#pragma unroll
              for (int jj = 0; jj < 32; ++jj)
                if (c + jj < n) mx = fmaxf(mx, __uint_as_float(v[jj]));
            }
          }
          xmax[grp * 128 + r] = mx;
          named_bar_sync(1, 256);
          mx = fmaxf(xmax[r], xmax[128 + r]);
          float sum = 0.0f;
          if (active && good) {
            const float mxs = mx * kscale;
            for (int c = cb; c < cb + half; c += 32) {
              uint32_t v[32], pk[16];
              tmem_ld_32x32b_x32(lane_base + c, v);
              tmem_ld_wait();
#pragma unroll
              for (int jj = 0; jj < 32; jj += 2) {
                const float p0 = (c + jj < n) ? ex2_approx(fmaf(__uint_as_float(v[jj]), kscale, -mxs)) : 0.0f;
                const float p1 =
                    (c + jj + 1 < n) ? ex2_approx(fmaf(__uint_as_float(v[jj + 1]), kscale, -mxs)) : 0.0f;
                sum += p0 + p1;
                pk[jj >> 1] = pack_bf16x2(p0, p1);
              }
              tmem_st_16(lane_base + PK_P_COL + (c >> 1), pk);
            }
            tmem_st_wait();
          }
          xsum[grp * 128 + r] = sum;
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(p_full);
          named_bar_sync(1, 256);
          const float total = xsum[r] + xsum[128 + r];
          good = good && __all_sync(0xffffffffu, mbar_wait(o_full, e_na & 1));
          tc_fence_after();
          uint32_t o[32];
          if (active && good) {
            tmem_ld_32x32b_x32(lane_base + PK_O_COL + grp * 32, o);
            tmem_ld_wait();
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(o_empty);
          if (active && good) {
            // O row * (1 / row sum) -> bf16 -> staging box -> one TMA store of 32 rows x 32 columns
            const float inv = 1.0f / total;
#pragma unroll
            for (int q = 0; q < 16; ++q)
              o[q] = pack_bf16x2(__uint_as_float(o[2 * q]) * inv, __uint_as_float(o[2 * q + 1]) * inv);
            uint8_t* box = stg + (warp - 2) * PK_STG_WARP;
            if (lane == 0) bulk_wait_read_all();
            __syncwarp();
            stage_row(box, lane, 4, o);
            fence_async_smem();
            __syncwarp();
            if (lane == 0) {
              tma_store_2d(&maps[ph.mapO], box, j * PK_HD + grp * 32, t * 128 + quarter * 32);
              bulk_commit();
            }
          }
          ++e_na;
          if (!good) ok = false;
        }
      }
    } else if (kind == PK_REDUCE) {
      // -------------------------------------------------- rows blockIdx.x + j * gridDim.x of this CTA, one
      // at a time over warps 2-9: four channels per thread, every load of
      // the row issued before the first is used (one memory round trip)
      if (warp >= 2) {
        const int d = ph.d, q = threadIdx.x - 64, nw = 8;
        const bool has = 4 * q < d;
        const float inv_d = 1.0f / static_cast<float>(ph.d_true), pad = static_cast<float>(d - ph.d_true);
        for (int row = blockIdx.x; row < n; row += gridDim.x) {
          const size_t base = static_cast<size_t>(row) * d;
          const float* xs = ph.xsrc ? ph.xsrc + base : ph.X + base;
          float4 pp[kSplitMax], old = make_float4(0.f, 0.f, 0.f, 0.f), bb = old;
          if (has) {
#pragma unroll
            for (int sp = 0; sp < kSplitMax; ++sp)
              if (sp < ph.ks) pp[sp] = *reinterpret_cast<const float4*>(ph.part + sp * ph.split_stride + base + 4 * q);
            old = *reinterpret_cast<const float4*>(xs + 4 * q);
            if (ph.bias) bb = __ldg(reinterpret_cast<const float4*>(ph.bias + 4 * q));
          }
          float4 x = old;
          float sum = 0.0f;
          if (has) {
            // x_old + (sum of the partials in split order + bias)
            float4 acc = ph.ks > 0 ? pp[0] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int sp = 1; sp < kSplitMax; ++sp)
              if (sp < ph.ks) {
                acc.x += pp[sp].x;
                acc.y += pp[sp].y;
                acc.z += pp[sp].z;
                acc.w += pp[sp].w;
              }
            x = make_float4(old.x + (acc.x + bb.x), old.y + (acc.y + bb.y), old.z + (acc.z + bb.z),
                            old.w + (acc.w + bb.w));
            *reinterpret_cast<float4*>(ph.X + base + 4 * q) = x;
            sum = (x.x + x.y) + (x.z + x.w);
          }
          if (ph.g || (ph.fg && row == 0)) {
            sum = pk_warp_sum(sum);
            if (lane == 0) xmax[warp - 2] = sum;
            named_bar_sync(2, 256);
            float tot = 0.0f;
#pragma unroll
            for (int w = 0; w < nw; ++w) tot += xmax[w];
            const float mean = tot * inv_d;
            const float a0 = x.x - mean, a1 = x.y - mean, a2 = x.z - mean, a3 = x.w - mean;
            float ss = has ? (a0 * a0 + a1 * a1) + (a2 * a2 + a3 * a3) : 0.0f;
            ss = pk_warp_sum(ss);
            if (lane == 0) xsum[warp - 2] = ss;
            named_bar_sync(2, 256);
            float tss = 0.0f;
#pragma unroll
            for (int w = 0; w < nw; ++w) tss += xsum[w];
            const float rstd = rsqrtf((tss - pad * mean * mean) * inv_d + 1e-6f);
            if (has && ph.g) {
              const float4 gg = __ldg(reinterpret_cast<const float4*>(ph.g + 4 * q));
              const float4 be = __ldg(reinterpret_cast<const float4*>(ph.b + 4 * q));
              *reinterpret_cast<uint2*>(ph.y + base + 4 * q) =
                  make_uint2(pack_bf16x2(a0 * rstd * gg.x + be.x, a1 * rstd * gg.y + be.y),
                             pack_bf16x2(a2 * rstd * gg.z + be.z, a3 * rstd * gg.w + be.w));
            }
            if (has && ph.fg && row == 0) {
              const float4 gg = __ldg(reinterpret_cast<const float4*>(ph.fg + 4 * q));
              const float4 be = __ldg(reinterpret_cast<const float4*>(ph.fb + 4 * q));
              *reinterpret_cast<float4*>(ph.y32 + 4 * q) = make_float4(
                  a0 * rstd * gg.x + be.x, a1 * rstd * gg.y + be.y, a2 * rstd * gg.z + be.z, a3 * rstd * gg.w + be.w);
            }
          }
        }
      }
    } else if (kind == PK_PATCH) {
      // -------------------------------------------------- patch rows, 8 values per thread (warps 2-9)
      if (warp >= 2) {
        const int P = ph.patch, C = ph.img_c, W = ph.img_w, K = ph.kpe, gw = W / P, pcs = K / 8;
        const int total = n * pcs;
        for (int i = (warp - 2) * 32 + lane + blockIdx.x * 256; i < total; i += 256 * gridDim.x) {
          const int row = i / pcs, k0 = (i - row * pcs) * 8;
          uint32_t w4[4] = {0u, 0u, 0u, 0u};
          if (row > 0) {
            const int pt = row - 1, y0 = (pt / gw) * P, x0 = (pt % gw) * P;
            float f[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const int k = k0 + e, ky = k / (P * C), rem = k - ky * (P * C), kx = rem / C, c = rem - kx * C;
              const size_t idx = (static_cast<size_t>(y0 + ky) * W + x0 + kx) * C + c;
              f[e] = ph.img_dtype == ELASTO_BF16 ? __bfloat162float(static_cast<const bf16*>(images)[idx])
                                                 : static_cast<const float*>(images)[idx];
            }
#pragma unroll
            for (int e = 0; e < 4; ++e) w4[e] = pack_bf16x2(f[2 * e], f[2 * e + 1]);
          }
          *reinterpret_cast<uint4*>(ph.prow + static_cast<size_t>(row) * K + k0) = make_uint4(w4[0], w4[1], w4[2], w4[3]);
        }
      }
    } else if (kind == PK_HEAD) {
      // -------------------------------------------------- one class per warp (warps 2-9)
      if (warp >= 2) {
        const int nwarps = 8 * gridDim.x, d = ph.d;
        for (int c = (warp - 2) * gridDim.x + blockIdx.x; c < ph.classes; c += nwarps) {
          const float* wr = ph.hw + static_cast<size_t>(c) * d;
          float s = 0.0f;
          for (int k = lane * 4; k < d; k += 128) {
            const float4 wv = __ldg(reinterpret_cast<const float4*>(wr + k));
            const float4 yv = *reinterpret_cast<const float4*>(ph.y32 + k);
            s += wv.x * yv.x + wv.y * yv.y + wv.z * yv.z + wv.w * yv.w;
          }
          s = pk_warp_sum(s);
          if (lane == 0) logits[c] = s + __ldg(ph.hb + c);
        }
      }
    }
    // the producer starts the weights of its first unit of the next GEMM phase
    // this phase's TMA stores have landed before the barrier releases them
    if (warp >= 2 && lane == 0) bulk_wait_all();
    if (warp == 0) __syncwarp();  // the next descriptor is in shared memory
    if (warp == 0 && lane == 0) {
      pre_unit = -1;
      if (ok && p + 1 < n_phases) {
        const PkPhase& nx = sphase[(p + 1) & 1];
        if (nx.kind == PK_GEMM && static_cast<int>(blockIdx.x) < nx.units) {
          if (load_b(nx, gemm_unit(nx, blockIdx.x)))
            pre_unit = blockIdx.x;
          else
            ok = false;
        }
      }
    }
    if (!ok) {
      pk_fail(status, sync);
      *s_fail = 1;
    }
    if (p + 1 < n_phases && !grid_sync(sync, static_cast<unsigned>(p), status, s_ok, s_fail)) break;
  }

  // Exit: no copy may still be landing in shared memory and no MMA still
  // running (on the normal path every wait below returns at once).
  if (warp == 0 && lane == 0) {
    int st = p_ast;
    uint32_t ph_bit = p_aph;
    for (long i = 0; i < PK_STAGES && i < p_issued; ++i) {
      if (st == 0) {
        st = PK_STAGES;
        ph_bit ^= 1;
      }
      --st;
      mbar_wait(&afull[st], ph_bit);
    }
    if (p_nb > 0) mbar_wait(bfull, (p_nb - 1) & 1);
    if (p_na > 0) mbar_wait(at_full, (p_na - 1) & 1);
  }
  if (warp == 1 && lane == 0 && m_issued) {
    tc_commit(drain);
    mbar_wait(drain, 0);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, PK_TMEM_COLS);
  }
}

}  // namespace

// ---------------------------------------------------------------- barrier self-test
namespace {

// Two grid barriers over one CTA per SM (cooperative launch, 96 threads so
// that the polling thread 64 exists); unreachable != 0 makes the second one
// wait for arrivals that never come, so it gives up after its limit.
__global__ void __launch_bounds__(96) barrier_selftest_kernel(unsigned* sync, int unreachable, int* status,
                                                                unsigned long long* elapsed_ns) {
  __shared__ int s_ok, s_fail;
  if (threadIdx.x == 0) s_fail = 0;
  __syncthreads();
  const uint64_t t0 = global_timer_ns();
  if (grid_sync(sync, 0, status, &s_ok, &s_fail)) grid_sync(sync, unreachable ? 4 : 1, status, &s_ok, &s_fail);
  if (blockIdx.x == 0 && threadIdx.x == 0) *elapsed_ns = global_timer_ns() - t0;
}

}  // namespace

cudaError_t pk_barrier_selftest(cudaStream_t s, int unreachable, unsigned* sync, int* status,
                                unsigned long long* elapsed_ns) {
  cudaError_t e = cudaMemsetAsync(sync, 0, 2 * sizeof(unsigned), s);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(num_sms());
  cfg.blockDim = dim3(96);
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeCooperative;
  at[0].val.cooperative = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, barrier_selftest_kernel, sync, unreachable, status, elapsed_ns);
}

// ---------------------------------------------------------------- host side
struct PkPlan {
  struct Mode {
    const PkPhase* phases = nullptr;  // device; null: this mode has no one-launch plan
    const CUtensorMap* maps = nullptr;
    const unsigned long long* pf = nullptr;  // 128-byte lines of the small parameters, prefetched at start
    int n_phases = 0, n_maps = 0, n_pf = 0;
    std::string why;                  // the reason when it has none
  };
  std::vector<Mode> modes;
  char* dev = nullptr;       // one allocation: every mode's maps, then their phases
  unsigned* sync = nullptr;  // [2] barrier counter, abort flag (in the handle's arena)
  float* y32 = nullptr;      // final norm of the class-token row (in the handle's arena)
  int grid = 0;
  bool enabled = false;      // off by default: measured slower than the kernel-by-kernel chain
};

namespace {

// Builds one mode's phase list and tensor maps.
struct PkBuilder {
  const elasto_s* h;
  int n, grid;
  std::vector<PkPhase> ph;
  std::vector<CUtensorMap> maps;
  std::vector<unsigned long long> pf;  // lines of the small parameters
  std::string why;

  void prefetch(const void* p, size_t bytes) {
    if (!p) return;
    const uint64_t a = reinterpret_cast<uint64_t>(p) & ~uint64_t(127), e = reinterpret_cast<uint64_t>(p) + bytes;
    for (uint64_t l = a; l < e; l += 128) pf.push_back(l);
  }

  // [outer][inner] bf16 with rows ld elements apart, box 64 x box_outer, 128-byte swizzle
  int map2d(const void* base, uint64_t inner, uint64_t outer, uint64_t ld, uint32_t box_outer) {
    CUtensorMap tm;
    if (!encode_tmap_2d(&tm, base, inner, outer, ld * 2, 64, box_outer)) {
      why = "tensor map (alignment or size)";
      return -1;
    }
    maps.push_back(tm);
    return static_cast<int>(maps.size()) - 1;
  }

  // unswizzled map for TMA stores: dims innermost first, byte strides of dims 1.., box
  int map_plain(const void* base, int rank, const uint64_t* dims, const uint64_t* strides, const uint32_t* box,
                bool fp32, bool sw128) {
    CUtensorMap tm;
    if (!encode_tmap_plain(&tm, base, rank, dims, strides, box, fp32, sw128)) {
      why = "output tensor map (alignment or size)";
      return -1;
    }
    maps.push_back(tm);
    return static_cast<int>(maps.size()) - 1;
  }

  // out = epi(A[n, K] . W[N, K]^T) (W rows ldw apart, out rows ldo apart);
  // PKE_PART writes fp32 partial sums of ks splits split_stride apart.
  // Returns the split count, 0 on failure.
  int gemm(const bf16* A, int K, const bf16* W, int ldw, int N, const float* bias, void* out, int ldo, int epi,
           long long split_stride) {
    if (K <= 0 || N <= 0 || K % 8 != 0 || N % 8 != 0 || ldo % 8 != 0 || ldw < K || ldw % 8 != 0 ||
        (epi != PKE_PART && !bias)) {
      why = "GEMM shape";
      return 0;
    }
    PkPhase p;
    p.kind = PK_GEMM;
    p.epi = epi;
    p.N = N;
    p.ldo = ldo;
    p.bias = bias;
    p.out = out;
    p.split_stride = split_stride;
    p.mt = (n + 127) / 128;
    p.nk = (K + 63) / 64;
    const int bmax = PK_B_BYTES / 128;  // B rows x k-blocks of one unit
    p.bn = 0;
    if (epi != PKE_PART) {
      // the narrowest tile whose units fit one wave (A traffic per unit is
      // the same for any width), else the widest whose weights fit
      p.ks = 1;
      for (int c = 16; c <= PK_MAX_BN; c += 16) {
        if (c * p.nk > bmax) break;
        p.bn = c;
        if (p.mt * ((N + c - 1) / c) <= grid) break;
      }
    } else {
      // the widest tile, split as far as the idle SMs allow (fewer k-blocks
      // of A per unit), further if its weights would not fit
      for (int c = PK_MAX_BN; c >= 16 && p.bn == 0; c -= 16) {
        const int tiles = p.mt * ((N + c - 1) / c), kmax = std::min(kSplitMax, p.nk);
        int ks = std::max(1, std::min(kmax, grid / tiles));
        while (ks < kmax && c * ((p.nk + ks - 1) / ks) > bmax) ++ks;
        if (c * ((p.nk + ks - 1) / ks) <= bmax) {
          p.bn = c;
          p.ks = ks;
        }
      }
    }
    if (p.bn == 0) {
      why = "the weights of one tile do not fit shared memory";
      return 0;
    }
    p.nt = (N + p.bn - 1) / p.bn;
    p.units = p.mt * p.nt * p.ks;
    prefetch(bias, static_cast<size_t>(N) * 4);
    p.mapA = map2d(A, K, n, K, 128);
    p.mapB = map2d(W, K, N, ldw, p.bn);
    if (epi == PKE_PART) {  // [ks][n][N] fp32, ldo == N
      const uint64_t dims[3] = {uint64_t(N), uint64_t(n), uint64_t(p.ks)};
      const uint64_t st[2] = {uint64_t(ldo) * 4, uint64_t(split_stride) * 4};
      const uint32_t box[3] = {uint32_t(p.bn / 2), 32, 1};
      p.mapC = ldo == N ? map_plain(out, 3, dims, st, box, true, p.bn == 64) : -1;
    } else {  // [n][N] bf16, rows ldo apart (rows of at most 64 bytes: unswizzled)
      const uint64_t dims[2] = {uint64_t(N), uint64_t(n)};
      const uint64_t st[1] = {uint64_t(ldo) * 2};
      const uint32_t box[2] = {uint32_t(p.bn / 2), 32};
      p.mapC = map_plain(out, 2, dims, st, box, false, false);
    }
    if (p.mapA < 0 || p.mapB < 0 || p.mapC < 0) return 0;
    ph.push_back(p);
    return p.ks;
  }

  // X = base + (partials + bias), then y = LN(X) (g, b non-null) and / or the
  // final norm of row 0 into y32 (fg, fb non-null)
  void reduce(int ks, const float* xsrc, const float* bias, const float* g, const float* b, const float* fg,
              const float* fb, float* y32, int d, int d_true) {
    PkPhase p;
    p.kind = PK_REDUCE;
    p.units = n;
    p.ks = ks;
    p.split_stride = static_cast<long long>(n) * d;
    p.part = h->splitk_part;
    p.xsrc = xsrc;
    p.X = h->X;
    p.bias = bias;
    p.g = g;
    p.b = b;
    p.y = h->Y;
    p.fg = fg;
    p.fb = fb;
    p.y32 = y32;
    p.d = d;
    p.d_true = d_true;
    for (const float* v : {bias, g, b, fg, fb}) prefetch(v, static_cast<size_t>(d) * 4);
    ph.push_back(p);
  }

  bool build(const VitMode& vm, float* y32) {
    const elasto_model_desc& d = h->d;
    const VitEmbed& em = vm.emb;
    const int Dm = em.d_pad, dm = em.d, L = d.layers, kpe = h->kpe;
    const long long part_stride = static_cast<long long>(n) * Dm;
    if (d.weight_dtype != ELASTO_BF16) {
      why = "fp32-stored weights (two bf16 planes)";
      return false;
    }
    if (n > 256 || Dm % 64 != 0 || Dm > 1024 || kpe % 8 != 0) {
      why = "more than 256 tokens or an unsupported width";
      return false;
    }
    PkPhase pa;
    pa.kind = PK_PATCH;
    pa.units = n * kpe / 8;
    pa.img_dtype = d.weight_dtype;
    pa.img_h = d.img_h;
    pa.img_w = d.img_w;
    pa.img_c = d.img_c;
    pa.patch = d.patch;
    pa.kpe = kpe;
    pa.prow = h->P;
    ph.push_back(pa);
    int ks = gemm(h->P, kpe, em.pruned ? em.patch_w : h->patch_w, kpe, Dm, nullptr, h->splitk_part, Dm, PKE_PART,
                  part_stride);
    if (!ks) return false;
    reduce(ks, em.pruned ? em.addend : h->tok_addend, nullptr, em.ln1_w[0], em.ln1_b[0], nullptr, nullptr, nullptr,
           Dm, dm);
    for (int l = 0; l < L; ++l) {
      const VitLayerPack& lp = vm.layers[l];
      ks = 0;
      if (lp.w > 0) {
        if (!gemm(h->Y, Dm, lp.qkv_w, Dm, 3 * lp.w, lp.qkv_b, h->QKV, 3 * lp.w, PKE_BF16, 0)) return false;
        PkPhase a;
        a.kind = PK_ATTN;
        a.heads = lp.w / PK_HD;
        a.tiles = n > 128 ? 2 : 1;
        a.units = a.heads * a.tiles;
        a.n_pad = (n + 15) / 16 * 16;
        a.w = lp.w;
        a.o = h->O;
        a.blk_stride = h->prefix_shared ? PK_HD : lp.w;
        a.head_stride = h->prefix_shared ? 3 * PK_HD : PK_HD;
        a.mapQ = map2d(h->QKV, 3 * lp.w, n, 3 * lp.w, 128);
        a.mapKV = map2d(h->QKV, 3 * lp.w, n, 3 * lp.w, a.n_pad);
        {
          const uint64_t dims[2] = {uint64_t(lp.w), uint64_t(n)};
          const uint64_t st[1] = {uint64_t(lp.w) * 2};
          const uint32_t box[2] = {32, 32};
          a.mapO = map_plain(h->O, 2, dims, st, box, false, false);
        }
        if (a.mapQ < 0 || a.mapKV < 0 || a.mapO < 0) return false;
        ph.push_back(a);
        ks = gemm(h->O, lp.w, lp.proj_w, lp.ld_proj, Dm, nullptr, h->splitk_part, Dm, PKE_PART, part_stride);
        if (!ks) return false;
      }
      reduce(ks, nullptr, em.proj_b[l], em.ln2_w[l], em.ln2_b[l], nullptr, nullptr, nullptr, Dm, dm);
      ks = 0;
      if (lp.f > 0) {
        if (!gemm(h->Y, Dm, lp.fc1_w, Dm, lp.f_pad, lp.fc1_b, h->H, lp.f_pad, PKE_GELU, 0)) return false;
        ks = gemm(h->H, lp.f_pad, lp.fc2_w, lp.ld_fc2, Dm, nullptr, h->splitk_part, Dm, PKE_PART, part_stride);
        if (!ks) return false;
      }
      const bool last = l + 1 == L;
      reduce(ks, nullptr, em.fc2_b[l], last ? nullptr : em.ln1_w[l + 1], last ? nullptr : em.ln1_b[l + 1],
             last ? em.norm_w : nullptr, last ? em.norm_b : nullptr, last ? y32 : nullptr, Dm, dm);
    }
    PkPhase hd;
    hd.kind = PK_HEAD;
    hd.units = d.classes;
    hd.hw = em.head_w;
    hd.hb = h->head_b;
    hd.classes = d.classes;
    hd.d = Dm;
    hd.y32 = y32;
    prefetch(h->head_b, static_cast<size_t>(d.classes) * 4);
    ph.push_back(hd);
    return true;
  }
};

}  // namespace

cudaError_t pk_init_attributes() {
  return cudaFuncSetAttribute(dn_one_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, PK_SMEM);
}

size_t pk_workspace_floats(int d) { return static_cast<size_t>(d) + 16; }

void pk_free(PkPlan* p) {
  if (!p) return;
  if (p->dev) cudaFree(p->dev);
  delete p;
}

elasto_status pk_build(elasto_s* h, unsigned* sync, float* y32, PkPlan** out) {
  *out = nullptr;
  int dev = 0, coop = 0, per_sm = 0;
  ELASTO_CUDA_TRY(cudaGetDevice(&dev));
  ELASTO_CUDA_TRY(cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev));
  ELASTO_CUDA_TRY(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, dn_one_kernel, PK_THREADS, PK_SMEM));
  if (!coop || per_sm < 1 || num_sms() <= 0) return ELASTO_OK;  // no plan: forwards launch kernel by kernel
  PkPlan* p = new PkPlan();
  p->grid = num_sms();
  p->sync = sync;
  p->y32 = y32;
  std::vector<PkBuilder> bs;
  size_t maps_bytes = 0, phase_bytes = 0;
  for (const VitMode& vm : h->modes) {
    PkBuilder b{h, h->n, p->grid, {}, {}, {}};
    if (!b.build(vm, y32)) {
      b.ph.clear();
      b.maps.clear();
    }
    if (b.ph.empty()) b.pf.clear();
    maps_bytes += b.maps.size() * sizeof(CUtensorMap);
    phase_bytes += b.ph.size() * sizeof(PkPhase) + b.pf.size() * sizeof(unsigned long long);
    bs.push_back(std::move(b));
  }
  if (maps_bytes + phase_bytes > 0) {
    cudaError_t e = cudaMalloc(&p->dev, maps_bytes + phase_bytes);
    if (e != cudaSuccess) {
      cudaGetLastError();
      pk_free(p);
      return ELASTO_OK;  // the forwards stay kernel by kernel
    }
  }
  size_t mo = 0, po = maps_bytes;
  for (PkBuilder& b : bs) {
    PkPlan::Mode md;
    if (b.ph.empty()) {
      md.why = b.why;
    } else {
      const size_t mb = b.maps.size() * sizeof(CUtensorMap), pb = b.ph.size() * sizeof(PkPhase);
      const size_t lb = b.pf.size() * sizeof(unsigned long long);
      cudaError_t e = cudaMemcpy(p->dev + mo, b.maps.data(), mb, cudaMemcpyHostToDevice);
      if (e == cudaSuccess) e = cudaMemcpy(p->dev + po, b.ph.data(), pb, cudaMemcpyHostToDevice);
      if (e == cudaSuccess && lb) e = cudaMemcpy(p->dev + po + pb, b.pf.data(), lb, cudaMemcpyHostToDevice);
      if (e != cudaSuccess) {
        pk_free(p);
        return cuda_fail(e, "one-launch plan upload");
      }
      md.maps = reinterpret_cast<const CUtensorMap*>(p->dev + mo);
      md.phases = reinterpret_cast<const PkPhase*>(p->dev + po);
      md.pf = reinterpret_cast<const unsigned long long*>(p->dev + po + pb);
      md.n_maps = static_cast<int>(b.maps.size());
      md.n_phases = static_cast<int>(b.ph.size());
      md.n_pf = static_cast<int>(b.pf.size());
      mo += mb;
      po += pb + lb;
    }
    p->modes.push_back(md);
  }
  *out = p;
  return ELASTO_OK;
}

bool pk_ready(const PkPlan* p, int mode) {
  return p && p->enabled && mode >= 0 && mode < static_cast<int>(p->modes.size()) && p->modes[mode].phases;
}

void pk_enable(PkPlan* p, bool on) {
  if (p) p->enabled = on;
}

cudaError_t pk_launch(const PkPlan* p, int mode, int n, const void* images, float* logits, int* status,
                      cudaStream_t s) {
  const PkPlan::Mode& m = p->modes[mode];
  cudaError_t e = cudaMemsetAsync(p->sync, 0, 2 * sizeof(unsigned), s);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(p->grid);
  cfg.blockDim = dim3(PK_THREADS);
  cfg.dynamicSmemBytes = PK_SMEM;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeCooperative;
  at[0].val.cooperative = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, dn_one_kernel, m.phases, m.n_phases, m.maps, m.n_maps, m.pf, m.n_pf, n, images,
                            logits, p->sync, status);
}

}  // namespace elasto
