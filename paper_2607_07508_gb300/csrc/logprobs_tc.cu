// bf16 tensor-core path of the LM-head log-probs (Eq. 1-2) and their gradient.
//
// One persistent, warp-specialised GEMM kernel on the 5th-generation tensor
// cores serves all four contractions, with the per-element work fused into
// the epilogue so the [N, V] logits never reach memory:
//
//   forward   Z = H W^T          -> online (max, sum-exp) per row over each
//                                   256-wide vocabulary tile + gather of z[y]
//                                   (cached: also e = exp(z - kappa) in bf16,
//                                   one shift kappa per row)
//   backward  Z = H W^T (again)  -> dZ = G (1[v == y] - exp(z - lse)), bf16,
//                                   into a [N, Vc] chunk buffer
//             dH (+)= dZ W_chunk    (A K-major, B = W MN-major)
//             dW_chunk = dZ^T H     (A = dZ MN-major, B = H MN-major)
//   cached backward (dZ = s e row by row, s = -G exp(kappa - lse)):
//             dH = s (e W)          (A = e K-major, row scale in the epilogue)
//             dW = e^T (s H)        (A = e MN-major, B = s H MN-major)
//
// CTA layout (192 threads): warp 0 issues TMA loads of 128x64 A and 256x64 B
// bf16 tiles (128-byte swizzle) into a 4-stage shared-memory ring; warp 1
// owns 512 TMEM columns (two 128x256 fp32 accumulators) and issues
// tcgen05.mma (M=128, N=256, K=16) from one thread; warps 2-5 drain the
// accumulator through tcgen05.ld, one TMEM lane (= output row) per thread,
// while the MMA warp already fills the other accumulator. Every wait is
// bounded; a time-out raises SAO_DEVERR_PIPE_TIMEOUT and all roles wind down.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>
#include <math.h>
#include <stdint.h>

#include <mutex>

#include "logprobs_common.cuh"
#include "rows.cuh"
#include "sao_common.cuh"
#include "sao_internal.h"
#include "tc_ptx.cuh"

namespace sao {
namespace {

using namespace tc;

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr uint32_t A_BYTES = BM * BK * 2;
constexpr uint32_t B_BYTES = BN * BK * 2;
constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int NUM_THREADS = 192;
constexpr uint32_t TMEM_COLS = 2 * BN;
constexpr uint32_t MN_ATOM_BYTES = 64 * BK * 2;   // one 64(MN) x 64(K) box
constexpr uint32_t STAGE_OUT_BYTES = BM * 64 * 2; // one 128-row x 64-column bf16 output box
constexpr size_t SMEM_BYTES = 1024 + size_t(STAGES) * STAGE_BYTES + 2 * STAGE_OUT_BYTES + 256;
constexpr int EPI_BARRIER = 1;                    // named barrier of the 4 epilogue warps
constexpr float kLog2e = 1.4426950408889634f;

enum EpiKind : int { kSoftmax = 0, kDLogits = 1, kStoreF32 = 2, kStoreBF16 = 3, kSoftmaxStore = 4 };

// Epilogues that stage bf16 boxes in shared memory and write them with TMA
// stores; their 4 warps synchronise with named barriers.
template <int kEpi>
constexpr bool kTmaStoreEpi = (kEpi == kDLogits || kEpi == kSoftmaxStore);

struct GemmParams {
  int nM, nN, nK;      // tiles along M, N and 64-wide K blocks
  int group_m;         // tile raster: group_m M-tiles per group, M fastest inside
  int a_row_off;       // A K-major: row offset; A MN-major: column (M) offset
  int b_row_off;       // B K-major: row offset of N; B MN-major: K offset
  // epilogue
  int64_t rows;        // valid output rows (M extent)
  int cols;            // valid output columns (N extent)
  const int32_t *y;
  int vocab;           // V (softmax / dlogits)
  int v0;              // vocabulary index of GEMM column 0 (dlogits)
  float2 *part;        // softmax partials [nN][rows]
  float *zy;           // gathered logit of the sampled token
  const float *lse, *G;
  __nv_bfloat16 *dz;   // dlogits output [rows][ldz]
  int64_t ldz;
  float *cf;           // store f32 output (row-major, ldc)
  __nv_bfloat16 *cb;   // store bf16 output
  int64_t ldc;
  int64_t c_row_off;   // output row offset
  int accumulate;
  unsigned int *err;
  // row compaction (all optional): M extent and K extent read from the
  // device at start-up, and the original row of each compacted GEMM row
  const int *m_count;
  const int *k_count;
  const int *row_idx;
  // softmax+store: per-row shift and overflow flags (the cache's); plain
  // stores: optional per-row scale of the accumulator (GEMM row index)
  const float *kappa;
  uint8_t *flag;
  const float *row_scale;
};

constexpr int kMaxStages = 6;  // CTA pairs hold half a B tile per stage: 6 stages in the same bytes

struct __align__(8) SmemCtl {
  uint64_t full[kMaxStages], empty[kMaxStages], acc_full[2], acc_empty[2];
  uint32_t tmem_base;
  int abort;
};

__device__ __forceinline__ void tile_coords(int L, const GemmParams &p, int nM, int &m, int &n) {
  const int per_group = p.group_m * p.nN;
  const int g = L / per_group;
  const int within = L - g * per_group;
  const int m0 = g * p.group_m;
  const int gm = min(p.group_m, nM - m0);
  m = m0 + within % gm;
  n = within / gm;
}

// kMT = 2 (the long-K backward products, plain store epilogues): a CTA tile
// is two 128-row M tiles sharing every B stage, one per TMEM accumulator, so
// each B tile feeds two MMAs and W (or H) is read once per wave of 2 x 152
// row tiles instead of 152; the stages (A 32 KB + B 32 KB) shrink to 3. The
// tile's epilogue then waits for both accumulators, which costs little when
// K spans thousands of blocks.
//
// kCG = 2: the grid is made of CTA pairs (clusters of 2) and every MMA is a
// tcgen05.mma.cta_group::2 of M = 256 over the pair. Each CTA loads its own
// 128 rows of A and its half (128 columns) of the B tile into its own shared
// memory, so a pair moves 3/4 of the operand bytes two single CTAs would for
// the same flops, and accumulates its own 128 rows x 256 columns in its own
// TMEM. The even CTA's producer counts both CTAs' copies on its full barrier
// (the odd CTA's copies signal it across the pair), its one MMA thread issues
// for the pair and commits to both CTAs' empty and accumulator barriers, and
// both CTAs' epilogue threads release an accumulator on the even CTA's
// barrier. The stages hold half a B tile: 6 (or 4 with kMT = 2).
template <int kEpi, bool kAMN, bool kBMN, int kMT = 1, int kCG = 1>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
                   const __grid_constant__ CUtensorMap map_c, const GemmParams p) {
  static_assert(kMT == 1 || kMT == 2, "one or two M tiles per CTA tile");
  static_assert(kCG == 1 || kCG == 2, "single CTAs or CTA pairs");
  static_assert(kMT == 1 || kEpi == kStoreF32 || kEpi == kStoreBF16, "two M tiles: plain store epilogues only");
  constexpr uint32_t kABytes = A_BYTES * kMT;
  constexpr uint32_t kBBytes = B_BYTES / kCG;  // this CTA's part of a B stage
  constexpr uint32_t kStageBytes = kABytes + kBBytes;
  constexpr int kStages = int(size_t(STAGES) * STAGE_BYTES / kStageBytes);
  constexpr int kTM = BM * kMT * kCG;  // rows of a tile (of the pair's tile for kCG = 2)
  static_assert(kStages <= kMaxStages, "barrier arrays");
  static_assert(size_t(kStages) * kStageBytes <= size_t(STAGES) * STAGE_BYTES, "same shared-memory layout");
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t *gbase = smem_raw + (base - raw);
  const uint32_t out_base = base + uint32_t(STAGES) * STAGE_BYTES;  // 2 output staging boxes
  SmemCtl *ctl = reinterpret_cast<SmemCtl *>(gbase + size_t(STAGES) * STAGE_BYTES + 2 * STAGE_OUT_BYTES);
  volatile int *abort = &ctl->abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // CTA pairs: rank in the pair, the pair's index and the number of pairs
  const uint32_t rank = kCG == 2 ? cluster_ctarank() : 0u;
  const int cl = int(blockIdx.x) / kCG, ncl = int(gridDim.x) / kCG;
  int nM = p.nM, nK = p.nK;
  int64_t rows = p.rows;
  if (p.m_count) {
    const int c = *p.m_count;
    rows = c;
    nM = (c + kTM - 1) / kTM;
  }
  if (p.k_count) nK = (*p.k_count + BK - 1) / BK;
  // an empty contraction added to the output changes nothing: skip the grid
  if (kEpi == kStoreF32 && p.k_count && nK == 0 && p.accumulate) return;
  const int num_tiles = nM * p.nN;
  const bool kzero = (nK == 0);  // empty contraction: the tile is all zeros

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_u32(&ctl->full[s]), 1);
      mbar_init(smem_u32(&ctl->empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&ctl->acc_full[a]), 1);
      mbar_init(smem_u32(&ctl->acc_empty[a]), 4 * 32 * kCG);
    }
    ctl->abort = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    if constexpr (kCG == 2) {
      tmem_alloc_pair(smem_u32(&ctl->tmem_base), TMEM_COLS);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(smem_u32(&ctl->tmem_base), TMEM_COLS);
      tmem_relinquish();
    }
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&map_a);
    tma_prefetch_map(&map_b);
  }
  fence_before_sync();
  __syncthreads();
  // both CTAs' barriers exist before either CTA's copies, commits or arrivals reach them
  if constexpr (kCG == 2) cluster_sync();
  fence_after_sync();
  const uint32_t tmem_base = ctl->tmem_base;
  // releases an accumulator: on this CTA's barrier, or the even CTA's for a pair
  auto release_acc = [&](int a) {
    const uint32_t bar = smem_u32(&ctl->acc_empty[a]);
    if (kCG == 2 && rank != 0u)
      mbar_arrive_cluster(mapa_shared(bar, 0u));
    else
      mbar_arrive(bar);
  };

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      uint32_t issued = 0;  // bit s: stage s has a load whose full-barrier phase is phase_of(s)
      uint32_t issued_phase = 0;
      // a load lands in this CTA's shared memory; its bytes are counted on
      // this CTA's full barrier, or on the even CTA's for a pair
      auto load = [&](uint32_t dst, const CUtensorMap *map, uint32_t bar, int x, int y) {
        if constexpr (kCG == 2)
          tma_load_2d_pair(dst, map, bar, x, y);
        else
          tma_load_2d(dst, map, bar, x, y);
      };
      for (int L = cl; L < num_tiles && ok; L += ncl) {
        int m, n;
        tile_coords(L, p, nM, m, n);
        for (int kb = 0; kb < nK; ++kb) {
          if (!mbar_wait(smem_u32(&ctl->empty[stage]), phase ^ 1u, abort, p.err)) {
            ok = false;
            break;
          }
          const uint32_t fb_own = smem_u32(&ctl->full[stage]);
          const uint32_t fb = kCG == 2 ? mapa_shared(fb_own, 0u) : fb_own;
          issued |= 1u << stage;
          issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
          if (rank == 0u) mbar_arrive_expect_tx(fb_own, kStageBytes * kCG);
          const uint32_t sa = base + uint32_t(stage) * kStageBytes;
          const uint32_t sb = sa + kABytes;
          const int k0 = kb * BK;
#pragma unroll
          for (int j = 0; j < kMT; ++j) {  // this CTA's 128 rows of M tile j
            const int row = p.a_row_off + m * kTM + j * BM * kCG + int(rank) * BM;
            if (!kAMN) {
              load(sa + j * A_BYTES, &map_a, fb, k0, row);
            } else {
#pragma unroll
              for (int jj = 0; jj < BM / 64; ++jj) load(sa + j * A_BYTES + jj * MN_ATOM_BYTES, &map_a, fb, row + 64 * jj, k0);
            }
          }
          const int ncol = n * BN + int(rank) * (BN / kCG);  // this CTA's columns of the B tile
          if (!kBMN) {
            load(sb, &map_b, fb, k0, p.b_row_off + ncol);
          } else {
#pragma unroll
            for (int j = 0; j < BN / kCG / 64; ++j) load(sb + j * MN_ATOM_BYTES, &map_b, fb, ncol + 64 * j, p.b_row_off + k0);
          }
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok && rank == 0u) {
        // let the copies already in flight land before the CTA can exit (a
        // pair's full barriers, in the even CTA, count both CTAs' copies)
        for (int s = 0; s < kStages; ++s) {
          if (!((issued >> s) & 1u)) continue;
          const uint32_t par = (issued_phase >> s) & 1u;
          const uint64_t t0 = globaltimer_ns();
          while (!mbar_try_wait(smem_u32(&ctl->full[s]), par) && globaltimer_ns() - t0 < kWaitLimitNs) {
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    // a pair's MMAs are all issued by the even CTA
    if (lane == 0 && rank == 0u) {
      constexpr uint32_t idesc = idesc_bf16(BM * kCG, BN, kAMN, kBMN);
      int stage = 0;
      uint32_t phase = 0;
      int local = 0;
      bool ok = true;
      auto commit = [&](uint32_t bar) {
        if constexpr (kCG == 2)
          mma_commit_pair(bar, uint16_t(0x3));
        else
          mma_commit(bar);
      };
      auto mma = [&](uint32_t d, uint64_t ad, uint64_t bd, uint32_t accum) {
        if constexpr (kCG == 2)
          mma_bf16_pair(d, ad, bd, idesc, accum);
        else
          mma_bf16(d, ad, bd, idesc, accum);
      };
      for (int L = cl; L < num_tiles && ok; L += ncl, ++local) {
        // kMT == 2: both accumulators serve one tile, tracked as accumulator 0
        const int acc = kMT == 2 ? 0 : (local & 1);
        const uint32_t acc_phase = kMT == 2 ? (uint32_t(local) & 1u) : (uint32_t(local >> 1) & 1u);
        if (!mbar_wait(smem_u32(&ctl->acc_empty[acc]), acc_phase ^ 1u, abort, p.err)) break;
        fence_after_sync();
        const uint32_t d_tmem = tmem_base + uint32_t(acc) * BN;
        for (int kb = 0; kb < nK; ++kb) {
          if (!mbar_wait(smem_u32(&ctl->full[stage]), phase, abort, p.err)) {
            ok = false;
            break;
          }
          fence_after_sync();
          const uint32_t sa = base + uint32_t(stage) * kStageBytes;
          const uint32_t sb = sa + kABytes;
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
            const uint64_t bd = kBMN ? sdesc_sw128(sb + kk * 2048u, MN_ATOM_BYTES, 1024u)
                                     : sdesc_sw128(sb + kk * 32u, 16u, 1024u);
#pragma unroll
            for (int j = 0; j < kMT; ++j) {  // A tile j (rows j*128 ..) into accumulator acc + j
              const uint32_t aj = sa + uint32_t(j) * A_BYTES;
              const uint64_t ad = kAMN ? sdesc_sw128(aj + kk * 2048u, MN_ATOM_BYTES, 1024u)
                                       : sdesc_sw128(aj + kk * 32u, 16u, 1024u);
              mma(d_tmem + uint32_t(j) * BN, ad, bd, (kb | kk) != 0 ? 1u : 0u);
            }
          }
          commit(smem_u32(&ctl->empty[stage]));
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        commit(smem_u32(&ctl->acc_full[acc]));
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int quad = warp & 3;  // TMEM lane quadrant this warp may access
    const int r = quad * 32 + lane;
    int local = 0;
    for (int L = cl; L < num_tiles; L += ncl, ++local) {
      int m, n;
      tile_coords(L, p, nM, m, n);
      const int acc = kMT == 2 ? 0 : (local & 1);
      const uint32_t acc_phase = kMT == 2 ? (uint32_t(local) & 1u) : (uint32_t(local >> 1) & 1u);
      bool ok = mbar_wait(smem_u32(&ctl->acc_full[acc]), acc_phase, abort, p.err);
      // The dlogits epilogue synchronises its 4 warps with named barriers, so
      // they must agree on whether this tile goes ahead.
      if constexpr (kTmaStoreEpi<kEpi>) ok = named_barrier_and(EPI_BARRIER, 128, ok);
      if (!ok) break;
      fence_after_sync();
      const uint32_t taddr = tmem_base + (uint32_t(quad * 32) << 16) + uint32_t(acc) * BN;
      // this CTA's first row of the tile (M tile 0); M tile j starts BM * kCG rows further
      const int64_t row0 = int64_t(m) * kTM + int64_t(rank) * BM;
      const int64_t row = row0 + r;
      const bool row_ok = row < rows;
      const int64_t orig = (row_ok && p.row_idx) ? int64_t(__ldg(p.row_idx + row)) : row;

      if constexpr (kEpi == kSoftmax) {
        const int col0 = n * BN;
        const int yy = row_ok ? __ldg(p.y + orig) : -1;
        float mx = -INFINITY, sm = 0.f, zsel = 0.f;
        bool have = false;
#pragma unroll 1
        for (int c = 0; c < BN / 32; ++c) {
          uint32_t u[32];
          tmem_ld32(taddr + c * 32, u);
          tmem_wait_ld();
          const int cbase = col0 + c * 32;
          const int valid = p.vocab - cbase;
          float v[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = (j < valid) ? __uint_as_float(u[j]) : -INFINITY;
          float cm = v[0];
#pragma unroll
          for (int j = 1; j < 32; ++j) cm = fmaxf(cm, v[j]);
          const float mn = fmaxf(mx, cm);
          const float off = -mn * kLog2e;
          float s = 0.f;
#pragma unroll
          for (int j = 0; j < 32; ++j) s += ex2_approx(fmaf(v[j], kLog2e, off));
          sm = fmaf(sm, ex2_approx((mx - mn) * kLog2e), s);
          mx = mn;
          const unsigned rel = unsigned(yy - cbase);
          if (rel < 32u) {
            float z = v[0];
#pragma unroll
            for (int j = 1; j < 32; ++j) z = (unsigned(j) == rel) ? v[j] : z;
            zsel = z;
            have = true;
          }
        }
        fence_before_sync();
        release_acc(acc);
        if (row_ok) {
          p.part[int64_t(n) * p.rows + row] = make_float2(mx, sm);  // compacted row, stride N
          if (have) p.zy[row] = zsel;
        }
      } else if constexpr (kEpi == kSoftmaxStore) {
        // As kSoftmax, in one pass over TMEM, and also storing e = exp(z -
        // kappa) as bf16 with the row's own shift kappa (the sampled token's
        // logit + kKappaOffset): the backward then needs no per-tile maxima.
        // The tile's partial is (kappa, sum e). A 32-column chunk holding some
        // z > kappa + kFlagExponent (a sampled token far below the row's
        // maximum) flags the row, stores clamped values, and enters the
        // partial against its own maximum instead. Boxes of 128 rows x 64
        // columns go out through two swizzled staging buffers and TMA stores
        // issued by one thread.
        const bool issuer = (warp == 2 && lane == 0);
        const int col0 = n * BN;
        const int yy = row_ok ? __ldg(p.y + orig) : -1;
        const float kap = row_ok ? __ldg(p.kappa + row) : 0.f;
        const float off = -kap * kLog2e;
        // a flagged row's values are clamped to 2^64: its row of e W stays far
        // from fp32 overflow in the backward, which scales that row by 0
        constexpr float kClampLog2 = 64.f;
        float sk = 0.f;                      // sum of e over the unflagged chunks
        float bm = -INFINITY, bs = 0.f;      // flagged chunks: online (max, sum exp(z - max))
        float zsel = 0.f;
        bool have = false;
#pragma unroll 1
        for (int box = 0; box < BN / 64; ++box) {
          const uint32_t buf = out_base + uint32_t(box & 1) * STAGE_OUT_BYTES;
          if (issuer) bulk_wait_group_read<1>();  // the store that last read `buf` is done
          named_barrier(EPI_BARRIER, 128);
#pragma unroll
          for (int half = 0; half < 2; ++half) {
            const int c = box * 2 + half;
            uint32_t u[32];
            tmem_ld32(taddr + c * 32, u);
            tmem_wait_ld();
            if (c == BN / 32 - 1) {
              fence_before_sync();
              release_acc(acc);
            }
            const int cbase = col0 + c * 32;
            const int valid = p.vocab - cbase;
            uint32_t pk[16];
            float cs = 0.f, cm = -INFINITY;
#pragma unroll
            for (int j = 0; j < 32; j += 2) {
              const float z0 = __uint_as_float(u[j]), z1 = __uint_as_float(u[j + 1]);
              const float e0 = (j < valid) ? ex2_approx(fminf(fmaf(z0, kLog2e, off), kClampLog2)) : 0.f;
              const float e1 = (j + 1 < valid) ? ex2_approx(fminf(fmaf(z1, kLog2e, off), kClampLog2)) : 0.f;
              cm = (j < valid) ? fmaxf(cm, z0) : cm;
              cm = (j + 1 < valid) ? fmaxf(cm, z1) : cm;
              cs += e0 + e1;
              const __nv_bfloat162 b2 = __floats2bfloat162_rn(e0, e1);
              pk[j / 2] = *reinterpret_cast<const uint32_t *>(&b2);
            }
            if (cm - kap > kFlagExponent) {  // rare: redo the chunk's sum against its maximum
              float s2 = 0.f;
#pragma unroll
              for (int j = 0; j < 32; ++j)
                s2 += (j < valid) ? ex2_approx((__uint_as_float(u[j]) - cm) * kLog2e) : 0.f;
              const float mn = fmaxf(bm, cm);
              bs = fmaf(bs, ex2_approx((bm - mn) * kLog2e), s2 * ex2_approx((cm - mn) * kLog2e));
              bm = mn;
            } else {
              sk += cs;
            }
            const unsigned rel = unsigned(yy - cbase);
            if (rel < 32u) {
              float z = __uint_as_float(u[0]);
#pragma unroll
              for (int j = 1; j < 32; ++j) z = (unsigned(j) == rel) ? __uint_as_float(u[j]) : z;
              zsel = z;
              have = true;
            }
            const uint32_t row_addr = buf + uint32_t(r) * 128u;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const uint32_t chunk = uint32_t(half * 4 + q) ^ uint32_t(r & 7);
              asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(row_addr + chunk * 16u),
                           "r"(pk[4 * q]), "r"(pk[4 * q + 1]), "r"(pk[4 * q + 2]), "r"(pk[4 * q + 3])
                           : "memory");
            }
          }
          fence_proxy_async_smem();
          named_barrier(EPI_BARRIER, 128);
          // (the odd CTA of a pair may hold no row of the last tile: nothing to store)
          if (issuer && row0 < rows) {  // e is read again only by the backward: evict it first from L2
            tma_store_2d_hint(&map_c, buf, col0 + box * 64, int(row0), l2_evict_first());
            bulk_commit_group();
          }
        }
        if (row_ok) {
          float2 part = make_float2(kap, sk);
          if (bm != -INFINITY) {  // a flagged chunk: merge the two partials
            const float mn = fmaxf(kap, bm);
            part = make_float2(mn, fmaf(sk, ex2_approx((kap - mn) * kLog2e), bs * ex2_approx((bm - mn) * kLog2e)));
            p.flag[row] = 1;
          }
          p.part[int64_t(n) * p.rows + row] = part;  // compacted row, stride N
          if (have) p.zy[row] = zsel;
        }
      } else if constexpr (kEpi == kDLogits) {
        // dZ goes out through two swizzled 128x64 staging boxes and TMA
        // stores; one epilogue thread issues the stores and tracks them.
        const bool issuer = (warp == 2 && lane == 0);
        const int lc0 = n * BN;  // column inside the chunk
        int yy = -1;
        float g = 0.f, l2 = 0.f;
        if (row_ok) {
          yy = __ldg(p.y + orig) - p.v0;
          g = __ldg(p.G + orig);
          l2 = __ldg(p.lse + orig) * kLog2e;
        }
#pragma unroll 1
        for (int box = 0; box < BN / 64; ++box) {
          const uint32_t buf = out_base + uint32_t(box & 1) * STAGE_OUT_BYTES;
          if (issuer) bulk_wait_group_read<1>();  // the store that last read `buf` is done
          named_barrier(EPI_BARRIER, 128);
#pragma unroll
          for (int half = 0; half < 2; ++half) {
            const int c = box * 2 + half;
            uint32_t u[32];
            tmem_ld32(taddr + c * 32, u);
            tmem_wait_ld();
            if (c == BN / 32 - 1) {
              fence_before_sync();
              release_acc(acc);
            }
            const int lc = lc0 + c * 32;
            uint32_t pk[16];
#pragma unroll
            for (int j = 0; j < 32; j += 2) {
              float d0 = 0.f, d1 = 0.f;
              if (g != 0.f) {
                d0 = -g * ex2_approx(fmaf(__uint_as_float(u[j]), kLog2e, -l2));
                d1 = -g * ex2_approx(fmaf(__uint_as_float(u[j + 1]), kLog2e, -l2));
                if (lc + j == yy) d0 += g;
                if (lc + j + 1 == yy) d1 += g;
              }
              const __nv_bfloat162 b2 = __floats2bfloat162_rn(d0, d1);
              pk[j / 2] = *reinterpret_cast<const uint32_t *>(&b2);
            }
            // 128-byte swizzle: 16-byte chunk j of row r sits at chunk j ^ (r % 8)
            const uint32_t row_addr = buf + uint32_t(r) * 128u;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const uint32_t chunk = uint32_t(half * 4 + q) ^ uint32_t(r & 7);
              asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(row_addr + chunk * 16u),
                           "r"(pk[4 * q]), "r"(pk[4 * q + 1]), "r"(pk[4 * q + 2]), "r"(pk[4 * q + 3])
                           : "memory");
            }
          }
          fence_proxy_async_smem();
          named_barrier(EPI_BARRIER, 128);
          if (issuer && row0 < rows) {
            tma_store_2d(&map_c, buf, lc0 + box * 64, int(row0));
            bulk_commit_group();
          }
        }
      } else {
        // kStoreF32 / kStoreBF16: plain tile store (optionally accumulating); with
        // kMT == 2 the second M tile comes from the second accumulator
#pragma unroll 1
        for (int j = 0; j < kMT; ++j) {
        const int64_t rowj = row + int64_t(j) * BM * kCG;
        const bool okj = rowj < rows;
        const int64_t origj = j == 0 ? orig : ((okj && p.row_idx) ? int64_t(__ldg(p.row_idx + rowj)) : rowj);
        const int64_t orow = p.c_row_off + origj;
        const float rs = (p.row_scale && okj) ? __ldg(p.row_scale + rowj) : 1.f;
#pragma unroll 1
        for (int c = 0; c < BN / 32; ++c) {
          uint32_t u[32];
          tmem_ld32(taddr + uint32_t(j) * BN + c * 32, u);
          tmem_wait_ld();
          if (kzero) {
#pragma unroll
            for (int j = 0; j < 32; ++j) u[j] = 0u;
          }
          if (p.row_scale) {  // a zero scale gives zeros whatever the accumulator holds
#pragma unroll
            for (int j = 0; j < 32; ++j) u[j] = rs == 0.f ? 0u : __float_as_uint(__uint_as_float(u[j]) * rs);
          }
          const int col = n * BN + c * 32;
          if (!okj || col >= p.cols) continue;
          const bool full = col + 32 <= p.cols;
          if constexpr (kEpi == kStoreF32) {
            float *dst = p.cf + orow * p.ldc + col;
            if (full) {
              float4 *d4 = reinterpret_cast<float4 *>(dst);
#pragma unroll
              for (int q = 0; q < 8; ++q) {
                float4 w = make_float4(__uint_as_float(u[4 * q]), __uint_as_float(u[4 * q + 1]),
                                       __uint_as_float(u[4 * q + 2]), __uint_as_float(u[4 * q + 3]));
                if (p.accumulate) {
                  const float4 o = d4[q];
                  w.x += o.x;
                  w.y += o.y;
                  w.z += o.z;
                  w.w += o.w;
                }
                d4[q] = w;
              }
            } else {
#pragma unroll
              for (int j = 0; j < 32; ++j)
                if (col + j < p.cols) dst[j] = p.accumulate ? dst[j] + __uint_as_float(u[j]) : __uint_as_float(u[j]);
            }
          } else {
            __nv_bfloat16 *dst = p.cb + orow * p.ldc + col;
            if (full) {
              uint32_t pk[16];
#pragma unroll
              for (int j = 0; j < 32; j += 2) {
                const __nv_bfloat162 b2 = __floats2bfloat162_rn(__uint_as_float(u[j]), __uint_as_float(u[j + 1]));
                pk[j / 2] = *reinterpret_cast<const uint32_t *>(&b2);
              }
              uint4 *d4 = reinterpret_cast<uint4 *>(dst);
#pragma unroll
              for (int q = 0; q < 4; ++q) d4[q] = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
            } else {
#pragma unroll
              for (int j = 0; j < 32; ++j)
                if (col + j < p.cols) dst[j] = __float2bfloat16_rn(__uint_as_float(u[j]));
            }
          }
        }
        }
        fence_before_sync();
        release_acc(acc);
      }
    }
  }

  if constexpr (kTmaStoreEpi<kEpi>) {
    if (warp == 2 && lane == 0) bulk_wait_group<0>();
  }
  fence_before_sync();
  __syncthreads();
  // neither CTA of a pair frees its TMEM or exits while the other may still
  // reach its shared memory (copies counted on the even CTA's barriers,
  // releases of its accumulators, commits to the odd CTA's barriers)
  if constexpr (kCG == 2) cluster_sync();
  if (warp == 1) {
    fence_after_sync();
    if constexpr (kCG == 2)
      tmem_dealloc_pair(tmem_base, TMEM_COLS);
    else
      tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------
// the probability cache: row shifts, the sampled token's entry, backward scales
// ---------------------------------------------------------------------------
constexpr int kRowWarps = 8;  // rows (one per warp) per CTA of the row kernels

// kappa[f] = H[t] . W[y[t]] + kKappaOffset (fp32 sums of the bf16 products) for
// forward row f < count, A being the forward GEMM's A operand (row f is token
// t = idx[f]); flag[f] = 0. One warp per row, 16-byte loads (h % 8 == 0).
__global__ void __launch_bounds__(32 * kRowWarps) kappa_kernel(const __nv_bfloat16 *A, int h,
                                                              const __nv_bfloat16 *W, const int32_t *y, int V,
                                                              const int *idx, const int *count, float *kappa,
                                                              uint8_t *flag) {
  const int f = blockIdx.x * kRowWarps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (f >= *count) return;
  const int yy = __ldg(y + __ldg(idx + f));
  float acc = 0.f;
  if (yy >= 0 && yy < V) {
    const __nv_bfloat16 *a = A + int64_t(f) * h, *w = W + int64_t(yy) * h;
    for (int k = lane * 8; k < h; k += 256) {
      const uint4 av = __ldg(reinterpret_cast<const uint4 *>(a + k));
      const uint4 wv = __ldg(reinterpret_cast<const uint4 *>(w + k));
      const uint32_t aw[4] = {av.x, av.y, av.z, av.w}, ww[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&aw[q]));
        const float2 z = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&ww[q]));
        acc = fmaf(x.x, z.x, acc);
        acc = fmaf(x.y, z.y, acc);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  }
  if (lane == 0) {
    kappa[f] = acc + kKappaOffset;
    flag[f] = 0;
  }
}

// Once lse is known: e[f, y] = exp(z_y - kappa) - exp(lse - kappa) =
// -exp(z_y - kappa) expm1(-logp), for the unflagged rows with a valid token,
// so that dZ[f, .] = -G exp(kappa - lse) e[f, .] holds at v = y as well.
__global__ void patch_target_kernel(__nv_bfloat16 *e, int64_t lde, const int *idx, const int *count,
                                    const int32_t *y, int V, const float *zy, const float *logp,
                                    const float *kappa, const uint8_t *flag) {
  const int f = blockIdx.x * blockDim.x + threadIdx.x;
  if (f >= *count || flag[f]) return;
  const int t = idx[f];
  const int yy = y[t];
  if (yy < 0 || yy >= V) return;
  const float a = expf(zy[f] - kappa[f]);
  e[int64_t(f) * lde + yy] = __float2bfloat16_rn(-a * expm1f(-logp[t]));
}

// Forward rows = tokens (no row was skipped).
__global__ void cache_identity_kernel(int *idx, int *pos, int *count, int64_t N) {
  const int64_t t = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (t < N) idx[t] = pos[t] = int(t);
  if (t == 0) *count = int(N);
}

// fb[t] = 1 when grad[t] != 0 and the token's forward row is flagged (those
// rows are recomputed); grad != 0 on a token the forward skipped raises
// SAO_DEVERR_CACHE_ROW (it contributes nothing).
__global__ void bwd_token_kernel(const float *G, const int *pos, const uint8_t *flag, int64_t N, uint8_t *fb,
                                 unsigned int *err) {
  const int64_t t = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (t >= N) return;
  uint8_t v = 0;
  if (G[t] != 0.f) {
    const int f = pos[t];
    if (f < 0)
      raise_device_error(err, SAO_DEVERR_CACHE_ROW);
    else
      v = flag[f];
  }
  fb[t] = v;
}

// For forward row f < round_up(count, 128): sc[f] = -G[t] exp(kappa[f] -
// lse[t]) (0 past count and on flagged rows) and Hs[f] = bf16(sc[f] H[t]),
// the dW GEMM's B operand. One warp per row, 16-byte loads and stores.
__global__ void __launch_bounds__(32 * kRowWarps) bwd_scale_kernel(const __nv_bfloat16 *H, int h,
                                                                  const int *idx, const int *count,
                                                                  const float *G, const float *lse,
                                                                  const float *kappa, const uint8_t *flag,
                                                                  float *sc, __nv_bfloat16 *Hs,
                                                                  int64_t rows_cap) {
  const int64_t f = int64_t(blockIdx.x) * kRowWarps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  const int n = *count;
  const int64_t pad = (int64_t(n) + BM - 1) / BM * BM;
  if (f >= pad || f >= rows_cap) return;
  float sf = 0.f;
  int t = -1;
  if (f < n) {
    t = __ldg(idx + f);
    if (!flag[f]) sf = -__ldg(G + t) * expf(__ldg(kappa + f) - __ldg(lse + t));
  }
  if (lane == 0) sc[f] = sf;
  __nv_bfloat16 *dst = Hs + f * h;
  for (int k = lane * 8; k < h; k += 256) {
    uint4 o = make_uint4(0u, 0u, 0u, 0u);
    if (sf != 0.f) {
      const uint4 v = __ldg(reinterpret_cast<const uint4 *>(H + int64_t(t) * h + k));
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
      uint32_t r[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&w[q]));
        const __nv_bfloat162 b2 = __floats2bfloat162_rn(sf * x.x, sf * x.y);
        r[q] = *reinterpret_cast<const uint32_t *>(&b2);
      }
      o = make_uint4(r[0], r[1], r[2], r[3]);
    }
    *reinterpret_cast<uint4 *>(dst + k) = o;
  }
}

// ---------------------------------------------------------------------------
// host side: tensor maps and launches
// ---------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 2-D bf16 tensor map over a row-major [outer][inner] array with row pitch
// `pitch_elems`, box {box_inner (64 = 128 bytes), box_outer}, 128-byte swizzle,
// zero fill outside the array.
sao_status make_map(CUtensorMap *m, const void *ptr, uint64_t inner, uint64_t outer, uint64_t pitch_elems,
                    uint32_t box_inner, uint32_t box_outer) {
  auto fn = encode_fn();
  if (!fn) return fail(SAO_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  if ((reinterpret_cast<uintptr_t>(ptr) & 15u) != 0) return fail(SAO_ERR_INVALID_ARG, "bf16 operand not 16-byte aligned");
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {pitch_elems * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(SAO_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", int(r));
  return SAO_OK;
}

template <int kEpi, bool kAMN, bool kBMN, int kMT = 1, int kCG = 1>
sao_status launch_gemm(const char *name, const CUtensorMap &ma, const CUtensorMap &mb, const CUtensorMap &mc,
                       const GemmParams &p, cudaStream_t s) {
  auto kern = tc_gemm_kernel<kEpi, kAMN, kBMN, kMT, kCG>;
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  static int max_pairs = 0;  // CTA pairs that fit on the device at once
  std::call_once(once, [&] {
    attr_err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(SMEM_BYTES));
    if (attr_err == cudaSuccess && kCG == 2) {
      cudaLaunchAttribute at[1];
      at[0].id = cudaLaunchAttributeClusterDimension;
      at[0].val.clusterDim.x = 2;
      at[0].val.clusterDim.y = 1;
      at[0].val.clusterDim.z = 1;
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(2);
      cfg.blockDim = dim3(NUM_THREADS);
      cfg.dynamicSmemBytes = SMEM_BYTES;
      cfg.attrs = at;
      cfg.numAttrs = 1;
      attr_err = cudaOccupancyMaxActiveClusters(&max_pairs, kern, &cfg);
    }
  });
  if (attr_err != cudaSuccess) return fail(SAO_ERR_CUDA, "kernel set-up: %s", cudaGetErrorString(attr_err));
  DeviceInfo di;
  SAO_TRY(device_info(&di));
  const int tiles = p.nM * p.nN;
  if (tiles == 0 || p.nK == 0) return SAO_OK;
  if constexpr (kCG == 2) {
    if (max_pairs < 1) return fail(SAO_ERR_UNSUPPORTED, "no CTA pair of the GEMM kernel fits on this device");
    const int pairs = tiles < max_pairs ? tiles : max_pairs;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(unsigned(2 * pairs));
    cfg.blockDim = dim3(NUM_THREADS);
    cfg.dynamicSmemBytes = SMEM_BYTES;
    cfg.stream = s;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int slot = launch_begin(name, s);
    const cudaError_t e = cudaLaunchKernelEx(&cfg, kern, ma, mb, mc, p);
    if (e != cudaSuccess) return fail(SAO_ERR_CUDA, "cudaLaunchKernelEx (%s): %s", name, cudaGetErrorString(e));
    return launch_end(slot, s);
  } else {
    const int grid = tiles < di.sm_count ? tiles : di.sm_count;
    int slot = launch_begin(name, s);
    kern<<<grid, NUM_THREADS, SMEM_BYTES, s>>>(ma, mb, mc, p);
    return launch_end(slot, s);
  }
}

// The same GEMM with kmt M tiles per CTA tile (plain store epilogues may take
// two) on single CTAs (cg = 1) or CTA pairs (cg = 2).
template <int kEpi, bool kAMN, bool kBMN>
sao_status launch_gemm_cfg(const char *name, int kmt, int cg, const CUtensorMap &ma, const CUtensorMap &mb,
                           const CUtensorMap &mc, const GemmParams &p, cudaStream_t s) {
  if constexpr (kEpi == kStoreF32 || kEpi == kStoreBF16) {
    if (kmt == 2)
      return cg == 2 ? launch_gemm<kEpi, kAMN, kBMN, 2, 2>(name, ma, mb, mc, p, s)
                     : launch_gemm<kEpi, kAMN, kBMN, 2, 1>(name, ma, mb, mc, p, s);
  }
  return cg == 2 ? launch_gemm<kEpi, kAMN, kBMN, 1, 2>(name, ma, mb, mc, p, s)
                 : launch_gemm<kEpi, kAMN, kBMN, 1, 1>(name, ma, mb, mc, p, s);
}

// Two M tiles per CTA tile halve the re-reads of the shared operand but also
// the number of tiles: worth it while at least four waves of tiles remain
// (at 8k tokens dH has 176 paired tiles on 152 SMs and runs 15 % slower).
// `workers` = SMs, or SM pairs for CTA pairs.
bool pair_tiles(int64_t paired_tiles, int workers) { return paired_tiles >= 4 * int64_t(workers); }

// M tiles per CTA tile (1 or 2) for a long-K product with `rows` output rows
// and `cols` output columns, and the tiles along M that gives.
struct MTiles {
  int kmt, nM;
};
MTiles m_tiles(int64_t rows, int cols, int cg, int sms) {
  const int64_t per = int64_t(BM) * cg;
  const int64_t nN = (cols + BN - 1) / BN;
  const int64_t two = (rows + 2 * per - 1) / (2 * per);
  if (pair_tiles(two * nN, sms / cg)) return MTiles{2, int(two)};
  return MTiles{1, int((rows + per - 1) / per)};
}

// Rows per block (a multiple of 128, or N) and vocabulary columns per chunk (a
// multiple of 256, or V rounded up to 256) of the recompute backward.
struct BwdPlan {
  int64_t rows;
  int vc;
};

// The recompute backward holds dZ for one block of rows and one chunk of the
// vocabulary at a time, at most dz_budget() bytes of bf16 whatever N and V.
// Several vocabulary chunks add an fp32 dH accumulator that the dH GEMM reads
// and writes once per extra chunk; several row blocks make the dW GEMM add
// into dW once per extra block. The plan takes the split with the least of
// that extra traffic (plus a fixed cost per block and chunk for the launches
// and the partial last wave).
BwdPlan bwd_plan(int64_t N, int32_t h, int32_t V) {
  const int64_t vpad = (int64_t(V) + BN - 1) / BN * BN;
  const double budget = double(dz_budget());
  BwdPlan best{N > 0 ? N : 1, int(vpad)};
  if (N <= 0 || double(N) * double(vpad) * 2.0 <= budget) return best;
  double best_cost = -1.0;
  const int64_t max_blocks = (N + BM - 1) / BM;
  for (int64_t nb = 1; nb <= max_blocks && nb <= 4096; ++nb) {
    int64_t rows = (N + nb - 1) / nb;
    rows = (rows + BM - 1) / BM * BM;
    if (rows > N) rows = N;
    const int64_t blocks = (N + rows - 1) / rows;
    if (blocks != nb) continue;  // the same split as a smaller nb
    int64_t vc = int64_t(budget / (2.0 * double(rows))) / BN * BN;
    if (vc < BN) vc = BN;
    if (vc > vpad) vc = vpad;
    const int64_t chunks = (V + vc - 1) / vc;
    const double nh = double(N) * double(h), vh = double(V) * double(h);
    double cost = double(chunks - 1) * nh * 8.0 + (chunks > 1 ? nh * 6.0 : 0.0) + double(blocks - 1) * vh * 8.0 +
                  double(blocks * chunks) * double(256 << 20);
    if (best_cost < 0.0 || cost < best_cost) {
      best_cost = cost;
      best = BwdPlan{rows, int(vc)};
    }
  }
  return best;
}

}  // namespace

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() { return encode_fn(); }

// Workspace of the log-prob calls: the forward's row compaction, tile
// partials and gathered logits; the backward's row compaction of one row
// block, its dZ chunk buffer and fp32 dH accumulator (recompute path; the
// cached path runs it on its flagged rows), after the cached path's row
// scales, scaled H rows and per-token flags.
size_t tc_ws_bytes(int64_t N, int32_t h, int32_t V) {
  const int64_t nvt = (int64_t(V) + BN - 1) / BN;
  const int64_t cap = (N + BM - 1) / BM * BM;
  const size_t fwd = compact_ws_bytes(N, h) + round256(sizeof(float2) * size_t(nvt) * size_t(N)) +
                     round256(sizeof(float) * size_t(N));
  const BwdPlan pl = bwd_plan(N, h, V);
  size_t rec = compact_ws_bytes(pl.rows, h) + round256(size_t(pl.rows) * size_t(pl.vc) * 2);
  if (pl.vc < V) rec += round256(size_t(pl.rows) * size_t(h) * sizeof(float));
  const size_t cached = round256(sizeof(float) * size_t(cap)) + round256(size_t(cap) * size_t(h) * 2) +
                        round256(size_t(N));
  const size_t bwd = cached + rec;
  return fwd > bwd ? fwd : bwd;
}

LogprobCache logprob_cache_view(void *base, int64_t N, int32_t V) {
  LogprobCache k;
  k.rows = (N + BM - 1) / BM * BM;
  k.lde = (int64_t(V) + 63) / 64 * 64;
  Carver c(base, ~size_t(0));
  k.e = c.take<__nv_bfloat16>(size_t(k.rows) * size_t(k.lde));
  k.idx = c.take<int>(size_t(N));
  k.pos = c.take<int>(size_t(N));
  k.count = c.take<int>(4);
  k.kappa = c.take<float>(size_t(N));
  k.flag = c.take<uint8_t>(size_t(N));
  k.bytes = c.off;
  return k;
}

sao_status tc_fwd(const void *H, const void *W, const int32_t *y, const uint8_t *row_mask, int64_t N, int32_t h,
                  int32_t V, float *logp, float *lse, unsigned int *err, void *ws, size_t ws_bytes,
                  const LogprobCache *cache, cudaStream_t s) {
  const int nvt = (V + BN - 1) / BN;
  Carver c(ws, ws_bytes);
  // Rows with row_mask == 0 are skipped: the GEMM runs on the compacted rows.
  CompactRows cr{};
  if (row_mask) SAO_TRY(compact_rows(row_mask, nullptr, N, static_cast<const __nv_bfloat16 *>(H), h, &cr, c, s));
  float2 *part = c.take<float2>(size_t(nvt) * size_t(N));
  float *zy = c.take<float>(size_t(N));
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for the log-prob forward");
  const void *A = row_mask ? static_cast<const void *>(cr.Hc) : H;
  CUtensorMap ma, mb;
  if (row_mask)
    SAO_TRY(make_map(&ma, cr.Hc, uint64_t(h), uint64_t(cr.cap), uint64_t(h), 64, BM));
  else
    SAO_TRY(make_map(&ma, H, uint64_t(h), uint64_t(N), uint64_t(h), 64, BM));
  // CTA pairs: each CTA of a pair loads half of the 256-row W tile
  const int cg = cta_group();
  SAO_TRY(make_map(&mb, W, uint64_t(h), uint64_t(V), uint64_t(h), 64, BN / cg));
  GemmParams p{};
  p.nM = int((N + BM * cg - 1) / (BM * cg));
  p.nN = nvt;
  p.nK = (h + BK - 1) / BK;
  // 64 row tiles per raster group (32 MB of H) stay in L2 while W streams: W is
  // read from HBM once per group, about 6 times per moe step instead of 25
  p.group_m = 64;
  p.rows = N;
  p.cols = V;
  p.y = y;
  p.vocab = V;
  p.part = part;
  p.zy = zy;
  p.err = err;
  if (row_mask) {
    p.m_count = cr.count;
    p.row_idx = cr.idx;
  }
  if (cache) {
    // the forward rows and their tokens, then each row's shift
    if (row_mask) {
      SAO_CUDA_TRY(cudaMemcpyAsync(cache->idx, cr.idx, sizeof(int) * size_t(N), cudaMemcpyDeviceToDevice, s));
      SAO_CUDA_TRY(cudaMemcpyAsync(cache->pos, cr.pos, sizeof(int) * size_t(N), cudaMemcpyDeviceToDevice, s));
      SAO_CUDA_TRY(cudaMemcpyAsync(cache->count, cr.count, sizeof(int), cudaMemcpyDeviceToDevice, s));
    } else {
      int slot = launch_begin("cache_rows", s);
      cache_identity_kernel<<<unsigned((N + 255) / 256), 256, 0, s>>>(cache->idx, cache->pos, cache->count, N);
      SAO_TRY(launch_end(slot, s));
    }
    int slot = launch_begin("cache_kappa", s);
    kappa_kernel<<<unsigned((N + kRowWarps - 1) / kRowWarps), 32 * kRowWarps, 0, s>>>(
        static_cast<const __nv_bfloat16 *>(A), h, static_cast<const __nv_bfloat16 *>(W), y, V, cache->idx,
        cache->count, cache->kappa, cache->flag);
    SAO_TRY(launch_end(slot, s));
    // also store e = exp(z - kappa)
    p.kappa = cache->kappa;
    p.flag = cache->flag;
    CUtensorMap me;
    SAO_TRY(make_map(&me, cache->e, uint64_t(V), uint64_t(cache->rows), uint64_t(cache->lde), 64, BM));
    SAO_TRY((launch_gemm_cfg<kSoftmaxStore, false, false>("tc_logits_lse_fwd", 1, cg, ma, mb, me, p, s)));
  } else {
    SAO_TRY((launch_gemm_cfg<kSoftmax, false, false>("tc_logits_lse_fwd", 1, cg, ma, mb, ma, p, s)));
  }
  SAO_TRY(lse_merge_launch(part, nvt, zy, y, nullptr, row_mask ? cr.pos : nullptr, N, V, logp, lse, err, s));
  if (cache) {
    int slot = launch_begin("cache_patch", s);
    patch_target_kernel<<<unsigned((N + 255) / 256), 256, 0, s>>>(cache->e, cache->lde, cache->idx, cache->count, y,
                                                                   V, zy, logp, cache->kappa, cache->flag);
    SAO_TRY(launch_end(slot, s));
  }
  return SAO_OK;
}

namespace {

// The backward with the logits recomputed, on the rows with mask[t] != 0
// (mask given) or G[t] != 0: dZ per vocabulary chunk by the dlogits GEMM, then
// dH and dW. overwrite_dH: dH is written on every row (zeros on inactive
// ones); otherwise only the active rows of dH are written. `names` label the
// three GEMMs' launches for the library's timers.
struct BwdNames {
  const char *dlogits, *dH, *dW;
};
constexpr BwdNames kBwdNames{"tc_dlogits", "tc_dH_gemm", "tc_dW_gemm"};
constexpr BwdNames kFlaggedNames{"flagged_dlogits", "flagged_dH_gemm", "flagged_dW_gemm"};

sao_status bwd_recompute_block(const void *H, const void *W, const int32_t *y, const float *lse, const float *G,
                               const uint8_t *mask, int64_t N, int32_t h, int32_t V, int Vc, void *dH, float *dW,
                               int accumulate, bool overwrite_dH, const BwdNames &names, unsigned int *err, Carver &c,
                               cudaStream_t s) {
  const bool multi = Vc < V;
  // Rows whose incoming gradient is zero contribute nothing: compact the rest.
  CompactRows cr{};
  SAO_TRY(compact_rows(mask, mask ? nullptr : G, N, static_cast<const __nv_bfloat16 *>(H), h, &cr, c, s));
  __nv_bfloat16 *dz = c.take<__nv_bfloat16>(size_t(N) * size_t(Vc));
  float *dh_acc = multi ? c.take<float>(size_t(N) * size_t(h)) : nullptr;
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for the log-prob backward");
  if (!multi && overwrite_dH) SAO_CUDA_TRY(cudaMemsetAsync(dH, 0, size_t(N) * size_t(h) * 2, s));

  CUtensorMap mHc_K, mW_K, mHc_MN, mW_MN;
  SAO_TRY(make_map(&mHc_K, cr.Hc, uint64_t(h), uint64_t(cr.cap), uint64_t(h), 64, BM));
  const int cg = cta_group();
  SAO_TRY(make_map(&mW_K, W, uint64_t(h), uint64_t(V), uint64_t(h), 64, BN / cg));
  SAO_TRY(make_map(&mHc_MN, cr.Hc, uint64_t(h), uint64_t(cr.cap), uint64_t(h), 64, 64));
  SAO_TRY(make_map(&mW_MN, W, uint64_t(h), uint64_t(V), uint64_t(h), 64, 64));
  DeviceInfo di;
  SAO_TRY(device_info(&di));
  const int sms = di.sm_count;

  for (int v0 = 0; v0 < V; v0 += Vc) {
    const int vc = (V - v0) < Vc ? (V - v0) : Vc;
    const bool first = (v0 == 0), last = (v0 + Vc >= V);
    CUtensorMap mZ_K, mZ_MN;
    SAO_TRY(make_map(&mZ_K, dz, uint64_t(vc), uint64_t(N), uint64_t(Vc), 64, BM));
    SAO_TRY(make_map(&mZ_MN, dz, uint64_t(vc), uint64_t(N), uint64_t(Vc), 64, 64));
    {  // dZ for vocabulary [v0, v0 + vc), compacted rows: recompute the logits
      GemmParams p{};
      p.nM = int((N + BM * cg - 1) / (BM * cg));
      p.nN = (vc + BN - 1) / BN;
      p.nK = (h + BK - 1) / BK;
      p.group_m = 64;  // as the forward
      p.b_row_off = v0;
      p.rows = N;
      p.cols = vc;
      p.y = y;
      p.vocab = V;
      p.v0 = v0;
      p.lse = lse;
      p.G = G;
      p.dz = dz;
      p.ldz = Vc;
      p.err = err;
      p.m_count = cr.count;
      p.row_idx = cr.idx;
      SAO_TRY((launch_gemm_cfg<kDLogits, false, false>(names.dlogits, 1, cg, mHc_K, mW_K, mZ_K, p, s)));
    }
    {  // dH (+)= dZ W[v0:v0+vc]: two 128-row tiles per CTA tile share each W stage when enough tiles remain
      GemmParams p{};
      const MTiles mt = m_tiles(N, h, cg, sms);
      p.nM = mt.nM;
      p.nN = (h + BN - 1) / BN;
      p.nK = (vc + BK - 1) / BK;
      p.group_m = 1;
      p.b_row_off = v0;
      p.rows = N;
      p.cols = h;
      p.ldc = h;
      p.err = err;
      p.m_count = cr.count;
      if (multi) {
        p.cf = dh_acc;  // compacted rows
        p.accumulate = first ? 0 : 1;
        SAO_TRY((launch_gemm_cfg<kStoreF32, false, true>(names.dH, mt.kmt, cg, mZ_K, mW_MN, mZ_K, p, s)));
      } else {
        p.cb = static_cast<__nv_bfloat16 *>(dH);
        p.row_idx = cr.idx;  // scatter to the original rows
        SAO_TRY((launch_gemm_cfg<kStoreBF16, false, true>(names.dH, mt.kmt, cg, mZ_K, mW_MN, mZ_K, p, s)));
      }
    }
    {  // dW[v0:v0+vc] (+)= dZ^T H over the compacted tokens: two 128-row vocabulary tiles per CTA tile
      GemmParams p{};
      const MTiles mt = m_tiles(vc, h, cg, sms);
      p.nM = mt.nM;
      p.nN = (h + BN - 1) / BN;
      p.nK = int((N + BK - 1) / BK);
      p.group_m = 1;
      p.rows = vc;
      p.cols = h;
      p.cf = dW;
      p.ldc = h;
      p.c_row_off = v0;
      p.accumulate = accumulate;
      p.err = err;
      p.k_count = cr.count;
      SAO_TRY((launch_gemm_cfg<kStoreF32, true, true>(names.dW, mt.kmt, cg, mZ_MN, mHc_MN, mZ_MN, p, s)));
    }
    if (multi && last)
      SAO_TRY(scatter_rows_to_bf16(dh_acc, h, cr.pos, cr.idx, cr.count, N, static_cast<__nv_bfloat16 *>(dH),
                                   overwrite_dH, s));
  }
  return SAO_OK;
}

// The whole backward: one bwd_recompute_block per block of rows of the plan,
// each on its own slice of H, y, lse, G, the mask and dH, all adding into dW
// after the first; the blocks reuse the same scratch in stream order.
sao_status bwd_recompute(const void *H, const void *W, const int32_t *y, const float *lse, const float *G,
                         const uint8_t *mask, int64_t N, int32_t h, int32_t V, void *dH, float *dW, int accumulate,
                         bool overwrite_dH, const BwdNames &names, unsigned int *err, Carver &c, cudaStream_t s) {
  const BwdPlan pl = bwd_plan(N, h, V);
  const __nv_bfloat16 *Hb = static_cast<const __nv_bfloat16 *>(H);
  __nv_bfloat16 *dHb = static_cast<__nv_bfloat16 *>(dH);
  for (int64_t r0 = 0; r0 < N; r0 += pl.rows) {
    const int64_t nr = (N - r0) < pl.rows ? (N - r0) : pl.rows;
    Carver cb = c;
    SAO_TRY(bwd_recompute_block(Hb + r0 * h, W, y + r0, lse + r0, G + r0, mask ? mask + r0 : nullptr, nr, h, V,
                                pl.vc, dHb + r0 * h, dW, r0 == 0 ? accumulate : 1, overwrite_dH, names, err, cb,
                                s));
  }
  return SAO_OK;
}

}  // namespace

sao_status tc_bwd(const void *H, const void *W, const int32_t *y, const float *lse, const float *G, int64_t N,
                  int32_t h, int32_t V, void *dH, float *dW, int accumulate, unsigned int *err, void *ws,
                  size_t ws_bytes, const LogprobCache *cache, cudaStream_t s) {
  Carver c(ws, ws_bytes);
  if (!cache) return bwd_recompute(H, W, y, lse, G, nullptr, N, h, V, dH, dW, accumulate, true, kBwdNames, err, c, s);

  // From the stored probabilities: dZ[f, .] = sc[f] e[f, .] with sc[f] =
  // -G exp(kappa - lse), so dH[t] = sc[f] (e W)[f] (row scale in the GEMM's
  // epilogue) and dW = e^T (sc H) over the forward rows.
  const int64_t cap = cache->rows;
  float *sc = c.take<float>(size_t(cap));
  __nv_bfloat16 *Hs = c.take<__nv_bfloat16>(size_t(cap) * size_t(h));
  uint8_t *fb = c.take<uint8_t>(size_t(N));
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for the log-prob backward");
  SAO_CUDA_TRY(cudaMemsetAsync(dH, 0, size_t(N) * size_t(h) * 2, s));
  int slot = launch_begin("cache_scales", s);
  bwd_token_kernel<<<unsigned((N + 255) / 256), 256, 0, s>>>(G, cache->pos, cache->flag, N, fb, err);
  bwd_scale_kernel<<<unsigned((cap + kRowWarps - 1) / kRowWarps), 32 * kRowWarps, 0, s>>>(
      static_cast<const __nv_bfloat16 *>(H), h, cache->idx, cache->count, G, lse, cache->kappa, cache->flag, sc, Hs,
      cap);
  SAO_TRY(launch_end(slot, s));

  CUtensorMap mE_K, mE_MN, mW_MN, mHs_MN;
  SAO_TRY(make_map(&mE_K, cache->e, uint64_t(V), uint64_t(cap), uint64_t(cache->lde), 64, BM));
  SAO_TRY(make_map(&mE_MN, cache->e, uint64_t(V), uint64_t(cap), uint64_t(cache->lde), 64, 64));
  SAO_TRY(make_map(&mW_MN, W, uint64_t(h), uint64_t(V), uint64_t(h), 64, 64));
  SAO_TRY(make_map(&mHs_MN, Hs, uint64_t(h), uint64_t(cap), uint64_t(h), 64, 64));
  DeviceInfo di;
  SAO_TRY(device_info(&di));
  const int sms = di.sm_count;
  const int cg = cta_group();
  {  // dH[t] = sc[f] (e W)[f], scattered to the tokens: two 128-row tiles per CTA tile share each W stage
    GemmParams p{};
    const MTiles mt = m_tiles(N, h, cg, sms);
    p.nM = mt.nM;
    p.nN = (h + BN - 1) / BN;
    p.nK = (V + BK - 1) / BK;
    p.group_m = 1;
    p.rows = N;
    p.cols = h;
    p.ldc = h;
    p.err = err;
    p.m_count = cache->count;
    p.row_idx = cache->idx;
    p.row_scale = sc;
    p.cb = static_cast<__nv_bfloat16 *>(dH);
    SAO_TRY((launch_gemm_cfg<kStoreBF16, false, true>("tc_dH_gemm", mt.kmt, cg, mE_K, mW_MN, mE_K, p, s)));
  }
  {  // dW (+)= e^T (sc H) over the forward rows: two 128-row vocabulary tiles per CTA tile
    GemmParams p{};
    const MTiles mt = m_tiles(V, h, cg, sms);
    p.nM = mt.nM;
    p.nN = (h + BN - 1) / BN;
    p.nK = int((N + BK - 1) / BK);
    p.group_m = 1;
    p.rows = V;
    p.cols = h;
    p.cf = dW;
    p.ldc = h;
    p.accumulate = accumulate;
    p.err = err;
    p.k_count = cache->count;
    SAO_TRY((launch_gemm_cfg<kStoreF32, true, true>("tc_dW_gemm", mt.kmt, cg, mE_MN, mHs_MN, mE_MN, p, s)));
  }
  // Flagged rows (a sampled token more than kFlagExponent - kKappaOffset nats
  // below its row's maximum) got sc = 0 above: recompute their logits, write
  // their dH rows and add their dW. With none, these GEMMs find no rows.
  return bwd_recompute(H, W, y, lse, G, fb, N, h, V, dH, dW, 1, false, kFlaggedNames, err, c, s);
}

}  // namespace sao
