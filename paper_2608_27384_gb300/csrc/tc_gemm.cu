// bf16 GEMM on the 5th-generation tensor cores (tcgen05) of sm_103a.
//
//   C[M, N] = A[M, K] * B[N, K]^T      A = activations, B = weights (both K-major)
//
// One CTA computes one 128 x BN output tile (optionally one K-slice of it):
//   warp 0      TMA producer: 128x64 A and BNx64 B tiles, 128-byte swizzle,
//               into a STAGES-deep shared-memory ring (full/empty mbarriers);
//   warp 1      allocates BN TMEM columns; one lane issues tcgen05.mma
//               (M=128, N=BN, K=16) into the fp32 accumulator in TMEM and
//               frees ring slots with tcgen05.commit;
//   warps 2..5  epilogue: tcgen05.ld of the accumulator (one TMEM lane = one
//               output row per thread), fused post-processing, global stores.
// Epilogues (GemmMode): bias (fp32 out), bias+SiLU (bf16 out), split-K partial
// planes (fp32 or bf16), RoPE + q / KV-workspace scatter for the packed QKV
// projection, and tanh-GELU(gate) * up for the packed gate/up projection.
// Two more forms share the epilogues: a persistent weight-streaming kernel for
// at most 16 rows (the FiLM projection) and a persistent multi-tile kernel with
// two TMEM accumulators for shapes with many more tiles than SMs.
// Every wait is bounded (common.cuh); on timeout the kernel records an error
// code and finishes without touching the accumulator.
#include "common.cuh"
#include "gemm_epilogue.cuh"
#include "kernels.h"

namespace fva {

namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;  // 64 bf16 = 128 bytes = one swizzle row
constexpr int kThreads = 192;
// rows of the FiLM condition (one 16-row TMA box)
constexpr int kStreamRows = 16;

template <int BN>
struct GemmCfg {
  static constexpr int kABytes = kBM * kBK * 2;
  static constexpr int kBBytes = BN * kBK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kStages = (BN <= 64) ? 8 : (BN <= 128 ? 6 : 4);
  static constexpr int kTmemCols = BN < 32 ? 32 : BN;
  static constexpr int kSmemBytes = kStages * kStageBytes + 1024 /*align*/ + 256 /*barriers*/;
  // full[kStages], empty[kStages], acc_full and the TMEM slot fit the 256-byte area
  static_assert((2 * kStages + 1) * 8 + 4 <= 256, "barrier area too small for the ring");
  static_assert(kSmemBytes <= 227 * 1024, "shared memory above the per-CTA limit");
};

// One FiLM column tile (kFilmTile wide) in a CTA of a projection's launch
// (FilmTiles): out = cond W^T + bias for the <= 16 condition rows, the same MMA
// sequence and epilogue as the FiLM kernel.  Its own layout of the host kernel's
// ring (kRingBytes): the condition rows of every k-block (16-row boxes, 2 KB each)
// in one area and the weights in a ring of up to 14 stages, a few of which are
// requested before the dependency wait (the weights depend on nothing; only the
// condition, written earlier in the step, is loaded after it).  The M = 128 MMA
// reads 112 rows past each condition box (later boxes and the ring): those
// accumulator rows are garbage and never stored.
constexpr int kFilmMaxKb = 16;  // K <= 1024

template <int kRingBytes>
struct FilmCfg {
  static constexpr int kABox = kStreamRows * kBK * 2;  // 2 KB
  static constexpr int kMaxKb = kFilmMaxKb;
  static constexpr int kABytes = kMaxKb * kABox;
  static constexpr int kBBytes = kFilmTile * kBK * 2;
  static constexpr int kStages =
      (kRingBytes - kABytes) / kBBytes < 14 ? (kRingBytes - kABytes) / kBBytes : 14;
  // fullB[kStages], emptyB[kStages], fullA, acc_full and the TMEM slot in 256 bytes
  static_assert((2 * kStages + 2) * 8 + 4 <= 256, "barrier area too small");
  static_assert(kStages >= 4 && kABytes + kStages * kBBytes <= kRingBytes,
                "FiLM layout beyond the ring");
};

template <int kRingBytes>
__device__ void film_tile_cta(const FilmTiles& fj, uint8_t* smem, uint8_t* bar_area, int n0,
                              int nkb, int* err) {
  using F = FilmCfg<kRingBytes>;
  constexpr int BN = kFilmTile;
  uint64_t* fullB = (uint64_t*)bar_area;
  uint64_t* emptyB = fullB + F::kStages;
  uint64_t* fullA = emptyB + F::kStages;
  uint64_t* acc_full = fullA + 1;
  uint32_t* tmem_slot = (uint32_t*)(acc_full + 1);
  uint8_t* sA = smem;
  uint8_t* sB = smem + F::kABytes;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < F::kStages; ++s) {
      mbar_init(&fullB[s], 1);
      mbar_init(&emptyB[s], 1);
    }
    mbar_init(fullA, 1);
    mbar_init(acc_full, 1);
    fence_barrier_init();
    tma_prefetch_desc(&fj.a);
    tma_prefetch_desc(&fj.b);
  }
  if (warp == 1) tmem_alloc(tmem_slot, BN);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();

  if (warp == 0 && lane == 0) {
    // fj.pre_stages weight stages before the wait: inside a projection's launch a
    // few (more of them in flight while the previous kernel runs slowed the step
    // down: 4 measured best on GB300), alone all that fit
    const int pre = min(nkb, min(F::kStages, max(1, fj.pre_stages)));
    for (int i = 0; i < pre; ++i) {
      mbar_arrive_expect_tx(&fullB[i], F::kBBytes);
      tma_load_2d(sB + i * F::kBBytes, &fj.b, i * kBK, n0, &fullB[i]);
    }
    pdl_wait();
    mbar_arrive_expect_tx(fullA, (uint32_t)(nkb * F::kABox));
    for (int i = 0; i < nkb; ++i) tma_load_2d(sA + i * F::kABox, &fj.a, i * kBK, 0, fullA);
    for (int i = pre; i < nkb; ++i) {
      const int s = i % F::kStages;
      if (!mbar_wait(&emptyB[s], ((uint32_t)(i / F::kStages) & 1u) ^ 1u, err, KERR_WAIT_MMA))
        break;
      mbar_arrive_expect_tx(&fullB[s], F::kBBytes);
      tma_load_2d(sB + s * F::kBBytes, &fj.b, i * kBK, n0, &fullB[s]);
    }
  } else if (warp == 1 && lane == 0) {
    constexpr uint32_t idesc = umma_idesc_bf16(kBM, BN, false);
    const uint64_t a0 = umma_desc_sw128(smem_u32(sA), 16, 1024);
    const uint64_t b0 = umma_desc_sw128(smem_u32(sB), 16, 1024);
    bool good = mbar_wait(fullA, 0, err, KERR_WAIT_TMA);
    for (int i = 0; good && i < nkb; ++i) {
      const int s = i % F::kStages;
      if (!mbar_wait(&fullB[s], (uint32_t)(i / F::kStages) & 1u, err, KERR_WAIT_TMA)) {
        good = false;
        break;
      }
      tc_fence_after();
      const uint64_t ad = desc_advance(a0, i * F::kABox);
      const uint64_t bd = desc_advance(b0, s * F::kBBytes);
#pragma unroll
      for (int kk = 0; kk < kBK / 16; ++kk)
        umma_bf16(tmem, ad + 2 * kk, bd + 2 * kk, idesc, (i > 0 || kk > 0) ? 1u : 0u);
      umma_commit(&emptyB[s]);
    }
    if (good) umma_commit(acc_full);
  } else if (warp >= 2) {
    // the GEMM_BIAS_F32 epilogue (fp32 out = acc + bias, the same single rounding),
    // with the tile's bias fetched before the accumulator is ready: lane l holds
    // column c + l of every 32-column chunk c and hands it to the warp by shuffle.
    // Only the warp of TMEM lanes 0-31 has condition rows.
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    float bl[BN / 32];
#pragma unroll
    for (int c = 0; c < BN / 32; ++c) bl[c] = __ldg(fj.bias + n0 + c * 32 + lane);
    const bool good = __all_sync(0xffffffffu, mbar_wait(acc_full, 0, err, KERR_WAIT_MMA));
    tc_fence_after();
    if (good && nkb > 0 && quarter * 32 < fj.rows) {
      // every MMA is complete: the condition area is free to stage the stores
      const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
      uint8_t* stage = smem + (warp - 2) * (32 * 144);
      float* dst = row < fj.rows ? fj.out + (size_t)row * fj.ldo + n0 : nullptr;
#pragma unroll
      for (int c = 0; c < BN / 32; ++c) {
        float v[32];
        tmem_ld32(trow + c * 32, v);
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] += __shfl_sync(0xffffffffu, bl[c], i);
        uint4 u[8];
        pack_f32x32(v, u);
        warp_store_rows<128>(stage, u, dst ? dst + c * 32 : nullptr, lane);
      }
    }
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, BN);
  }
}

template <int BN, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const GemmEpi ep, int M, int N, int kb_total, int kb_per_split,
                   const __grid_constant__ FilmTiles fj) {
  using C = GemmCfg<BN>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint64_t* full = (uint64_t*)(smem + C::kStages * C::kStageBytes);
  uint64_t* empty = full + C::kStages;
  uint64_t* acc_full = empty + C::kStages;
  uint32_t* tmem_slot = (uint32_t*)(acc_full + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // the QKV and gate/up projections' launches may carry FiLM column tiles in extra
  // CTAs (grid.y >= fj.y0; same K, one split)
  if constexpr (MODE == GEMM_QKV_ROPE || MODE == GEMM_GEGLU) {
    if ((int)blockIdx.y >= fj.y0) {
      const int f = ((int)blockIdx.y - fj.y0) * (int)gridDim.x + (int)blockIdx.x;
      if (f < fj.tiles)  // uniform over the CTA
        film_tile_cta<C::kStages * C::kStageBytes>(fj, smem, (uint8_t*)full,
                                                   (fj.tile0 + f) * kFilmTile, kb_total, ep.err);
      return;
    }
  }
  const int m0 = blockIdx.x * kBM, n0 = blockIdx.y * BN;
  const int split = blockIdx.z;
  const int kb0 = split * kb_per_split;
  const int nkb = min(kb_total, kb0 + kb_per_split) - kb0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(acc_full, 1);
    fence_barrier_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  // Only one CTA of any tcgen05 kernel of this library fits on an SM (each uses
  // more than half of the shared memory), so this allocation never waits.
  if (warp == 1) tmem_alloc(tmem_slot, C::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer
    // The weights (B) do not depend on earlier kernels: the first ring stages of
    // B are requested before waiting for the predecessor grid.  A (activations)
    // and everything downstream of it come after the wait; the MMA and epilogue
    // threads only run behind these loads, so they are ordered after it too.
    // a short A box (every row fits a_rows < 128) writes part of the A stage: the
    // MMA's later rows then read stale shared memory and are never stored
    const uint32_t stage_tx = (uint32_t)(ep.a_rows > 0 ? ep.a_rows : kBM) * kBK * 2 + C::kBBytes;
    const int pre = min(nkb, C::kStages);
    for (int i = 0; i < pre; ++i) {
      mbar_arrive_expect_tx(&full[i], stage_tx);
      tma_load_2d(smem + i * C::kStageBytes + C::kABytes, &tmB, (kb0 + i) * kBK, n0, &full[i]);
    }
    if (ep.pf_count > 0 && blockIdx.x == 0 && blockIdx.y == 0 && blockIdx.z == 0)
      for (int i = 0; i < ep.pf_count; ++i) prefetch_l2(ep.pf_base + i * ep.pf_stride, ep.pf_bytes);
    pdl_wait();
    for (int i = 0; i < pre; ++i)
      tma_load_2d(smem + i * C::kStageBytes, &tmA, (kb0 + i) * kBK, m0, &full[i]);
    for (int i = pre; i < nkb; ++i) {
      const int s = i % C::kStages;
      const uint32_t ph = (uint32_t)(i / C::kStages) & 1u;
      if (!mbar_wait(&empty[s], ph ^ 1u, ep.err, KERR_WAIT_MMA)) break;
      uint8_t* sa = smem + s * C::kStageBytes;
      mbar_arrive_expect_tx(&full[s], stage_tx);
      tma_load_2d(sa, &tmA, (kb0 + i) * kBK, m0, &full[s]);
      tma_load_2d(sa + C::kABytes, &tmB, (kb0 + i) * kBK, n0, &full[s]);
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer
    constexpr uint32_t idesc = umma_idesc_bf16(kBM, BN, false);
    const uint64_t d0 = umma_desc_sw128(smem_u32(smem), 16, 1024);  // A of stage 0
    bool good = true;
    int s = 0;
    uint32_t ph = 0;
    for (int i = 0; i < nkb; ++i) {
      if (!mbar_wait(&full[s], ph, ep.err, KERR_WAIT_TMA)) {
        good = false;
        break;
      }
      tc_fence_after();
      const uint64_t ad = desc_advance(d0, s * C::kStageBytes);
      const uint64_t bd = desc_advance(ad, C::kABytes);
#pragma unroll
      for (int kk = 0; kk < kBK / 16; ++kk)  // 16 bf16 = 32 bytes along K per step
        umma_bf16(tmem, ad + 2 * kk, bd + 2 * kk, idesc, (i > 0 || kk > 0) ? 1u : 0u);
      umma_commit(&empty[s]);
      if (++s == C::kStages) {
        s = 0;
        ph ^= 1u;
      }
    }
    if (good) umma_commit(acc_full);
  } else if (warp >= 2) {
    // ---------------- epilogue: warp w reads TMEM lanes 32*(w%4) .. +31
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    uint4 rh[MODE == GEMM_QKV_ROPE ? BN / 8 : 1];
    if constexpr (MODE == GEMM_QKV_ROPE) gemm_epilogue_load_rope<BN>(ep, m0 + row, M, n0, rh);
    const bool good = __all_sync(0xffffffffu, mbar_wait(acc_full, 0, ep.err, KERR_WAIT_MMA));
    tc_fence_after();
    if (good && nkb > 0) {
      // all MMAs (and so all TMA loads into the ring) are complete: the ring's
      // first stage is free to stage this warp's coalesced stores
      const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
      uint8_t* stage = smem + (warp - 2) * (32 * 144);
      if constexpr (MODE == GEMM_QKV_ROPE)
        gemm_epilogue_qkv<BN>(ep, trow, m0 + row, M, n0, stage, lane, rh);
      else
        gemm_epilogue<BN, MODE>(ep, trow, m0 + row, M, n0, split, stage, lane);
    }
  }
  // the producer and MMA lanes rejoin their warps first: a CTA barrier reached
  // by a split warp does not wait for the rest of the CTA
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

// ---------------------------------------------------------------------------
// Persistent variant for weight streaming (the FiLM projection: M = B*K rows,
// hundreds of column tiles).  Two CTAs per SM walk column tiles
// blockIdx.x, blockIdx.x + gridDim.x, ...; the producer streams every tile's
// k-blocks through one ring without draining between tiles, and the MMA
// alternates between two TMEM accumulators so a tile's epilogue overlaps the next
// tile's MMAs.  M <= 128 (one row tile).
// ---------------------------------------------------------------------------
// The condition has at most kStreamRows rows, and each stage holds only those rows
// of A.  The M = 128 MMA reads 112 more rows past them (the stage's weights):
// those accumulator rows are garbage and never stored, and the small A region
// leaves room for a deeper weight ring.

template <int BN>
struct GemmStreamCfg {
  static constexpr int kABytes = kStreamRows * kBK * 2;  // 2 KB, 1024-byte aligned
  static constexpr int kATx = kABytes;
  static constexpr int kBBytes = BN * kBK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  // two CTAs per SM (two independent weight streams per SM read HBM faster than
  // one with a ring twice as deep: FiLM 53.7 -> 48.7 us on GB300), each with as many
  // ring stages as fit in half the shared memory next to the barriers and the
  // epilogue stages; TMEM: 2 x 2 x BN = 512 columns per SM
  static constexpr int kCtasPerSm = 2;
  static constexpr int kEpiBytes = 4 * 32 * 144;
  static constexpr int kStages = (113 * 1024 - 1024 - 256 - kEpiBytes) / kStageBytes;
  // ring + barriers (256 B) + four 32 x 144 B epilogue stages
  static constexpr int kSmemBytes = kStages * kStageBytes + 1024 + 256 + kEpiBytes;
  // full[kStages], empty[kStages], acc_full[2], acc_empty[2], drain and the TMEM slot
  static_assert((2 * kStages + 5) * 8 + 4 <= 256, "barrier area too small for the ring");
  static_assert(kSmemBytes <= 227 * 1024, "shared memory above the per-CTA limit");
};

template <int BN, int MODE>
__global__ void __launch_bounds__(kThreads, GemmStreamCfg<BN>::kCtasPerSm)
    tc_gemm_stream_kernel(const __grid_constant__ CUtensorMap tmA,
                          const __grid_constant__ CUtensorMap tmB, const GemmEpi ep, int M,
                          int n_tiles, int nkb) {
  using C = GemmStreamCfg<BN>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint64_t* full = (uint64_t*)(smem + C::kStages * C::kStageBytes);
  uint64_t* empty = full + C::kStages;
  uint64_t* acc_full = empty + C::kStages;  // [2]
  uint64_t* acc_empty = acc_full + 2;       // [2]
  uint64_t* drain = acc_empty + 2;
  uint32_t* tmem_slot = (uint32_t*)(drain + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 4);  // one arrival per epilogue warp
    }
    mbar_init(drain, 1);
    fence_barrier_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  // the two CTAs an SM holds take 2 x 2 BN = 512 TMEM columns together: the
  // allocation never waits (no other tcgen05 kernel's CTA fits next to them)
  if (warp == 1) tmem_alloc(tmem_slot, 2 * BN);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer: weights of the first stages before the wait
    // the first tile's first stages: weights before waiting for the predecessor,
    // which writes A (the condition rows)
    const int pre = (int)blockIdx.x < n_tiles ? min(nkb, C::kStages) : 0;
    for (int i = 0; i < pre; ++i) {
      mbar_arrive_expect_tx(&full[i], C::kATx + C::kBBytes);
      tma_load_2d(smem + i * C::kStageBytes + C::kABytes, &tmB, i * kBK, blockIdx.x * BN, &full[i]);
    }
    pdl_wait();
    for (int i = 0; i < pre; ++i) tma_load_2d(smem + i * C::kStageBytes, &tmA, i * kBK, 0, &full[i]);
    uint32_t it = 0;
    bool ok = true;
    for (int t = blockIdx.x; ok && t < n_tiles; t += gridDim.x) {
      const int n0 = t * BN;
      for (int i = 0; i < nkb; ++i, ++it) {
        if (it < (uint32_t)pre) continue;  // issued above
        const int s = it % C::kStages;
        if (!mbar_wait(&empty[s], ((it / C::kStages) & 1u) ^ 1u, ep.err, KERR_WAIT_MMA)) {
          ok = false;
          break;
        }
        uint8_t* sa = smem + s * C::kStageBytes;
        mbar_arrive_expect_tx(&full[s], C::kATx + C::kBBytes);
        tma_load_2d(sa + C::kABytes, &tmB, i * kBK, n0, &full[s]);
        tma_load_2d(sa, &tmA, i * kBK, 0, &full[s]);
      }
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer
    constexpr uint32_t idesc = umma_idesc_bf16(kBM, BN, false);
    const uint64_t d0 = umma_desc_sw128(smem_u32(smem), 16, 1024);  // A of stage 0
    uint32_t it = 0, acc = 0, rph = 0;
    int rs = 0;
    bool ok = true;
    for (int t = blockIdx.x; ok && t < n_tiles; t += gridDim.x, ++acc) {
      const uint32_t buf = acc & 1u;
      if (!mbar_wait(&acc_empty[buf], ((acc >> 1) & 1u) ^ 1u, ep.err, KERR_WAIT_SYNC)) break;
      tc_fence_after();
      const uint32_t d = tmem + buf * BN;
      for (int i = 0; i < nkb; ++i, ++it) {
        if (!mbar_wait(&full[rs], rph, ep.err, KERR_WAIT_TMA)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint64_t ad = desc_advance(d0, rs * C::kStageBytes);
        const uint64_t bd = desc_advance(ad, C::kABytes);
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk)  // 16 bf16 = 32 bytes along K per step
          umma_bf16(d, ad + 2 * kk, bd + 2 * kk, idesc, (i > 0 || kk > 0) ? 1u : 0u);
        umma_commit(&empty[rs]);
        if (++rs == C::kStages) {
          rs = 0;
          rph ^= 1u;
        }
      }
      if (ok) umma_commit(&acc_full[buf]);
    }
    // every MMA of this thread completes before TMEM is released
    umma_commit(drain);
    mbar_wait(drain, 0, nullptr, 0);
  } else if (warp >= 2) {
    // ---------------- epilogue: one output row per thread
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    uint8_t* stage = smem + C::kStages * C::kStageBytes + 256 + (warp - 2) * (32 * 144);
    uint32_t acc = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++acc) {
      const uint32_t buf = acc & 1u;
      if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&acc_full[buf], (acc >> 1) & 1u, ep.err,
                                                     KERR_WAIT_MMA));
      if (!ok) break;
      tc_fence_after();
      const uint32_t trow = tmem + buf * BN + ((uint32_t)(quarter * 32) << 16);
      gemm_epilogue<BN, MODE>(ep, trow, row, M, t * BN, 0, stage, lane);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[buf]);
    }
  }
  // the producer and MMA lanes rejoin their warps first: a CTA barrier reached
  // by a split warp does not wait for the rest of the CTA
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 2 * BN);
  }
}

// ---------------------------------------------------------------------------
// Persistent form of the per-op GEMM for shapes with many more tiles than SMs:
// each CTA walks tiles t = blockIdx.x, + gridDim.x, ... (row tile t % m_tiles,
// column tile t / m_tiles, so concurrent CTAs share a weight tile) through one
// continuous load ring, with two TMEM accumulators so that the epilogue of one
// tile runs under the MMAs of the next.  No split-K.
// ---------------------------------------------------------------------------
template <int BN>
struct GemmPersistCfg {
  static constexpr int kABytes = kBM * kBK * 2;
  static constexpr int kBBytes = BN * kBK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kEpiBytes = 4 * 32 * 144;
  static constexpr int kStages = (227 * 1024 - 1024 - 256 - kEpiBytes) / kStageBytes;
  static constexpr int kSmemBytes = kStages * kStageBytes + 1024 + 256 + kEpiBytes;
  // full[kStages], empty[kStages], acc_full[2], acc_empty[2], drain and the TMEM slot
  static_assert((2 * kStages + 5) * 8 + 4 <= 256, "barrier area too small for the ring");
  static_assert(kSmemBytes <= 227 * 1024, "shared memory above the per-CTA limit");
  static_assert(2 * BN <= 512, "two accumulators must fit TMEM");
};

template <int BN, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    tc_gemm_persist_kernel(const __grid_constant__ CUtensorMap tmA,
                           const __grid_constant__ CUtensorMap tmB, const GemmEpi ep, int M,
                           int m_tiles, int n_tiles, int nkb) {
  using C = GemmPersistCfg<BN>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint64_t* full = (uint64_t*)(smem + C::kStages * C::kStageBytes);
  uint64_t* empty = full + C::kStages;
  uint64_t* acc_full = empty + C::kStages;  // [2]
  uint64_t* acc_empty = acc_full + 2;       // [2]
  uint64_t* drain = acc_empty + 2;
  uint32_t* tmem_slot = (uint32_t*)(drain + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tiles = m_tiles * n_tiles;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 4);  // one arrival per epilogue warp
    }
    mbar_init(drain, 1);
    fence_barrier_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) tmem_alloc(tmem_slot, 2 * BN);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer: the first tile's weight stages go out
    // before waiting for the predecessor grid, which writes A
    const int t0 = blockIdx.x;
    const int pre = t0 < tiles ? min(nkb, C::kStages) : 0;
    for (int i = 0; i < pre; ++i) {
      mbar_arrive_expect_tx(&full[i], C::kStageBytes);
      tma_load_2d(smem + i * C::kStageBytes + C::kABytes, &tmB, i * kBK, (t0 / m_tiles) * BN,
                  &full[i]);
    }
    pdl_wait();
    for (int i = 0; i < pre; ++i)
      tma_load_2d(smem + i * C::kStageBytes, &tmA, i * kBK, (t0 % m_tiles) * kBM, &full[i]);
    uint32_t it = 0;
    bool ok = true;
    for (int t = t0; ok && t < tiles; t += gridDim.x) {
      const int m0 = (t % m_tiles) * kBM, n0 = (t / m_tiles) * BN;
      for (int i = 0; i < nkb; ++i, ++it) {
        if (it < (uint32_t)pre) continue;  // issued above
        const int s = it % C::kStages;
        if (!mbar_wait(&empty[s], ((it / C::kStages) & 1u) ^ 1u, ep.err, KERR_WAIT_MMA)) {
          ok = false;
          break;
        }
        uint8_t* sa = smem + s * C::kStageBytes;
        mbar_arrive_expect_tx(&full[s], C::kStageBytes);
        tma_load_2d(sa, &tmA, i * kBK, m0, &full[s]);
        tma_load_2d(sa + C::kABytes, &tmB, i * kBK, n0, &full[s]);
      }
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer
    constexpr uint32_t idesc = umma_idesc_bf16(kBM, BN, false);
    const uint64_t d0 = umma_desc_sw128(smem_u32(smem), 16, 1024);  // A of stage 0
    uint32_t it = 0, acc = 0, rph = 0;
    int rs = 0;
    bool ok = true;
    for (int t = blockIdx.x; ok && t < tiles; t += gridDim.x, ++acc) {
      const uint32_t buf = acc & 1u;
      if (!mbar_wait(&acc_empty[buf], ((acc >> 1) & 1u) ^ 1u, ep.err, KERR_WAIT_SYNC)) break;
      tc_fence_after();
      const uint32_t d = tmem + buf * BN;
      for (int i = 0; i < nkb; ++i, ++it) {
        if (!mbar_wait(&full[rs], rph, ep.err, KERR_WAIT_TMA)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint64_t ad = desc_advance(d0, rs * C::kStageBytes);
        const uint64_t bd = desc_advance(ad, C::kABytes);
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk)  // 16 bf16 = 32 bytes along K per step
          umma_bf16(d, ad + 2 * kk, bd + 2 * kk, idesc, (i > 0 || kk > 0) ? 1u : 0u);
        umma_commit(&empty[rs]);
        if (++rs == C::kStages) {
          rs = 0;
          rph ^= 1u;
        }
      }
      if (ok) umma_commit(&acc_full[buf]);
    }
    // every MMA of this thread completes before TMEM is released
    umma_commit(drain);
    mbar_wait(drain, 0, nullptr, 0);
  } else if (warp >= 2) {
    // ---------------- epilogue: one output row per thread
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    uint8_t* stage = smem + C::kStages * C::kStageBytes + 256 + (warp - 2) * (32 * 144);
    uint32_t acc = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++acc) {
      const int m0 = (t % m_tiles) * kBM, n0 = (t / m_tiles) * BN;
      const uint32_t buf = acc & 1u;
      uint4 rh[MODE == GEMM_QKV_ROPE ? BN / 8 : 1];
      if constexpr (MODE == GEMM_QKV_ROPE) gemm_epilogue_load_rope<BN>(ep, m0 + row, M, n0, rh);
      if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&acc_full[buf], (acc >> 1) & 1u, ep.err,
                                                     KERR_WAIT_MMA));
      if (!ok) break;
      tc_fence_after();
      const uint32_t trow = tmem + buf * BN + ((uint32_t)(quarter * 32) << 16);
      if constexpr (MODE == GEMM_QKV_ROPE)
        gemm_epilogue_qkv<BN>(ep, trow, m0 + row, M, n0, stage, lane, rh);
      else
        gemm_epilogue<BN, MODE>(ep, trow, m0 + row, M, n0, 0, stage, lane);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[buf]);
    }
  }
  // the producer and MMA lanes rejoin their warps first: a CTA barrier reached
  // by a split warp does not wait for the rest of the CTA
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 2 * BN);
  }
}

template <int BN, int MODE>
cudaError_t set_attr_persist() {
  return cudaFuncSetAttribute(tc_gemm_persist_kernel<BN, MODE>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize,
                              GemmPersistCfg<BN>::kSmemBytes);
}

template <int BN, int MODE>
cudaError_t launch_persist(const CUtensorMap* a, const CUtensorMap* b, const GemmEpi& ep, int M,
                           int N, int K, int grid, cudaStream_t s) {
  const int m_tiles = (M + kBM - 1) / kBM, n_tiles = N / BN;
  return launch_pdl(tc_gemm_persist_kernel<BN, MODE>, dim3(std::min(grid, m_tiles * n_tiles)),
                    dim3(kThreads), GemmPersistCfg<BN>::kSmemBytes, s, *a, *b, ep, M, m_tiles,
                    n_tiles, K / kBK);
}

template <int BN, int MODE>
cudaError_t set_attr() {
  return cudaFuncSetAttribute(tc_gemm_kernel<BN, MODE>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize,
                              GemmCfg<BN>::kSmemBytes);
}

template <int BN, int MODE>
cudaError_t launch(const CUtensorMap* a, const CUtensorMap* b, const GemmEpi& ep, int M, int N,
                   int K, int splits, cudaStream_t s) {
  const int kb_total = K / kBK;
  const int kbps = (kb_total + splits - 1) / splits;
  dim3 grid((M + kBM - 1) / kBM, N / BN, splits);
  FilmTiles none{};
  none.y0 = N / BN;
  return launch_pdl(tc_gemm_kernel<BN, MODE>, grid, dim3(kThreads), GemmCfg<BN>::kSmemBytes, s,
                    *a, *b, ep, M, N, kb_total, kbps, none);
}

template <int BN, int MODE>
cudaError_t launch_film(const CUtensorMap* a, const CUtensorMap* b, const GemmEpi& ep, int M,
                        int N, int K, const FilmTiles& film, cudaStream_t s) {
  const int m_tiles = (M + kBM - 1) / kBM;
  FilmTiles f = film;
  f.y0 = N / BN;
  const int extra_y = film.tiles > 0 ? (film.tiles + m_tiles - 1) / m_tiles : 0;
  dim3 grid(m_tiles, N / BN + extra_y, 1);
  return launch_pdl(tc_gemm_kernel<BN, MODE>, grid, dim3(kThreads), GemmCfg<BN>::kSmemBytes, s,
                    *a, *b, ep, M, N, K / kBK, K / kBK, f);
}

bool film_ok(const FilmTiles& film, int K) {
  if (film.tiles == 0) return true;
  return film.tiles > 0 && K % kBK == 0 && K / kBK <= kFilmMaxKb &&
         film.rows >= 1 && film.rows <= kStreamRows && film.tile0 >= 0 &&
         film.ldo % kFilmTile == 0 && (film.tile0 + film.tiles) * kFilmTile <= film.ldo;
}

}  // namespace

cudaError_t tc_gemm_init() {
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(tc_gemm_stream_kernel<kBnFilm, GEMM_BIAS_F32>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                GemmStreamCfg<kBnFilm>::kSmemBytes)) != cudaSuccess)
    return e;
  if ((e = set_attr<kBnTime, GEMM_BIAS_SILU_BF16>()) != cudaSuccess) return e;
  if ((e = set_attr<kBnFilm, GEMM_BIAS_F32>()) != cudaSuccess) return e;
  if ((e = set_attr<kBnQKV, GEMM_QKV_ROPE>()) != cudaSuccess) return e;
  if ((e = set_attr<kBnResid, GEMM_PARTIAL_F32>()) != cudaSuccess) return e;
  if ((e = set_attr<kBnResid, GEMM_PARTIAL_BF16>()) != cudaSuccess) return e;
  if ((e = set_attr<kBnGU, GEMM_GEGLU>()) != cudaSuccess) return e;
  if ((e = set_attr<kBnSmall, GEMM_QKV_ROPE>()) != cudaSuccess) return e;
  if ((e = set_attr<kBnSmall, GEMM_GEGLU>()) != cudaSuccess) return e;
  if ((e = set_attr_persist<kBnQKV, GEMM_QKV_ROPE>()) != cudaSuccess) return e;
  if ((e = set_attr_persist<kBnGU, GEMM_GEGLU>()) != cudaSuccess) return e;
  if ((e = set_attr_persist<kBnResid, GEMM_PARTIAL_BF16>()) != cudaSuccess) return e;
  if ((e = set_attr_persist<kBnFilm, GEMM_BIAS_F32>()) != cudaSuccess) return e;
  return cudaSuccess;
}

cudaError_t launch_tc_gemm_persist(int bn, int mode, const CUtensorMap* a, const CUtensorMap* b,
                                   const GemmEpi& ep, int M, int N, int K, int grid,
                                   cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  if (N % bn != 0 || K % kBK != 0 || grid < 1) return cudaErrorInvalidValue;
  if (bn == kBnQKV && mode == GEMM_QKV_ROPE)
    return launch_persist<kBnQKV, GEMM_QKV_ROPE>(a, b, ep, M, N, K, grid, s);
  if (bn == kBnGU && mode == GEMM_GEGLU)
    return launch_persist<kBnGU, GEMM_GEGLU>(a, b, ep, M, N, K, grid, s);
  if (bn == kBnResid && mode == GEMM_PARTIAL_BF16)
    return launch_persist<kBnResid, GEMM_PARTIAL_BF16>(a, b, ep, M, N, K, grid, s);
  if (bn == kBnFilm && mode == GEMM_BIAS_F32)
    return launch_persist<kBnFilm, GEMM_BIAS_F32>(a, b, ep, M, N, K, grid, s);
  return cudaErrorInvalidValue;
}

cudaError_t launch_tc_gemm_film(int bn, int mode, const CUtensorMap* a, const CUtensorMap* b,
                                const GemmEpi& ep, int M, int N, int K, const FilmTiles& film,
                                cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  if (N % bn != 0 || K % kBK != 0 || !film_ok(film, K)) return cudaErrorInvalidValue;
  if (bn == kBnQKV && mode == GEMM_QKV_ROPE)
    return launch_film<kBnQKV, GEMM_QKV_ROPE>(a, b, ep, M, N, K, film, s);
  if (bn == kBnSmall && mode == GEMM_QKV_ROPE)
    return launch_film<kBnSmall, GEMM_QKV_ROPE>(a, b, ep, M, N, K, film, s);
  if (bn == kBnGU && mode == GEMM_GEGLU)
    return launch_film<kBnGU, GEMM_GEGLU>(a, b, ep, M, N, K, film, s);
  if (bn == kBnSmall && mode == GEMM_GEGLU)
    return launch_film<kBnSmall, GEMM_GEGLU>(a, b, ep, M, N, K, film, s);
  return cudaErrorInvalidValue;
}

cudaError_t launch_tc_film_tiles(const FilmTiles& film, int K, int* err, cudaStream_t s) {
  if (film.tiles <= 0) return cudaSuccess;
  if (!film_ok(film, K)) return cudaErrorInvalidValue;
  FilmTiles f = film;
  f.y0 = 0;  // every CTA is a FiLM tile
  GemmEpi ep{};
  ep.err = err;
  return launch_pdl(tc_gemm_kernel<kBnSmall, GEMM_QKV_ROPE>, dim3(1, film.tiles, 1),
                    dim3(kThreads), GemmCfg<kBnSmall>::kSmemBytes, s, f.a, f.b, ep, 0, 0, K / kBK,
                    K / kBK, f);
}

cudaError_t launch_tc_gemm(int bn, int mode, const CUtensorMap* a, const CUtensorMap* b,
                           const GemmEpi& ep, int M, int N, int K, int splits,
                           cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  if (bn == kBnTime && mode == GEMM_BIAS_SILU_BF16)
    return launch<kBnTime, GEMM_BIAS_SILU_BF16>(a, b, ep, M, N, K, splits, s);
  if (bn == kBnFilm && mode == GEMM_BIAS_F32)
    return launch<kBnFilm, GEMM_BIAS_F32>(a, b, ep, M, N, K, splits, s);
  if (bn == kBnQKV && mode == GEMM_QKV_ROPE)
    return launch<kBnQKV, GEMM_QKV_ROPE>(a, b, ep, M, N, K, splits, s);
  if (bn == kBnResid && mode == GEMM_PARTIAL_F32)
    return launch<kBnResid, GEMM_PARTIAL_F32>(a, b, ep, M, N, K, splits, s);
  if (bn == kBnResid && mode == GEMM_PARTIAL_BF16)
    return launch<kBnResid, GEMM_PARTIAL_BF16>(a, b, ep, M, N, K, splits, s);
  if (bn == kBnGU && mode == GEMM_GEGLU)
    return launch<kBnGU, GEMM_GEGLU>(a, b, ep, M, N, K, splits, s);
  if (bn == kBnSmall && mode == GEMM_QKV_ROPE)
    return launch<kBnSmall, GEMM_QKV_ROPE>(a, b, ep, M, N, K, splits, s);
  if (bn == kBnSmall && mode == GEMM_GEGLU)
    return launch<kBnSmall, GEMM_GEGLU>(a, b, ep, M, N, K, splits, s);
  return cudaErrorInvalidValue;
}

}  // namespace fva

namespace fva {

cudaError_t launch_tc_gemm_stream(const CUtensorMap* a, const CUtensorMap* b, const GemmEpi& ep,
                                  int M, int N, int K, int grid, cudaStream_t s) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  if (M > kStreamRows || N % kBnFilm != 0 || K % kBK != 0) return cudaErrorInvalidValue;
  const int n_tiles = N / kBnFilm;
  return launch_pdl(tc_gemm_stream_kernel<kBnFilm, GEMM_BIAS_F32>, dim3(std::min(grid, n_tiles)),
                    dim3(kThreads), GemmStreamCfg<kBnFilm>::kSmemBytes, s, *a, *b, ep, M, n_tiles,
                    K / kBK);
}

}  // namespace fva
