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
// planes (fp32), RoPE + q / KV-workspace scatter for the packed QKV projection,
// and tanh-GELU(gate) * up for the packed gate/up projection.
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

template <int BN>
struct GemmCfg {
  static constexpr int kABytes = kBM * kBK * 2;
  static constexpr int kBBytes = BN * kBK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kStages = (BN <= 64) ? 8 : (BN <= 128 ? 6 : 4);
  static constexpr int kTmemCols = BN < 32 ? 32 : BN;
  static constexpr int kSmemBytes = kStages * kStageBytes + 1024 /*align*/ + 256 /*barriers*/;
};

template <int BN, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const GemmEpi ep, int M, int N, int kb_total, int kb_per_split) {
  using C = GemmCfg<BN>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint64_t* full = (uint64_t*)(smem + C::kStages * C::kStageBytes);
  uint64_t* empty = full + C::kStages;
  uint64_t* acc_full = empty + C::kStages;
  uint32_t* tmem_slot = (uint32_t*)(acc_full + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m0 = blockIdx.x * kBM, n0 = blockIdx.y * BN, split = blockIdx.z;
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
    const int pre = min(nkb, C::kStages);
    for (int i = 0; i < pre; ++i) {
      mbar_arrive_expect_tx(&full[i], C::kStageBytes);
      tma_load_2d(smem + i * C::kStageBytes + C::kABytes, &tmB, (kb0 + i) * kBK, n0, &full[i]);
    }
    pdl_wait();
    for (int i = 0; i < pre; ++i)
      tma_load_2d(smem + i * C::kStageBytes, &tmA, (kb0 + i) * kBK, m0, &full[i]);
    for (int i = pre; i < nkb; ++i) {
      const int s = i % C::kStages;
      const uint32_t ph = (uint32_t)(i / C::kStages) & 1u;
      if (!mbar_wait(&empty[s], ph ^ 1u, ep.err, KERR_WAIT_MMA)) break;
      uint8_t* sa = smem + s * C::kStageBytes;
      mbar_arrive_expect_tx(&full[s], C::kStageBytes);
      tma_load_2d(sa, &tmA, (kb0 + i) * kBK, m0, &full[s]);
      tma_load_2d(sa + C::kABytes, &tmB, (kb0 + i) * kBK, n0, &full[s]);
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer
    constexpr uint32_t idesc = umma_idesc_bf16(kBM, BN, false);
    bool good = true;
    for (int i = 0; i < nkb; ++i) {
      const int s = i % C::kStages;
      const uint32_t ph = (uint32_t)(i / C::kStages) & 1u;
      if (!mbar_wait(&full[s], ph, ep.err, KERR_WAIT_TMA)) {
        good = false;
        break;
      }
      tc_fence_after();
      const uint32_t sa = smem_u32(smem + s * C::kStageBytes);
      const uint32_t sb = sa + C::kABytes;
#pragma unroll
      for (int kk = 0; kk < kBK / 16; ++kk) {
        const uint64_t ad = umma_desc_sw128(sa + kk * 32, 16, 1024);
        const uint64_t bd = umma_desc_sw128(sb + kk * 32, 16, 1024);
        umma_bf16(tmem, ad, bd, idesc, (i > 0 || kk > 0) ? 1u : 0u);
      }
      umma_commit(&empty[s]);
    }
    if (good) umma_commit(acc_full);
  } else if (warp >= 2) {
    // ---------------- epilogue: warp w reads TMEM lanes 32*(w%4) .. +31
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    const bool good = __all_sync(0xffffffffu, mbar_wait(acc_full, 0, ep.err, KERR_WAIT_MMA));
    tc_fence_after();
    if (good && nkb > 0) {
      // all MMAs (and so all TMA loads into the ring) are complete: the ring's
      // first stage is free to stage this warp's coalesced stores
      const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
      uint8_t* stage = smem + (warp - 2) * (32 * 144);
      gemm_epilogue<BN, MODE>(ep, trow, m0 + row, M, n0, split, stage, lane);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
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
  return launch_pdl(tc_gemm_kernel<BN, MODE>, grid, dim3(kThreads), GemmCfg<BN>::kSmemBytes, s,
                    *a, *b, ep, M, N, kb_total, kbps);
}

}  // namespace

cudaError_t tc_gemm_init() {
  cudaError_t e;
  if ((e = set_attr<kBnTime, GEMM_BIAS_SILU_BF16>()) != cudaSuccess) return e;
  if ((e = set_attr<kBnFilm, GEMM_BIAS_F32>()) != cudaSuccess) return e;
  if ((e = set_attr<kBnQKV, GEMM_QKV_ROPE>()) != cudaSuccess) return e;
  if ((e = set_attr<kBnResid, GEMM_PARTIAL_F32>()) != cudaSuccess) return e;
  if ((e = set_attr<kBnGU, GEMM_GEGLU>()) != cudaSuccess) return e;
  return cudaSuccess;
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
  if (bn == kBnGU && mode == GEMM_GEGLU)
    return launch<kBnGU, GEMM_GEGLU>(a, b, ep, M, N, K, splits, s);
  return cudaErrorInvalidValue;
}

}  // namespace fva
