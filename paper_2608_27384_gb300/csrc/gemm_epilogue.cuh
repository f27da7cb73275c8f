// Epilogues of the tcgen05 GEMMs: one output row per thread, read from TMEM in
// 32-column chunks.  bf16 rows are stored straight from registers; fp32 rows go
// through a per-warp shared-memory stage for coalesced 16-byte stores.  Shared by
// the per-op GEMM kernel and the fused block kernel.
#pragma once

#include <cuda_fp16.h>
#include "common.cuh"
#include "kernels.h"

namespace fva {

// 32 bytes (one L2 sector) in one 256-bit store; dst 32-byte aligned.
__device__ __forceinline__ void st_global_v8(void* dst, const uint4& a, const uint4& b) {
  asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(dst), "r"(a.x),
               "r"(a.y), "r"(a.z), "r"(a.w), "r"(b.x), "r"(b.y), "r"(b.z), "r"(b.w)
               : "memory");
}

// 64 bytes of one output row, straight from registers as two 256-bit stores (each a
// whole L2 sector; the 32 lanes of a warp write 32 different rows); dst 32-byte
// aligned (every caller's row pieces start on 64-byte boundaries).  No shared-memory
// staging, whose write and read-back would compete with the MMAs' operand traffic
// for the SM's shared-memory bandwidth.
__device__ __forceinline__ void store_row64(const uint4 (&u)[4], void* dst) {
  if (dst) {
    st_global_v8(dst, u[0], u[1]);
    st_global_v8(reinterpret_cast<uint8_t*>(dst) + 32, u[2], u[3]);
  }
}

__device__ __forceinline__ void pack_f32x32(const float (&v)[32], uint4 (&u)[8]) {
#pragma unroll
  for (int i = 0; i < 8; ++i)
    u[i] = make_uint4(__float_as_uint(v[4 * i]), __float_as_uint(v[4 * i + 1]),
                      __float_as_uint(v[4 * i + 2]), __float_as_uint(v[4 * i + 3]));
}

__device__ __forceinline__ void pack_bf16x32(const float (&v)[32], uint4 (&u)[4]) {
#pragma unroll
  for (int i = 0; i < 4; ++i) u[i] = pack_bf16x8(&v[8 * i]);
}

// This row's fp16 RoPE (cos, sin) pairs for tile column n0 (BN/2 pairs, 2*BN
// bytes), loaded into registers while the MMAs still run; zeros where the row
// is past M or the tile is not rotated (v).
template <int BN>
__device__ __forceinline__ void gemm_epilogue_load_rope(const GemmEpi& ep, int m, int M, int n0,
                                                        uint4 (&rh)[BN / 8]) {
  const int dh = ep.dh, seg = n0 / dh, tj = (n0 % dh) / BN;
  const bool need = m < M && seg <= ep.nq;
  int pos = 0;
  if (need) {
    const int r = m / ep.T;
    pos = __ldg(ep.prefix_len + r) + (m - r * ep.T);
  }
  const uint4* src = reinterpret_cast<const uint4*>(ep.rope_h + (size_t)pos * (dh / 2) + tj * (BN / 2));
#pragma unroll
  for (int i = 0; i < BN / 8; ++i) rh[i] = need ? __ldg(src + i) : make_uint4(0u, 0u, 0u, 0u);
}

// The QKV epilogue (GEMM_QKV_ROPE) with the row's RoPE pairs already in
// registers (gemm_epilogue_load_rope).  Weight rows are permuted so that tile
// column c < BN/2 holds head dim d = tj*BN/2 + c of segment `seg` and column
// c + BN/2 holds its rotate-half partner d + dh/2.  Segments: q heads 0..nq-1,
// then k, then v.
template <int BN>
__device__ __forceinline__ void gemm_epilogue_qkv(const GemmEpi& ep, uint32_t trow, int m, int M,
                                                  int n0, uint8_t* stage, int lane,
                                                  const uint4 (&rh)[BN / 8]) {
  constexpr int half = BN / 2;
  const bool ok = m < M;
  const int dh = ep.dh, seg = n0 / dh, tj = (n0 % dh) / BN;
  int r = 0, t = 0, pos = 0;
  if (ok) {
    r = m / ep.T;
    t = m - r * ep.T;
    pos = __ldg(ep.prefix_len + r) + t;
  }
  bf16* dst;
  if (seg < ep.nq)
    dst = (bf16*)ep.q + (size_t)m * ep.nq * dh + seg * dh;
  else
    dst = (bf16*)(seg == ep.nq ? ep.kc : ep.vc) + ((size_t)r * ep.S_cap + pos) * dh;
  const bool rotate = seg <= ep.nq;
  const __half2* hp = reinterpret_cast<const __half2*>(rh);
#pragma unroll
  for (int c = 0; c < half; c += 32) {
    float x1[32], x2[32];
    tmem_ld32(trow + c, x1);
    tmem_ld32(trow + half + c, x2);
    if (rotate) {
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const float2 cs = __half22float2(hp[c + i]);
        const float a0 = x1[i], b0 = x2[i];
        x1[i] = a0 * cs.x - b0 * cs.y;
        x2[i] = b0 * cs.x + a0 * cs.y;
      }
    }
    const int d0 = tj * half + c;
    uint4 p1[4], p2[4];
    pack_bf16x32(x1, p1);
    pack_bf16x32(x2, p2);
    store_row64(p1, ok ? dst + d0 : nullptr);
    store_row64(p2, ok ? dst + d0 + dh / 2 : nullptr);
  }
}

// Epilogue of one output row per thread; `stage` is this warp's private shared
// memory (32 * 144 bytes): every 32-column fp32 chunk is stored through it with
// coalesced 16-byte stores (warp_store_rows); bf16 chunks are stored directly.
template <int BN, int MODE>
__device__ __forceinline__ void gemm_epilogue(const GemmEpi& ep, uint32_t trow, int m, int M,
                                              int n0, int split, uint8_t* stage, int lane) {
  const bool ok = m < M;
  if constexpr (MODE == GEMM_PARTIAL_BF16) {
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
      float v[32];
      tmem_ld32(trow + c, v);
      uint4 u[4];
      pack_bf16x32(v, u);
      bf16* dst = ok ? (bf16*)ep.out + split * ep.split_stride + (size_t)m * ep.ldo + n0 + c
                     : nullptr;
      store_row64(u, dst);
    }
  } else if constexpr (MODE == GEMM_BIAS_F32 || MODE == GEMM_BIAS_SILU_BF16 ||
                       MODE == GEMM_PARTIAL_F32) {
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
      float v[32];
      tmem_ld32(trow + c, v);
      if constexpr (MODE == GEMM_PARTIAL_F32) {
        uint4 u[8];
        pack_f32x32(v, u);
        float* dst = ok ? (float*)ep.out + split * ep.split_stride + (size_t)m * ep.ldo + n0 + c
                        : nullptr;
        warp_store_rows<128>(stage, u, dst, lane);
      } else {
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          v[i] += __ldg(ep.bias + n0 + c + i);
          if constexpr (MODE == GEMM_BIAS_SILU_BF16) v[i] = silu_f(v[i]);
        }
        if constexpr (MODE == GEMM_BIAS_F32) {
          uint4 u[8];
          pack_f32x32(v, u);
          warp_store_rows<128>(stage, u, ok ? (float*)ep.out + (size_t)m * ep.ldo + n0 + c : nullptr,
                               lane);
        } else {
          uint4 u[4];
          pack_bf16x32(v, u);
          store_row64(u, ok ? (bf16*)ep.out + (size_t)m * ep.ldo + n0 + c : nullptr);
        }
      }
    }
  } else if constexpr (MODE == GEMM_GEGLU) {
    // Tile columns [0, BN/2) hold gate rows n0/2 + c, [BN/2, BN) the matching up rows.
    constexpr int half = BN / 2;
#pragma unroll 1
    for (int c = 0; c < half; c += 32) {
      float g[32], u[32];
      tmem_ld32(trow + c, g);
      tmem_ld32(trow + half + c, u);
#pragma unroll
      for (int i = 0; i < 32; ++i) g[i] = gelu_tanh_bf16out(g[i]) * u[i];
      uint4 pk[4];
      pack_bf16x32(g, pk);
      store_row64(pk, ok ? (bf16*)ep.out + (size_t)m * ep.ldo + n0 / 2 + c : nullptr);
    }
  } else if constexpr (MODE == GEMM_QKV_ROPE) {
    // Weight rows are permuted so that tile column c < BN/2 holds head dim
    // d = tj*BN/2 + c of segment `seg` and column c + BN/2 holds its rotate-half
    // partner d + dh/2.  Segments: q heads 0..nq-1, then k, then v.
    constexpr int half = BN / 2;
    const int dh = ep.dh, seg = n0 / dh, tj = (n0 % dh) / BN;
    int r = 0, t = 0, pos = 0;
    if (ok) {
      r = m / ep.T;
      t = m - r * ep.T;
      pos = __ldg(ep.prefix_len + r) + t;
    }
    bf16* dst;
    if (seg < ep.nq)
      dst = (bf16*)ep.q + (size_t)m * ep.nq * dh + seg * dh;
    else
      dst = (bf16*)(seg == ep.nq ? ep.kc : ep.vc) + ((size_t)r * ep.S_cap + pos) * dh;
    const bool rotate = seg <= ep.nq;
    const float4* cs4 = reinterpret_cast<const float4*>(ep.rope + (size_t)pos * (dh / 2) +
                                                        tj * half);  // (cos, sin) pairs
#pragma unroll 1
    for (int c = 0; c < half; c += 32) {
      float4 cs[16];
      if (ok && rotate) {
#pragma unroll
        for (int i = 0; i < 16; ++i) cs[i] = __ldg(cs4 + c / 2 + i);
      }
      float x1[32], x2[32];
      tmem_ld32(trow + c, x1);
      tmem_ld32(trow + half + c, x2);
      const int d0 = tj * half + c;
      if (ok && rotate) {
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
          const float a0 = x1[i], b0 = x2[i], a1 = x1[i + 1], b1 = x2[i + 1];
          x1[i] = a0 * cs[i / 2].x - b0 * cs[i / 2].y;
          x2[i] = b0 * cs[i / 2].x + a0 * cs[i / 2].y;
          x1[i + 1] = a1 * cs[i / 2].z - b1 * cs[i / 2].w;
          x2[i + 1] = b1 * cs[i / 2].z + a1 * cs[i / 2].w;
        }
      }
      uint4 p1[4], p2[4];
      pack_bf16x32(x1, p1);
      pack_bf16x32(x2, p2);
      store_row64(p1, ok ? dst + d0 : nullptr);
      store_row64(p2, ok ? dst + d0 + dh / 2 : nullptr);
    }
  }
}

}  // namespace fva
