// Row-wise kernels of the streaming step: timestep embedding, the fused action
// in-projection + first FiLM RMSNorm, the fused split-K reduction + gated
// residual + FiLM RMSNorm, and the fused final norm + out-projection + Euler
// update + emit + buffer roll + tail noise.  Plus small table / debug helpers.
#include <cuda_fp16.h>

#include <algorithm>
#include "common.cuh"
#include "kernels.h"

namespace fva {

// ----------------------------------------------------------------------------
// sinusoidal timestep embedding of every chunk's noise level (App. A.4 FiLM
// condition input): e = [sin(2 pi tau / p_j) | cos(2 pi tau / p_j)],
// p_j = t_min (t_max / t_min)^(j / (W/2 - 1)).
// The argument in half turns, x = tau * (2 / p_j), is formed from a two-float
// split c_hi + c_lo of 2 / p_j (computed in double on the host): the product
// tau * c_hi is split exactly with an fma, its integer part is removed exactly,
// and sincospi of the small remainder gives sin / cos to fp32 accuracy.
// ----------------------------------------------------------------------------
// (sin, cos) of tau * (2 / p_j) half turns, with c = (hi, lo) split of 2 / p_j.
__device__ __forceinline__ float2 temb_sincos(float t, float2 c) {
  const float p = t * c.x;
  const float p_err = fmaf(t, c.x, -p);      // exact remainder of the product
  const float n = rintf(p);                  // |p| < 2^23: exact
  const float r = (p - n) + fmaf(t, c.y, p_err);
  float sn, cs;
  sincospif(r, &sn, &cs);
  const int odd = ((int)n) & 1;              // sin / cos of (n + r) pi
  if (odd) {
    sn = -sn;
    cs = -cs;
  }
  return make_float2(sn, cs);
}

template <typename Act>
__global__ void temb_kernel(const float* __restrict__ tau, const float2* __restrict__ freq,
                            int W, Act* __restrict__ out) {
  const int row = blockIdx.y;
  const int half = W / 2;
  pdl_trigger();
  pdl_wait();
  const float t = tau[row];
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= half) return;
  const float2 sc = temb_sincos(t, freq[j]);
  out[(size_t)row * W + j] = from_float<Act>(sc.x);
  out[(size_t)row * W + half + j] = from_float<Act>(sc.y);
}

void launch_temb(const float* tau, const float2* freq, int rows, int W, void* out,
                 bool act_bf16, cudaStream_t s) {
  if (rows <= 0) return;
  dim3 grid((W / 2 + 127) / 128, rows);
  if (act_bf16)
    launch_pdl(temb_kernel<bf16>, grid, dim3(128), 0, s, tau, freq, W, (bf16*)out);
  else
    launch_pdl(temb_kernel<float>, grid, dim3(128), 0, s, tau, freq, W, (float*)out);
}

// ----------------------------------------------------------------------------
// row helpers (W a multiple of 4)
// ----------------------------------------------------------------------------
template <typename Act>
__device__ __forceinline__ void store4(Act* dst, float a, float b, float c, float d);
template <>
__device__ __forceinline__ void store4<float>(float* dst, float a, float b, float c, float d) {
  *reinterpret_cast<float4*>(dst) = make_float4(a, b, c, d);
}
template <>
__device__ __forceinline__ void store4<bf16>(bf16* dst, float a, float b, float c, float d) {
  __nv_bfloat162 lo = __floats2bfloat162_rn(a, b), hi = __floats2bfloat162_rn(c, d);
  uint2 u;
  u.x = *reinterpret_cast<uint32_t*>(&lo);
  u.y = *reinterpret_cast<uint32_t*>(&hi);
  *reinterpret_cast<uint2*>(dst) = u;
}

// Sum over the CTA (blockDim.x a multiple of 32, at most 1024); every thread gets it.
__device__ __forceinline__ float block_sum(float v, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  v = warp_sum(v);
  __syncthreads();  // red may still be read by a previous call
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float t = 0.f;
  for (int w = 0; w < nw; ++w) t += red[w];
  return t;
}

// y = h * rsqrt(mean(h^2) + eps) * (1 + scale) + shift for a row already in h
// (each thread re-reads the columns it wrote itself).
template <typename Act>
__device__ __forceinline__ void modulated_norm_row(const float* __restrict__ hrow, float ss, int W,
                                                   float eps, const float* __restrict__ scale,
                                                   const float* __restrict__ shift,
                                                   Act* __restrict__ yrow) {
  const float r = rsqrtf(ss / (float)W + eps);
  for (int c = threadIdx.x * 4; c < W; c += blockDim.x * 4) {
    const float4 hv = *reinterpret_cast<const float4*>(hrow + c);
    const float4 sc = *reinterpret_cast<const float4*>(scale + c);
    const float4 sh = *reinterpret_cast<const float4*>(shift + c);
    store4<Act>(yrow + c, hv.x * r * (1.f + sc.x) + sh.x, hv.y * r * (1.f + sc.y) + sh.y,
                hv.z * r * (1.f + sc.z) + sh.z, hv.w * r * (1.f + sc.w) + sh.w);
  }
}

inline int row_threads(int W) {
  int t = W / 4;
  t = t < 32 ? 32 : (t > 1024 ? 1024 : t);
  return (t + 31) & ~31;
}

// ----------------------------------------------------------------------------
// action in-projection h = x W_in^T + b_in, then layer 0's FiLM RMSNorm.
// R token rows per CTA, so each CTA reads w_in_t (W_in transposed, [A, W] fp32)
// once for all of them; each thread owns 4 columns of every row.
// ----------------------------------------------------------------------------
constexpr int kEmbedMaxA = 32;  // action dims held in registers by the fast path

template <typename Act, int R>
__global__ void __launch_bounds__(256) embed_norm_kernel(StepDims d, int rows, const float* __restrict__ buffer,
                                  const float* __restrict__ w_in_t,
                                  const float* __restrict__ b_in, const float* __restrict__ mod,
                                  float* __restrict__ h, Act* __restrict__ y) {
  __shared__ float xs[R][128];
  __shared__ float red[32];
  const int m0 = blockIdx.x * R;
  const int nr = min(R, rows - m0);
  if (d.W == 4 * (int)blockDim.x && d.A <= kEmbedMaxA) {
    // one float4 column group per thread: W_in (static) is in registers before the
    // wait for the predecessor; after it one round of loads (this CTA's buffer rows
    // and their FiLM scale / shift), one CTA-wide reduction for all R rows
    __shared__ float red_r[R][32];
    const int col = threadIdx.x * 4;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    float4 wreg[kEmbedMaxA];
#pragma unroll
    for (int a = 0; a < kEmbedMaxA; ++a)
      if (a < d.A) wreg[a] = *reinterpret_cast<const float4*>(w_in_t + (size_t)a * d.W + col);
    const float4 bias = *reinterpret_cast<const float4*>(b_in + col);
    // the buffer rows were written by the previous step's roll, earlier on the
    // stream, and by nothing in this step before this kernel: read before the wait
    // too (from device memory, or from pinned host memory over the host link)
    for (int i = threadIdx.x; i < R * d.A; i += blockDim.x) {
      const int r = i / d.A, a = i % d.A;
      xs[r][a] = r < nr ? buffer[(size_t)(m0 + r) * d.A + a] : 0.f;
    }
    pdl_trigger();
    pdl_wait();
    float4 sc[R], sh[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int m = min(m0 + r, rows - 1);
      const int rq = m / d.T, c = (m % d.T) / d.H;
      const float* mrow = mod + (size_t)(rq * d.K + c) * d.N_mod;
      sc[r] = *reinterpret_cast<const float4*>(mrow + mod_off(0, 0, d.W) + col);
      sh[r] = *reinterpret_cast<const float4*>(mrow + mod_off(0, 1, d.W) + col);
    }
    __syncthreads();
    float4 acc[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      acc[r] = bias;
#pragma unroll
      for (int a = 0; a < kEmbedMaxA; ++a) {
        if (a >= d.A) break;
        const float xa = xs[r][a];
        acc[r].x = fmaf(xa, wreg[a].x, acc[r].x);
        acc[r].y = fmaf(xa, wreg[a].y, acc[r].y);
        acc[r].z = fmaf(xa, wreg[a].z, acc[r].z);
        acc[r].w = fmaf(xa, wreg[a].w, acc[r].w);
      }
      if (r < nr) *reinterpret_cast<float4*>(h + (size_t)(m0 + r) * d.W + col) = acc[r];
      const float ss = warp_sum(acc[r].x * acc[r].x + acc[r].y * acc[r].y +
                                acc[r].z * acc[r].z + acc[r].w * acc[r].w);
      if (lane == 0) red_r[r][warp] = ss;
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < R; ++r) {
      if (r >= nr) break;
      float tot = 0.f;
      for (int w = 0; w < nw; ++w) tot += red_r[r][w];
      const float rn = rsqrtf(tot / (float)d.W + d.eps);
      store4<Act>(y + (size_t)(m0 + r) * d.W + col, acc[r].x * rn * (1.f + sc[r].x) + sh[r].x,
                  acc[r].y * rn * (1.f + sc[r].y) + sh[r].y,
                  acc[r].z * rn * (1.f + sc[r].z) + sh[r].z,
                  acc[r].w * rn * (1.f + sc[r].w) + sh[r].w);
    }
    return;
  }
  // buffer [B, K, H, A] = rows of A, token rows m0 .. m0 + nr - 1 contiguous (read
  // before the wait, as above)
  for (int i = threadIdx.x; i < R * d.A; i += blockDim.x) {
    const int r = i / d.A, a = i % d.A;
    xs[r][a] = r < nr ? buffer[(size_t)(m0 + r) * d.A + a] : 0.f;
  }
  pdl_trigger();
  pdl_wait();
  __syncthreads();
  float ss[R];
#pragma unroll
  for (int r = 0; r < R; ++r) ss[r] = 0.f;
  for (int col = threadIdx.x * 4; col < d.W; col += blockDim.x * 4) {
    float4 acc[R];
    const float4 bias = *reinterpret_cast<const float4*>(b_in + col);
#pragma unroll
    for (int r = 0; r < R; ++r) acc[r] = bias;
    // 16 weight loads in flight per thread before the FMAs (one CTA per SM has to
    // cover the L2 latency on its own)
    for (int a0 = 0; a0 < d.A; a0 += 16) {
      float4 w[16];
#pragma unroll
      for (int j = 0; j < 16; ++j)
        if (a0 + j < d.A) w[j] = *reinterpret_cast<const float4*>(w_in_t + (size_t)(a0 + j) * d.W + col);
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        if (a0 + j >= d.A) break;
#pragma unroll
        for (int r = 0; r < R; ++r) {
          const float xa = xs[r][a0 + j];
          acc[r].x = fmaf(xa, w[j].x, acc[r].x);
          acc[r].y = fmaf(xa, w[j].y, acc[r].y);
          acc[r].z = fmaf(xa, w[j].z, acc[r].z);
          acc[r].w = fmaf(xa, w[j].w, acc[r].w);
        }
      }
    }
#pragma unroll
    for (int r = 0; r < R; ++r)
      if (r < nr) {
        *reinterpret_cast<float4*>(h + (size_t)(m0 + r) * d.W + col) = acc[r];
        ss[r] += acc[r].x * acc[r].x + acc[r].y * acc[r].y + acc[r].z * acc[r].z +
                 acc[r].w * acc[r].w;
      }
  }
#pragma unroll
  for (int r = 0; r < R; ++r) {
    if (r >= nr) break;  // uniform over the CTA
    const int m = m0 + r;
    const int rq = m / d.T, c = (m % d.T) / d.H;
    const float tot = block_sum(ss[r], red);
    const float* mrow = mod + (size_t)(rq * d.K + c) * d.N_mod;
    modulated_norm_row<Act>(h + (size_t)m * d.W, tot, d.W, d.eps, mrow + mod_off(0, 0, d.W),
                            mrow + mod_off(0, 1, d.W), y + (size_t)m * d.W);
  }
}

template <typename Act, int R>
static void launch_embed_norm_r(const StepDims& d, int rows, const float* buffer,
                                const float* w_in_t, const float* b_in, const float* mod,
                                float* h, Act* y, cudaStream_t s) {
  // at most 256 threads (the register budget of the fast path); wider rows loop
  launch_pdl(embed_norm_kernel<Act, R>, dim3((rows + R - 1) / R),
             dim3(std::min(row_threads(d.W), 256)), 0, s, d, rows, buffer, w_in_t, b_in, mod, h, y);
}

template <typename Act>
static void launch_embed_norm_t(const StepDims& d, int rows, int n_sms, const float* buffer,
                                const float* w_in_t, const float* b_in, const float* mod,
                                float* h, Act* y, cudaStream_t s) {
  // rows per CTA: about one CTA per SM, so w_in_t is read about once per SM
  const int per_sm = (rows + n_sms - 1) / n_sms;
  if (per_sm >= 8)
    launch_embed_norm_r<Act, 8>(d, rows, buffer, w_in_t, b_in, mod, h, y, s);
  else if (per_sm >= 4)
    launch_embed_norm_r<Act, 4>(d, rows, buffer, w_in_t, b_in, mod, h, y, s);
  else if (per_sm >= 2)
    launch_embed_norm_r<Act, 2>(d, rows, buffer, w_in_t, b_in, mod, h, y, s);
  else
    launch_embed_norm_r<Act, 1>(d, rows, buffer, w_in_t, b_in, mod, h, y, s);
}

void launch_embed_norm(const StepDims& d, const float* buffer, const float* w_in_t,
                       const float* b_in, const float* mod, float* h, void* y, bool act_bf16,
                       int n_sms, cudaStream_t s) {
  const int rows = d.B * d.T;
  if (rows <= 0) return;
  if (n_sms < 1) n_sms = 1;
  if (act_bf16)
    launch_embed_norm_t<bf16>(d, rows, n_sms, buffer, w_in_t, b_in, mod, h, (bf16*)y, s);
  else
    launch_embed_norm_t<float>(d, rows, n_sms, buffer, w_in_t, b_in, mod, h, (float*)y, s);
}

// ----------------------------------------------------------------------------
// h += gate_c * sum_z part[z]  (split-K partials reduced in fixed order z = 0..),
// then y = FiLM RMSNorm(h) with the next norm's (scale, shift).  One CTA per row.
// ----------------------------------------------------------------------------
// 4 consecutive partial-sum values as floats (fp32 or bf16 planes), L2 only.
__device__ __forceinline__ float4 load4_cg(const float* p) {
  return __ldcg(reinterpret_cast<const float4*>(p));
}
__device__ __forceinline__ float4 load4_cg(const bf16* p) {
  const uint2 u = __ldcg(reinterpret_cast<const uint2*>(p));
  return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xFFFF0000u),
                     __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xFFFF0000u));
}

template <typename Act, typename Part>
__global__ void resid_norm_kernel(StepDims d, float* __restrict__ h,
                                  const Part* __restrict__ part, int n_parts,
                                  long long part_stride, const float* __restrict__ mod,
                                  int gate_off, int scale_off, int shift_off,
                                  Act* __restrict__ y) {
  __shared__ float red[32];
  const int m = blockIdx.x;
  const int r = m / d.T, c = (m % d.T) / d.H;
  pdl_trigger();
  pdl_wait();
  const float* mrow = mod + (size_t)(r * d.K + c) * d.N_mod;
  float* hrow = h + (size_t)m * d.W;
  const int col = threadIdx.x * 4;
  if (d.W == 4 * (int)blockDim.x) {
    // one float4 per thread: every load in flight at once, values kept in registers
    float4 p[8];
#pragma unroll
    for (int z = 0; z < 8; ++z)
      if (z < n_parts)
        p[z] = load4_cg(part + z * part_stride + (size_t)m * d.W + col);
    const float4 g = *reinterpret_cast<const float4*>(mrow + gate_off + col);
    const float4 sc = *reinterpret_cast<const float4*>(mrow + scale_off + col);
    const float4 sh = *reinterpret_cast<const float4*>(mrow + shift_off + col);
    float4 hv = *reinterpret_cast<const float4*>(hrow + col);
    float4 acc = p[0];
#pragma unroll
    for (int z = 1; z < 8; ++z)
      if (z < n_parts) {
        acc.x += p[z].x; acc.y += p[z].y; acc.z += p[z].z; acc.w += p[z].w;
      }
    for (int z = 8; z < n_parts; ++z) {
      const float4 q = load4_cg(part + z * part_stride + (size_t)m * d.W + col);
      acc.x += q.x; acc.y += q.y; acc.z += q.z; acc.w += q.w;
    }
    hv.x = fmaf(g.x, acc.x, hv.x);
    hv.y = fmaf(g.y, acc.y, hv.y);
    hv.z = fmaf(g.z, acc.z, hv.z);
    hv.w = fmaf(g.w, acc.w, hv.w);
    *reinterpret_cast<float4*>(hrow + col) = hv;
    const float ss = block_sum(hv.x * hv.x + hv.y * hv.y + hv.z * hv.z + hv.w * hv.w, red);
    const float rn = rsqrtf(ss / (float)d.W + d.eps);
    store4<Act>(y + (size_t)m * d.W + col, hv.x * rn * (1.f + sc.x) + sh.x,
                hv.y * rn * (1.f + sc.y) + sh.y, hv.z * rn * (1.f + sc.z) + sh.z,
                hv.w * rn * (1.f + sc.w) + sh.w);
    return;
  }
  float ss = 0.f;
  for (int cc = col; cc < d.W; cc += blockDim.x * 4) {
    float4 acc = load4_cg(part + (size_t)m * d.W + cc);
    for (int z = 1; z < n_parts; ++z) {
      const float4 q = load4_cg(part + z * part_stride + (size_t)m * d.W + cc);
      acc.x += q.x; acc.y += q.y; acc.z += q.z; acc.w += q.w;
    }
    const float4 g = *reinterpret_cast<const float4*>(mrow + gate_off + cc);
    float4 hv = *reinterpret_cast<const float4*>(hrow + cc);
    hv.x = fmaf(g.x, acc.x, hv.x);
    hv.y = fmaf(g.y, acc.y, hv.y);
    hv.z = fmaf(g.z, acc.z, hv.z);
    hv.w = fmaf(g.w, acc.w, hv.w);
    *reinterpret_cast<float4*>(hrow + cc) = hv;
    ss += hv.x * hv.x + hv.y * hv.y + hv.z * hv.z + hv.w * hv.w;
  }
  ss = block_sum(ss, red);
  modulated_norm_row<Act>(hrow, ss, d.W, d.eps, mrow + scale_off, mrow + shift_off,
                          y + (size_t)m * d.W);
}

// The same operation for many rows: R rows per CTA (W = 4 x blockDim, at most
// two partial planes), every row's loads in flight before any reduction, one
// shared-memory exchange for the R row sums.  With one row per CTA the register
// budget keeps four rows per SM in flight, too few to cover DRAM latency when
// the activations no longer fit L2.
template <typename Act, typename Part, int R>
__global__ void __launch_bounds__(256)
    resid_norm_rows_kernel(StepDims d, int rows, float* __restrict__ h,
                           const Part* __restrict__ part, int n_parts, long long part_stride,
                           const float* __restrict__ mod, int gate_off, int scale_off,
                           int shift_off, Act* __restrict__ y) {
  __shared__ float red[R][8];
  const int m0 = blockIdx.x * R;
  const int col = threadIdx.x * 4;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  pdl_trigger();
  pdl_wait();
  float4 hv[R], acc[R], g[R], sc[R], sh[R];
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int m = min(m0 + r, rows - 1);  // rows past the end repeat the last (not stored)
    const int rq = m / d.T, c = (m % d.T) / d.H;
    const float* mrow = mod + (size_t)(rq * d.K + c) * d.N_mod;
    acc[r] = load4_cg(part + (size_t)m * d.W + col);
    if (n_parts > 1) {
      const float4 q = load4_cg(part + part_stride + (size_t)m * d.W + col);
      acc[r].x += q.x; acc[r].y += q.y; acc[r].z += q.z; acc[r].w += q.w;
    }
    hv[r] = *reinterpret_cast<const float4*>(h + (size_t)m * d.W + col);
    g[r] = *reinterpret_cast<const float4*>(mrow + gate_off + col);
    sc[r] = *reinterpret_cast<const float4*>(mrow + scale_off + col);
    sh[r] = *reinterpret_cast<const float4*>(mrow + shift_off + col);
  }
  float ss[R];
#pragma unroll
  for (int r = 0; r < R; ++r) {
    hv[r].x = fmaf(g[r].x, acc[r].x, hv[r].x);
    hv[r].y = fmaf(g[r].y, acc[r].y, hv[r].y);
    hv[r].z = fmaf(g[r].z, acc[r].z, hv[r].z);
    hv[r].w = fmaf(g[r].w, acc[r].w, hv[r].w);
    if (m0 + r < rows) *reinterpret_cast<float4*>(h + (size_t)(m0 + r) * d.W + col) = hv[r];
    ss[r] = warp_sum(hv[r].x * hv[r].x + hv[r].y * hv[r].y + hv[r].z * hv[r].z +
                     hv[r].w * hv[r].w);
    if (lane == 0) red[r][warp] = ss[r];
  }
  __syncthreads();
#pragma unroll
  for (int r = 0; r < R; ++r) {
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) t += red[r][w];
    const float rn = rsqrtf(t / (float)d.W + d.eps);
    if (m0 + r < rows)
      store4<Act>(y + (size_t)(m0 + r) * d.W + col, hv[r].x * rn * (1.f + sc[r].x) + sh[r].x,
                  hv[r].y * rn * (1.f + sc[r].y) + sh[r].y,
                  hv[r].z * rn * (1.f + sc[r].z) + sh[r].z,
                  hv[r].w * rn * (1.f + sc[r].w) + sh[r].w);
  }
}

template <typename Part>
static void launch_resid_norm_t(const StepDims& d, int rows, float* h, const Part* part,
                                int n_parts, long long part_stride, const float* mod,
                                int gate_off, int scale_off, int shift_off, void* y,
                                bool act_bf16, cudaStream_t s) {
  constexpr int R = 4;
  if (d.W == 1024 && n_parts <= 2 && d.n_sms > 0 && rows >= R * 4 * d.n_sms) {
    const dim3 grid((rows + R - 1) / R);
    if (act_bf16)
      launch_pdl(resid_norm_rows_kernel<bf16, Part, R>, grid, dim3(256), 0, s, d, rows, h, part,
                 n_parts, part_stride, mod, gate_off, scale_off, shift_off, (bf16*)y);
    else
      launch_pdl(resid_norm_rows_kernel<float, Part, R>, grid, dim3(256), 0, s, d, rows, h, part,
                 n_parts, part_stride, mod, gate_off, scale_off, shift_off, (float*)y);
    return;
  }
  if (act_bf16)
    launch_pdl(resid_norm_kernel<bf16, Part>, dim3(rows), dim3(row_threads(d.W)), 0, s, d, h,
               part, n_parts, part_stride, mod, gate_off, scale_off, shift_off, (bf16*)y);
  else
    launch_pdl(resid_norm_kernel<float, Part>, dim3(rows), dim3(row_threads(d.W)), 0, s, d, h,
               part, n_parts, part_stride, mod, gate_off, scale_off, shift_off, (float*)y);
}

void launch_resid_norm(const StepDims& d, float* h, const void* part, bool part_bf16,
                       int n_parts, long long part_stride, const float* mod, int gate_off,
                       int scale_off, int shift_off, void* y, bool act_bf16, cudaStream_t s) {
  const int rows = d.B * d.T;
  if (rows <= 0) return;
  if (part_bf16)
    launch_resid_norm_t(d, rows, h, (const bf16*)part, n_parts, part_stride, mod, gate_off,
                        scale_off, shift_off, y, act_bf16, s);
  else
    launch_resid_norm_t(d, rows, h, (const float*)part, n_parts, part_stride, mod, gate_off,
                        scale_off, shift_off, y, act_bf16, s);
}

// ----------------------------------------------------------------------------
// Philox4x32-10 (Salmon et al., SC'11) and Box-Muller for the tail chunk.
// ----------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox4x32_10(uint4 ctr, uint2 key) {
  const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u, W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;
#pragma unroll
  for (int i = 0; i < 10; ++i) {
    if (i) {
      key.x += W0;
      key.y += W1;
    }
    const uint32_t hi0 = __umulhi(M0, ctr.x), lo0 = M0 * ctr.x;
    const uint32_t hi1 = __umulhi(M1, ctr.z), lo1 = M1 * ctr.z;
    ctr = make_uint4(hi1 ^ ctr.y ^ key.x, lo1, hi0 ^ ctr.w ^ key.y, lo0);
  }
  return ctr;
}

// Element e (0-based, row-major [H, A]) of request r's tail chunk at step `step`.
__device__ __forceinline__ float tail_normal(unsigned long long seed, unsigned long long step,
                                             int r, int e) {
  const uint4 x = philox4x32_10(
      make_uint4((uint32_t)(e >> 2), (uint32_t)r, (uint32_t)step, (uint32_t)(step >> 32)),
      make_uint2((uint32_t)seed, (uint32_t)(seed >> 32)));
  const int pair = (e >> 1) & 1, which = e & 1;
  const uint32_t ba = pair ? x.z : x.x, bb = pair ? x.w : x.y;
  const float ua = (float)((ba >> 8) + 1u) * 5.9604644775390625e-8f;  // (0, 1], 2^-24 grid
  const float ub = (float)((bb >> 8) + 1u) * 5.9604644775390625e-8f;
  const float rad = sqrtf(-2.0f * logf(ua));
  float sn, cs;
  sincospif(2.0f * ub, &sn, &cs);
  return rad * (which ? sn : cs);
}

// ----------------------------------------------------------------------------
// Velocity, Euler update, emit, roll and tail.  The final FiLM RMSNorm has
// already written y_F [B*K*H, W] (fp32).  A cluster of `nsplit` CTAs per (token
// position j within a chunk, request r) owns column j of every chunk of request
// r; CTA q of the cluster takes the width range [q W/nsplit, (q+1) W/nsplit).
// Each stages its slice of the K rows of y_F and of W_out^T [W, A] in shared
// memory with all loads in flight at once and forms the partial sums
// v_q[k][a] = sum_w y_F[k][w] W_out^T[w][a] over its range; CTA 0 adds b_out[a]
// and the partials in the order q = 0, 1, ... through distributed shared memory
// and alone writes the buffer column, so the in-place roll is race-free.
// x'_k = x_k + dt_k v_k (fp32, separately rounded multiply and add), out = x'_1,
// slot k <- x'_{k+1}, tail <- z.
// ----------------------------------------------------------------------------
constexpr int kVelThreads = 512;

__global__ void __launch_bounds__(kVelThreads)
    velocity_euler_kernel(StepDims d, const float* __restrict__ yF,
                          const float* __restrict__ w_out_t, const float* __restrict__ b_out,
                          const float* __restrict__ dt, float* __restrict__ buffer,
                          float* __restrict__ out_chunk, float* __restrict__ vel_out,
                          const float* __restrict__ fresh, unsigned long long seed,
                          const unsigned long long* __restrict__ step_idx, int wchunk,
                          int nsplit) {
  extern __shared__ __align__(16) float sm[];
  __shared__ __align__(8) uint64_t bar;
  const int q = blockIdx.x, j = blockIdx.y, r = blockIdx.z;  // q: rank in the cluster
  const int wq = d.W / nsplit, wbeg = q * wq;
  const int KA = d.K * d.A;
  float* ys = sm;                    // [K][wchunk]
  float* ws = ys + d.K * wchunk;     // [wchunk][A]
  float* xs = ws + wchunk * d.A;     // [K][A] buffer values of this column
  float* vs = xs + KA;               // [K][A] velocities
  float* red = vs + KA;              // [16][K][A] partial sums of the w-range groups
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_barrier_init();
  }
  __syncthreads();
  pdl_trigger();
  // W_out^T does not depend on earlier kernels: with one chunk per CTA its slice is
  // requested before waiting for the predecessor (the y_F rows after it)
  const bool one_chunk = wchunk == wq;
  if (one_chunk && threadIdx.x == 0) {
    mbar_arrive_expect_tx(&bar, (uint32_t)(sizeof(float) * (d.K + d.A) * wchunk));
    bulk_load(ws, w_out_t + (size_t)wbeg * d.A, (uint32_t)(sizeof(float) * wchunk * d.A), &bar);
  }
  // this column of the buffer: written by the previous step's roll (earlier on the
  // stream) and only read by this step's kernels before this one writes it, so it is
  // read before the wait too
  const size_t slot = (size_t)d.H * d.A;
  const float* xcol = buffer + ((size_t)r * d.K * d.H + j) * d.A;  // + k*slot selects chunk k
  for (int i = threadIdx.x; i < KA; i += blockDim.x) {
    if (q == 0) xs[i] = xcol[(i / d.A) * slot + i % d.A];
    vs[i] = 0.f;
  }
  pdl_wait();
  uint32_t phase = 0;
  for (int w0 = wbeg; w0 < wbeg + wq; w0 += wchunk) {
    __syncthreads();  // previous chunk consumed
    if (threadIdx.x == 0) {
      // all staging as bulk copies in flight at once: K rows of y_F and the W_out^T slice
      if (!one_chunk)
        mbar_arrive_expect_tx(&bar, (uint32_t)(sizeof(float) * (d.K + d.A) * wchunk));
      for (int k = 0; k < d.K; ++k) {
        const size_t m = (size_t)r * d.T + (size_t)k * d.H + j;
        bulk_load(ys + k * wchunk, yF + m * d.W + w0, sizeof(float) * wchunk, &bar);
      }
      if (!one_chunk)
        bulk_load(ws, w_out_t + (size_t)w0 * d.A, (uint32_t)(sizeof(float) * wchunk * d.A), &bar);
    }
    mbar_wait(&bar, phase, nullptr, 0);
    phase ^= 1u;
    if (d.A % 4 == 0) {
      // thread = (w-range group, k, 4 consecutive a): 16-byte shared loads, each
      // y_F value reused for 4 outputs; groups split the w range and their
      // partial sums are added in group order below
      const int per = d.K * (d.A / 4);
      const int groups = min((int)blockDim.x / per, 16);
      const int span = ((wchunk / 4 + groups - 1) / groups) * 4;
      const int t = threadIdx.x;
      if (t < groups * per) {
        const int gi = t / per, rem = t % per, k = rem / (d.A / 4), a4 = (rem % (d.A / 4)) * 4;
        const int w0c = gi * span, w1c = min(wchunk, w0c + span);
        const float* yk = ys + k * wchunk;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int w = w0c; w < w1c; w += 4) {
          const float4 y4 = *reinterpret_cast<const float4*>(yk + w);
          const float yv[4] = {y4.x, y4.y, y4.z, y4.w};
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const float4 wv = *reinterpret_cast<const float4*>(ws + (w + u) * d.A + a4);
            acc.x = fmaf(yv[u], wv.x, acc.x);
            acc.y = fmaf(yv[u], wv.y, acc.y);
            acc.z = fmaf(yv[u], wv.z, acc.z);
            acc.w = fmaf(yv[u], wv.w, acc.w);
          }
        }
        *reinterpret_cast<float4*>(red + (size_t)gi * KA + k * d.A + a4) = acc;
      }
      __syncthreads();
      for (int i = threadIdx.x; i < KA; i += blockDim.x) {
        float v = 0.f;
        for (int gi = 0; gi < groups; ++gi) v += red[(size_t)gi * KA + i];
        vs[i] += v;
      }
    } else {
      for (int i = threadIdx.x; i < KA; i += blockDim.x) {
        const int k = i / d.A, a = i % d.A;
        const float* yk = ys + k * wchunk;
        float acc0 = 0.f, acc1 = 0.f, acc2 = 0.f, acc3 = 0.f;
        for (int w = 0; w < wchunk; w += 4) {
          acc0 = fmaf(yk[w], ws[w * d.A + a], acc0);
          acc1 = fmaf(yk[w + 1], ws[(w + 1) * d.A + a], acc1);
          acc2 = fmaf(yk[w + 2], ws[(w + 2) * d.A + a], acc2);
          acc3 = fmaf(yk[w + 3], ws[(w + 3) * d.A + a], acc3);
        }
        vs[i] += (acc0 + acc1) + (acc2 + acc3);
      }
    }
  }
  __syncthreads();
  // v = b_out + partials of the cluster's CTAs in rank order, on CTA 0
  if (nsplit > 1) cluster_sync();  // every partial is complete
  if (q == 0) {
    const uint32_t vs_addr = smem_u32(vs);
    for (int i = threadIdx.x; i < KA; i += blockDim.x) {
      // every peer's partial requested before any is added (rank order kept)
      float pv[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int p = 1; p < 4; ++p)
        if (p < nsplit) pv[p] = ld_shared_cluster_f32(mapa_shared(vs_addr + 4u * (uint32_t)i, (uint32_t)p));
      float v = vs[i];
#pragma unroll
      for (int p = 1; p < 4; ++p)
        if (p < nsplit) v += pv[p];
      vs[i] = b_out[i % d.A] + v;
    }
  }
  __syncthreads();
  if (nsplit > 1) cluster_sync();  // the other CTAs may leave once CTA 0 has read them
  if (q != 0) return;
  const unsigned long long step = *step_idx;
  const float* dtr = dt + (size_t)r * d.K;
  float* colw = buffer + ((size_t)r * d.K * d.H + j) * d.A;
  for (int i = threadIdx.x; i < KA; i += blockDim.x) {
    const int k = i / d.A, a = i % d.A;
    const float v = vs[i];
    const float xk = __fadd_rn(xs[i], __fmul_rn(dtr[k], v));
    if (k == 0)
      out_chunk[((size_t)r * d.H + j) * d.A + a] = xk;
    else
      colw[(size_t)(k - 1) * slot + a] = xk;
    if (vel_out) vel_out[(((size_t)r * d.K + k) * d.H + j) * d.A + a] = v;
  }
  for (int a = threadIdx.x; a < d.A; a += blockDim.x) {
    const int e = j * d.A + a;
    colw[(size_t)(d.K - 1) * slot + a] =
        fresh ? fresh[(size_t)r * d.H * d.A + e] : tail_normal(seed, step, r, e);
  }
}

// CTAs per velocity cluster: each takes W / nsplit of the width (a multiple of 4).
static int vel_split(const StepDims& d) { return d.W % 16 == 0 ? 4 : 1; }

// Largest chunk of a CTA's width range (a divisor of it, multiple of 4) whose
// staging fits ~200 KB.  Every bulk copy then starts 16-byte aligned.
static int vel_chunk(const StepDims& d) {
  const size_t budget = 200 * 1024 - sizeof(float) * 18 * d.K * d.A;
  const int wq = d.W / vel_split(d);
  int c = wq;
  while (c > 4 && (sizeof(float) * (size_t)(d.K + d.A) * c > budget || wq % c || c % 4)) --c;
  return c;
}

static size_t vel_smem_bytes(const StepDims& d) {
  return sizeof(float) * ((size_t)18 * d.K * d.A + (size_t)(d.K + d.A) * vel_chunk(d));
}

cudaError_t final_init(const StepDims& d) {
  return cudaFuncSetAttribute(velocity_euler_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)vel_smem_bytes(d));
}

void launch_final_norm(const StepDims& d, float* h, const void* part, bool part_bf16,
                       int n_parts, long long part_stride, const float* mod, float* yF,
                       cudaStream_t s) {
  launch_resid_norm(d, h, part, part_bf16, n_parts, part_stride, mod, mod_off(d.L - 1, 5, d.W),
                    modf_off(d.L, 0, d.W), modf_off(d.L, 1, d.W), yF, false, s);
}

void launch_velocity_euler(const StepDims& d, const float* yF, const float* w_out_t,
                           const float* b_out, const float* dt, float* buffer, float* out_chunk,
                           float* vel_out, const float* fresh, unsigned long long seed,
                           const unsigned long long* step_idx, cudaStream_t s) {
  const int ns = vel_split(d);
  launch_pdl_cluster(velocity_euler_kernel, dim3(ns, d.H, d.B), dim3(kVelThreads),
                     vel_smem_bytes(d), s, dim3(ns, 1, 1), d, yF, w_out_t, b_out, dt, buffer, out_chunk,
                     vel_out, fresh, seed, step_idx, vel_chunk(d), ns);
}

// ----------------------------------------------------------------------------
// Time MLP layer (App. A.4 condition): out = silu(in W^T + b) for the few rows
// M = B*K of per-chunk timestep features; bf16 in / weights / out, fp32 math.
// One warp per output column; each CTA stages 16 input rows in shared memory and
// each lane reads 8 contiguous weights per 16-byte load.  K a multiple of 8.
// ----------------------------------------------------------------------------
constexpr int kGemvRows = 16;
constexpr int kGemvWarps = 8;    // 4 output columns per CTA, two warps (halves of K) each
constexpr int kGemvCols = kGemvWarps / 2;
constexpr int kGemvMaxK8 = 512;  // K <= 4096: each lane keeps its weights in registers

// Sum of v[0..15] over the 32 lanes of the warp for all 16 values at once: four
// steps that each send half of the lane's values to the partner lane and add the
// other half (16 values -> 1), then one last exchange.  Lane l ends with the total
// of value index ((l >> 4) & 1) * 8 + ((l >> 3) & 1) * 4 + ((l >> 2) & 1) * 2 +
// ((l >> 1) & 1) (both lanes of a pair hold it).  16 shuffles instead of 80.
__device__ __forceinline__ float warp_sum16(float (&v)[16], int lane) {
#pragma unroll
  for (int step = 0; step < 4; ++step) {
    const int b = 16 >> step, n = 8 >> step;  // partner bit, values kept
    const bool up = lane & b;
#pragma unroll
    for (int i = 0; i < n; ++i) {
      const float mine = up ? v[i + n] : v[i];
      const float theirs = up ? v[i] : v[i + n];
      v[i] = mine + __shfl_xor_sync(0xffffffffu, theirs, b);
    }
  }
  return v[0] + __shfl_xor_sync(0xffffffffu, v[0], 1);
}

__device__ __forceinline__ int warp_sum16_index(int lane) {
  return ((lane >> 4) & 1) * 8 + ((lane >> 3) & 1) * 4 + ((lane >> 2) & 1) * 2 + ((lane >> 1) & 1);
}

__global__ void __launch_bounds__(32 * kGemvWarps)
    gemv_silu_kernel(const bf16* __restrict__ in, const bf16* __restrict__ w,
                     const float* __restrict__ bias, bf16* __restrict__ out, int M, int N,
                     int K) {
  extern __shared__ __align__(16) uint4 sin4[];  // [16][K/8]
  __shared__ __align__(8) uint64_t bar;
  __shared__ float part[kGemvCols][kGemvRows];   // the upper K halves' sums
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int col = warp >> 1, khalf = warp & 1;
  const int n = blockIdx.x * kGemvCols + col;
  const int k8 = K / 8, k8h = k8 / 2;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_barrier_init();
  }
  __syncthreads();
  // this warp's half of the weight row: lane holds chunks kh*k8h + lane + 32 i
  // (the weights do not depend on earlier kernels: requested before waiting)
  uint4 wv[kGemvMaxK8 / 64];
  const uint4* wr = reinterpret_cast<const uint4*>(w + (size_t)min(n, N - 1) * K) + khalf * k8h;
#pragma unroll
  for (int i = 0; i < kGemvMaxK8 / 64; ++i)
    if (lane + 32 * i < k8h) wv[i] = __ldg(wr + lane + 32 * i);
  pdl_trigger();
  pdl_wait();
  const float bn = n < N ? bias[n] : 0.f;
  uint32_t phase = 0;
  for (int m0 = 0; m0 < M; m0 += kGemvRows) {
    const int mr = min(kGemvRows, M - m0);
    __syncthreads();
    if (threadIdx.x == 0) {
      mbar_arrive_expect_tx(&bar, (uint32_t)(mr * K * 2));
      bulk_load(sin4, in + (size_t)m0 * K, (uint32_t)(mr * K * 2), &bar);
    }
    mbar_wait(&bar, phase, nullptr, 0);
    phase ^= 1u;
    float acc[kGemvRows];
#pragma unroll
    for (int mm = 0; mm < kGemvRows; ++mm) acc[mm] = 0.f;
#pragma unroll
    for (int i = 0; i < kGemvMaxK8 / 64; ++i) {
      const int c = lane + 32 * i;
      if (c >= k8h) break;
      const __nv_bfloat162* w2 = reinterpret_cast<const __nv_bfloat162*>(&wv[i]);
      float wf[8];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float2 f = __bfloat1622float2(w2[u]);
        wf[2 * u] = f.x;
        wf[2 * u + 1] = f.y;
      }
#pragma unroll
      for (int mm = 0; mm < kGemvRows; ++mm) {
        if (mm >= mr) break;
        const uint4 xv = sin4[mm * k8 + khalf * k8h + c];
        const __nv_bfloat162* x2 = reinterpret_cast<const __nv_bfloat162*>(&xv);
        float a0 = acc[mm], a1 = 0.f;
#pragma unroll
        for (int u = 0; u < 4; u += 2) {
          const float2 f0 = __bfloat1622float2(x2[u]);
          const float2 f1 = __bfloat1622float2(x2[u + 1]);
          a0 = fmaf(f0.x, wf[2 * u], a0);
          a1 = fmaf(f0.y, wf[2 * u + 1], a1);
          a0 = fmaf(f1.x, wf[2 * u + 2], a0);
          a1 = fmaf(f1.y, wf[2 * u + 3], a1);
        }
        acc[mm] = a0 + a1;
      }
    }
    const float tot = warp_sum16(acc, lane);
    const int mm = warp_sum16_index(lane);
    if (khalf == 1 && (lane & 1) == 0) part[col][mm] = tot;
    __syncthreads();
    if (khalf == 0 && (lane & 1) == 0 && mm < mr && n < N)
      out[(size_t)(m0 + mm) * N + n] = __float2bfloat16_rn(silu_f(tot + part[col][mm] + bn));
  }
}

cudaError_t gemv_init(int K) {
  return cudaFuncSetAttribute(gemv_silu_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              kGemvRows * K * 2);
}

void launch_gemv_silu(const void* in, const void* w, const float* bias, void* out, int M, int N,
                      int K, cudaStream_t s) {
  if (M <= 0) return;
  launch_pdl(gemv_silu_kernel, dim3((N + kGemvCols - 1) / kGemvCols), dim3(32 * kGemvWarps),
             (size_t)kGemvRows * K * 2, s, (const bf16*)in, (const bf16*)w, bias, (bf16*)out, M, N,
             K);
}

// ----------------------------------------------------------------------------
// Per-step parameters.  The host writes each step's block into the next slot of a
// pinned ring and launches the step; this kernel, the step's first, copies the
// block of the slot its counter names into device memory and advances the counter
// (one step at a time on the stream, so every step reads the slot its own call
// filled).  No copy-engine transfer on the stream.
// ----------------------------------------------------------------------------
// With temb != nullptr it also writes the sinusoidal timestep embeddings of the
// step's first temb_rows noise levels (the first values of the block), as
// temb_kernel does, so that the time MLP reads them instead of every one of its CTAs
// computing them.
__global__ void __launch_bounds__(1024)
    fetch_params_kernel(const float* __restrict__ ring_host, int floats, int ring,
                        int* __restrict__ ctr, float* __restrict__ dst, bf16* __restrict__ temb,
                        int temb_rows, int W, const float2* __restrict__ freq) {
  __shared__ int slot;
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x == 0) slot = *ctr % ring;
  __syncthreads();
  const float* src = ring_host + (size_t)slot * floats;
  for (int i = threadIdx.x; i < floats; i += blockDim.x) dst[i] = src[i];
  if (temb) {
    const int half = W / 2;
    for (int i = threadIdx.x; i < temb_rows * half; i += blockDim.x) {
      const int row = i / half, j = i - row * half;
      const float2 sc = temb_sincos(src[row], freq[j]);
      temb[(size_t)row * W + j] = __float2bfloat16_rn(sc.x);
      temb[(size_t)row * W + half + j] = __float2bfloat16_rn(sc.y);
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) *ctr = (*ctr + 1) % ring;
}

void launch_fetch_params(const float* ring_host, int floats, int ring, int* ctr, float* dst,
                         void* temb, int temb_rows, int W, const float2* freq, cudaStream_t s) {
  launch_pdl(fetch_params_kernel, dim3(1), dim3(temb ? 1024 : 128), 0, s, ring_host, floats,
             ring, ctr, dst, (bf16*)temb, temb_rows, W, freq);
}

// The bf16 GeGLU epilogue's GELU on an fp32 array (introspection of its accuracy).
__global__ void geglu_gelu_kernel(const float* __restrict__ x, float* __restrict__ y, long long n) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x)
    y[i] = gelu_tanh_bf16out(x[i]);
}

void launch_geglu_gelu(const float* x, float* y, long long n, cudaStream_t s) {
  if (n <= 0) return;
  const long long blocks = std::min<long long>((n + 255) / 256, 4096);
  geglu_gelu_kernel<<<(unsigned)blocks, 256, 0, s>>>(x, y, n);
}

// ----------------------------------------------------------------------------
// tables and debug helpers
// ----------------------------------------------------------------------------
__global__ void rope_table_kernel(float2* table, uint32_t* table_h, int n_pos, int dh,
                                  double theta) {
  const int half = dh / 2;
  const long long n = (long long)n_pos * half;
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x) {
    const int pos = (int)(i / half), p = (int)(i % half);
    float2 v = make_float2(1.f, 0.f);
    if (theta != 0.0) {
      const double ang = (double)pos * pow(theta, -2.0 * (double)p / (double)dh);
      double sn, cs;
      sincos(ang, &sn, &cs);
      v = make_float2((float)cs, (float)sn);
    }
    table[i] = v;
    const __half2 hv = __floats2half2_rn(v.x, v.y);
    table_h[i] = *reinterpret_cast<const uint32_t*>(&hv);
  }
}

void launch_rope_table(float2* table, uint32_t* table_h, int n_pos, int dh, float theta,
                       cudaStream_t s) {
  rope_table_kernel<<<304, 256, 0, s>>>(table, table_h, n_pos, dh, (double)theta);
}

__global__ void to_f32_kernel(const void* src, bool src_bf16, float* dst, long long n) {
  pdl_wait();
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x)
    dst[i] = src_bf16 ? __bfloat162float(((const bf16*)src)[i]) : ((const float*)src)[i];
}

void launch_to_f32(const void* src, bool src_bf16, float* dst, long long n, cudaStream_t s) {
  if (n > 0) to_f32_kernel<<<304, 256, 0, s>>>(src, src_bf16, dst, n);
}

__global__ void gather_action_kv_kernel(const void* kv, bool act_bf16,
                                        const int* __restrict__ prefix_len, int T, int S_cap,
                                        int dh, float* dst) {
  const int m = blockIdx.x, r = m / T, t = m % T;
  pdl_wait();
  const size_t row = (size_t)r * S_cap + prefix_len[r] + t;
  for (int i = threadIdx.x; i < dh; i += blockDim.x)
    dst[(size_t)m * dh + i] = act_bf16 ? __bfloat162float(((const bf16*)kv)[row * dh + i])
                                       : ((const float*)kv)[row * dh + i];
}

void launch_gather_action_kv(const void* kv_layer, bool act_bf16, const int* prefix_len,
                             int B, int T, int S_cap, int dh, float* dst, cudaStream_t s) {
  gather_action_kv_kernel<<<B * T, 128, 0, s>>>(kv_layer, act_bf16, prefix_len, T, S_cap, dh,
                                                dst);
}

__global__ void mask_table_kernel(const int* __restrict__ prefix_len, int B, int T, int H,
                                  int* key_limit) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  pdl_wait();
  if (i >= B * T) return;
  key_limit[i] = attn_key_limit(prefix_len[i / T], i % T, H);
}

void launch_mask_table(const int* prefix_len, int B, int T, int H, int* key_limit,
                       cudaStream_t s) {
  mask_table_kernel<<<(B * T + 255) / 256, 256, 0, s>>>(prefix_len, B, T, H, key_limit);
}

}  // namespace fva
