// Row-wise kernels of the streaming step: timestep embedding, the fused action
// in-projection + first FiLM RMSNorm, the fused split-K reduction + gated
// residual + FiLM RMSNorm, and the fused final norm + out-projection + Euler
// update + emit + buffer roll + tail noise.  Plus small table / debug helpers.
#include "common.cuh"
#include "kernels.h"

namespace fva {

// ----------------------------------------------------------------------------
// sinusoidal timestep embedding of every chunk's noise level (App. A.4 FiLM
// condition input): e = [sin(2 pi tau / p_j) | cos(2 pi tau / p_j)],
// p_j = t_min (t_max / t_min)^(j / (W/2 - 1)).  Arguments in double precision.
// ----------------------------------------------------------------------------
template <typename Act>
__global__ void temb_kernel(const float* __restrict__ tau, int W, double tmin, double tmax,
                            Act* __restrict__ out) {
  const int row = blockIdx.x;
  const int half = W / 2;
  pdl_trigger();
  pdl_wait();
  const double t = (double)tau[row];
  for (int j = threadIdx.x; j < half; j += blockDim.x) {
    const double period = tmin * pow(tmax / tmin, (double)j / (double)(half - 1));
    const double arg = 2.0 * 3.14159265358979323846 * t / period;
    double sn, cs;
    sincos(arg, &sn, &cs);
    out[(size_t)row * W + j] = from_float<Act>((float)sn);
    out[(size_t)row * W + half + j] = from_float<Act>((float)cs);
  }
}

void launch_temb(const float* tau, int rows, int W, float tmin, float tmax, void* out,
                 bool act_bf16, cudaStream_t s) {
  if (rows <= 0) return;
  if (act_bf16)
    launch_pdl(temb_kernel<bf16>, dim3(rows), dim3(256), 0, s, tau, W, (double)tmin,
               (double)tmax, (bf16*)out);
  else
    launch_pdl(temb_kernel<float>, dim3(rows), dim3(256), 0, s, tau, W, (double)tmin,
               (double)tmax, (float*)out);
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
  t = t < 32 ? 32 : (t > 256 ? 256 : t);
  return (t + 31) & ~31;
}

// ----------------------------------------------------------------------------
// action in-projection h = x W_in^T + b_in, then layer 0's FiLM RMSNorm.
// One CTA per token row; w_in_t is W_in transposed, [A, W] fp32.
// ----------------------------------------------------------------------------
template <typename Act>
__global__ void embed_norm_kernel(StepDims d, const float* __restrict__ buffer,
                                  const float* __restrict__ w_in_t,
                                  const float* __restrict__ b_in, const float* __restrict__ mod,
                                  float* __restrict__ h, Act* __restrict__ y) {
  __shared__ float xs[128];
  __shared__ float red[32];
  const int m = blockIdx.x;
  const int r = m / d.T, t = m % d.T, c = t / d.H;
  pdl_trigger();
  pdl_wait();
  const float* x = buffer + (size_t)m * d.A;  // buffer [B, K, H, A] = rows of A
  for (int a = threadIdx.x; a < d.A; a += blockDim.x) xs[a] = x[a];
  __syncthreads();
  float* hrow = h + (size_t)m * d.W;
  float ss = 0.f;
  for (int col = threadIdx.x * 4; col < d.W; col += blockDim.x * 4) {
    float4 acc = *reinterpret_cast<const float4*>(b_in + col);
    for (int a = 0; a < d.A; ++a) {
      const float xa = xs[a];
      const float4 w = *reinterpret_cast<const float4*>(w_in_t + (size_t)a * d.W + col);
      acc.x = fmaf(xa, w.x, acc.x);
      acc.y = fmaf(xa, w.y, acc.y);
      acc.z = fmaf(xa, w.z, acc.z);
      acc.w = fmaf(xa, w.w, acc.w);
    }
    *reinterpret_cast<float4*>(hrow + col) = acc;
    ss += acc.x * acc.x + acc.y * acc.y + acc.z * acc.z + acc.w * acc.w;
  }
  ss = block_sum(ss, red);
  const float* mrow = mod + (size_t)(r * d.K + c) * d.N_mod;
  modulated_norm_row<Act>(hrow, ss, d.W, d.eps, mrow + mod_off(0, 0, d.W),
                          mrow + mod_off(0, 1, d.W), y + (size_t)m * d.W);
}

void launch_embed_norm(const StepDims& d, const float* buffer, const float* w_in_t,
                       const float* b_in, const float* mod, float* h, void* y, bool act_bf16,
                       cudaStream_t s) {
  const int rows = d.B * d.T;
  if (rows <= 0) return;
  if (act_bf16)
    launch_pdl(embed_norm_kernel<bf16>, dim3(rows), dim3(row_threads(d.W)), 0, s, d, buffer,
               w_in_t, b_in, mod, h, (bf16*)y);
  else
    launch_pdl(embed_norm_kernel<float>, dim3(rows), dim3(row_threads(d.W)), 0, s, d, buffer,
               w_in_t, b_in, mod, h, (float*)y);
}

// ----------------------------------------------------------------------------
// h += gate_c * sum_z part[z]  (split-K partials reduced in fixed order z = 0..),
// then y = FiLM RMSNorm(h) with the next norm's (scale, shift).  One CTA per row.
// ----------------------------------------------------------------------------
template <typename Act>
__global__ void resid_norm_kernel(StepDims d, float* __restrict__ h,
                                  const float* __restrict__ part, int n_parts,
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
  float ss = 0.f;
  for (int col = threadIdx.x * 4; col < d.W; col += blockDim.x * 4) {
    float4 acc = __ldcg(reinterpret_cast<const float4*>(part + (size_t)m * d.W + col));
    for (int z = 1; z < n_parts; ++z) {
      const float4 p =
          __ldcg(reinterpret_cast<const float4*>(part + z * part_stride + (size_t)m * d.W + col));
      acc.x += p.x; acc.y += p.y; acc.z += p.z; acc.w += p.w;
    }
    const float4 g = *reinterpret_cast<const float4*>(mrow + gate_off + col);
    float4 hv = *reinterpret_cast<const float4*>(hrow + col);
    hv.x = fmaf(g.x, acc.x, hv.x);
    hv.y = fmaf(g.y, acc.y, hv.y);
    hv.z = fmaf(g.z, acc.z, hv.z);
    hv.w = fmaf(g.w, acc.w, hv.w);
    *reinterpret_cast<float4*>(hrow + col) = hv;
    ss += hv.x * hv.x + hv.y * hv.y + hv.z * hv.z + hv.w * hv.w;
  }
  ss = block_sum(ss, red);
  modulated_norm_row<Act>(hrow, ss, d.W, d.eps, mrow + scale_off, mrow + shift_off,
                          y + (size_t)m * d.W);
}

void launch_resid_norm(const StepDims& d, float* h, const float* part, int n_parts,
                       long long part_stride, const float* mod, int gate_off, int scale_off,
                       int shift_off, void* y, bool act_bf16, cudaStream_t s) {
  const int rows = d.B * d.T;
  if (rows <= 0) return;
  if (act_bf16)
    launch_pdl(resid_norm_kernel<bf16>, dim3(rows), dim3(row_threads(d.W)), 0, s, d, h, part,
               n_parts, part_stride, mod, gate_off, scale_off, shift_off, (bf16*)y);
  else
    launch_pdl(resid_norm_kernel<float>, dim3(rows), dim3(row_threads(d.W)), 0, s, d, h, part,
               n_parts, part_stride, mod, gate_off, scale_off, shift_off, (float*)y);
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
// Final kernel.  One CTA per (token position j within a chunk, request r): it
// owns column j of every chunk of request r, so the in-place roll of the buffer
// is race-free.  For every chunk k: finish the residual stream, final FiLM
// RMSNorm, velocity v = y W_out^T + b_out; then x'_k = x_k + dt_k v_k (fp32,
// separately rounded multiply and add), out = x'_1, slot k <- x'_{k+1},
// tail <- z.
// ----------------------------------------------------------------------------
__global__ void final_kernel(StepDims d, float* __restrict__ h, const float* __restrict__ part,
                             int n_parts, long long part_stride, const float* __restrict__ mod,
                             const float* __restrict__ w_out, const float* __restrict__ b_out,
                             const float* __restrict__ dt, float* __restrict__ buffer,
                             float* __restrict__ out_chunk, float* __restrict__ vel_out,
                             const float* __restrict__ fresh, unsigned long long seed,
                             const unsigned long long* __restrict__ step_idx) {
  extern __shared__ float vs[];  // [K, A] velocities of this column
  const int j = blockIdx.x, r = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  const int lgate = mod_off(d.L - 1, 5, d.W);
  pdl_trigger();
  pdl_wait();
  for (int k = warp; k < d.K; k += nw) {
    const int t = k * d.H + j;
    const size_t m = (size_t)r * d.T + t;
    const float* mrow = mod + (size_t)(r * d.K + k) * d.N_mod;
    float* hrow = h + m * d.W;
    float ss = 0.f;
    for (int col = lane * 4; col < d.W; col += 128) {
      float4 acc = __ldcg(reinterpret_cast<const float4*>(part + m * d.W + col));
      for (int z = 1; z < n_parts; ++z) {
        const float4 p =
            __ldcg(reinterpret_cast<const float4*>(part + z * part_stride + m * d.W + col));
        acc.x += p.x; acc.y += p.y; acc.z += p.z; acc.w += p.w;
      }
      const float4 g = *reinterpret_cast<const float4*>(mrow + lgate + col);
      float4 hv = *reinterpret_cast<const float4*>(hrow + col);
      hv.x = fmaf(g.x, acc.x, hv.x);
      hv.y = fmaf(g.y, acc.y, hv.y);
      hv.z = fmaf(g.z, acc.z, hv.z);
      hv.w = fmaf(g.w, acc.w, hv.w);
      *reinterpret_cast<float4*>(hrow + col) = hv;
      ss += hv.x * hv.x + hv.y * hv.y + hv.z * hv.z + hv.w * hv.w;
    }
    ss = warp_sum(ss);
    const float rn = rsqrtf(ss / (float)d.W + d.eps);
    const float* sF = mrow + modf_off(d.L, 0, d.W);
    const float* bF = mrow + modf_off(d.L, 1, d.W);
    for (int a0 = 0; a0 < d.A; a0 += 32) {
      float acc[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) acc[i] = 0.f;
      for (int col = lane * 4; col < d.W; col += 128) {
        const float4 hv = *reinterpret_cast<const float4*>(hrow + col);
        const float4 sc = *reinterpret_cast<const float4*>(sF + col);
        const float4 sh = *reinterpret_cast<const float4*>(bF + col);
        const float y0 = hv.x * rn * (1.f + sc.x) + sh.x, y1 = hv.y * rn * (1.f + sc.y) + sh.y;
        const float y2 = hv.z * rn * (1.f + sc.z) + sh.z, y3 = hv.w * rn * (1.f + sc.w) + sh.w;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          if (a0 + i < d.A) {
            const float4 w = *reinterpret_cast<const float4*>(w_out + (size_t)(a0 + i) * d.W + col);
            acc[i] = fmaf(y0, w.x, fmaf(y1, w.y, fmaf(y2, w.z, fmaf(y3, w.w, acc[i]))));
          }
        }
      }
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const float s = warp_sum(acc[i]);
        if (lane == i && a0 + i < d.A) vs[k * d.A + a0 + i] = s + b_out[a0 + i];
      }
    }
  }
  __syncthreads();
  const unsigned long long step = *step_idx;
  const float* dtr = dt + (size_t)r * d.K;
  for (int a = threadIdx.x; a < d.A; a += blockDim.x) {
    float* col = buffer + ((size_t)r * d.K * d.H + j) * d.A + a;  // + k*H*A selects the slot
    const size_t slot = (size_t)d.H * d.A;
    out_chunk[((size_t)r * d.H + j) * d.A + a] = __fadd_rn(col[0], __fmul_rn(dtr[0], vs[a]));
    if (vel_out) vel_out[((size_t)r * d.K * d.H + j) * d.A + a] = vs[a];
    for (int k = 1; k < d.K; ++k) {
      const float v = vs[k * d.A + a];
      const float xk = __fadd_rn(col[k * slot], __fmul_rn(dtr[k], v));
      col[(k - 1) * slot] = xk;
      if (vel_out) vel_out[(((size_t)r * d.K + k) * d.H + j) * d.A + a] = v;
    }
    const int e = j * d.A + a;
    col[(size_t)(d.K - 1) * slot] =
        fresh ? fresh[(size_t)r * d.H * d.A + e] : tail_normal(seed, step, r, e);
  }
}

void launch_final(const StepDims& d, float* h, const float* part, int n_parts,
                  long long part_stride, const float* mod, const float* w_out,
                  const float* b_out, const float* dt, float* buffer, float* out_chunk,
                  float* vel_out, const float* fresh, unsigned long long seed,
                  const unsigned long long* step_idx, cudaStream_t s) {
  dim3 grid(d.H, d.B);
  const size_t smem = sizeof(float) * d.K * d.A;
  launch_pdl(final_kernel, grid, dim3(256), smem, s, d, h, part, n_parts, part_stride, mod,
             w_out, b_out, dt, buffer, out_chunk, vel_out, fresh, seed, step_idx);
}

// ----------------------------------------------------------------------------
// tables and debug helpers
// ----------------------------------------------------------------------------
__global__ void rope_table_kernel(float2* table, int n_pos, int dh, double theta) {
  const int half = dh / 2;
  const long long n = (long long)n_pos * half;
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x) {
    const int pos = (int)(i / half), p = (int)(i % half);
    if (theta == 0.0) {
      table[i] = make_float2(1.f, 0.f);
    } else {
      const double ang = (double)pos * pow(theta, -2.0 * (double)p / (double)dh);
      double sn, cs;
      sincos(ang, &sn, &cs);
      table[i] = make_float2((float)cs, (float)sn);
    }
  }
}

void launch_rope_table(float2* table, int n_pos, int dh, float theta, cudaStream_t s) {
  rope_table_kernel<<<304, 256, 0, s>>>(table, n_pos, dh, (double)theta);
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
