// fp32 kernels of the step for the fp32 dtype (CUDA cores, full fp32 accuracy).
// The GEMM writes a plain fp32 product; separate small kernels apply the same
// post-processing the bf16 path fuses into its tensor-core epilogues.
#include "common.cuh"
#include "kernels.h"

namespace fva {

// C[M, N] = A[M, K] * B[N, K]^T.  64x64 tile, 16-deep K slices, 4x4 per thread.
__global__ void __launch_bounds__(256) f32_gemm_kernel(const float* __restrict__ A, int lda,
                                                       const float* __restrict__ B,
                                                       float* __restrict__ C, int ldc, int M,
                                                       int N, int K) {
  __shared__ float sA[16][64 + 4];
  __shared__ float sB[16][64 + 4];
  pdl_trigger();
  pdl_wait();
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += 16) {
    for (int i = threadIdx.x; i < 64 * 16; i += 256) {
      const int r = i / 16, kk = i % 16;
      const int gm = m0 + r, gn = n0 + r, gk = k0 + kk;
      sA[kk][r] = (gm < M && gk < K) ? A[(size_t)gm * lda + gk] : 0.f;
      sB[kk][r] = (gn < N && gk < K) ? B[(size_t)gn * K + gk] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        a[i] = sA[kk][ty * 4 + i];
        b[i] = sB[kk][tx * 4 + i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int gm = m0 + ty * 4 + i, gn = n0 + tx * 4 + j;
      if (gm < M && gn < N) C[(size_t)gm * ldc + gn] = acc[i][j];
    }
}

void launch_f32_gemm(const float* A, int lda, const float* B, float* C, int ldc, int M, int N,
                     int K, cudaStream_t s) {
  if (M <= 0) return;
  dim3 grid((N + 63) / 64, (M + 63) / 64);
  launch_pdl(f32_gemm_kernel, grid, dim3(256), 0, s, A, lda, B, C, ldc, M, N, K);
}

__global__ void f32_bias_act_kernel(const float* __restrict__ C, const float* __restrict__ bias,
                                    float* __restrict__ out, long long n, int N, bool silu) {
  pdl_trigger();
  pdl_wait();
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x) {
    const float v = C[i] + bias[i % N];
    out[i] = silu ? silu_f(v) : v;
  }
}

void launch_f32_bias_act(const float* C, const float* bias, float* out, int M, int N,
                         bool silu, cudaStream_t s) {
  if (M <= 0) return;
  launch_pdl(f32_bias_act_kernel, dim3(304), dim3(256), 0, s, C, bias, out, (long long)M * N, N,
             silu);
}

// C [M, nq*dh + 2*dh] = [q heads | k | v]; rotate q and k (rotate-half RoPE at
// position P_r + t), scatter q to [M, nq*dh] and k, v to the KV workspace rows.
__global__ void f32_qkv_rope_kernel(const float* __restrict__ C, float* __restrict__ q,
                                    float* __restrict__ kc, float* __restrict__ vc,
                                    const int* __restrict__ prefix_len,
                                    const float2* __restrict__ rope, int T, int S_cap, int nq,
                                    int dh) {
  const int m = blockIdx.x, r = m / T, t = m % T;
  pdl_trigger();
  pdl_wait();
  const int pos = prefix_len[r] + t;
  const int half = dh / 2, N = (nq + 2) * dh;
  const float* row = C + (size_t)m * N;
  for (int i = threadIdx.x; i < (nq + 2) * half; i += blockDim.x) {
    const int seg = i / half, d = i % half;
    const float a = row[seg * dh + d], b = row[seg * dh + d + half];
    float o1 = a, o2 = b;
    if (seg <= nq) {
      const float2 cs = rope[(size_t)pos * half + d];
      o1 = a * cs.x - b * cs.y;
      o2 = b * cs.x + a * cs.y;
    }
    float* dst = seg < nq ? q + (size_t)m * nq * dh + seg * dh
                          : (seg == nq ? kc : vc) + ((size_t)r * S_cap + pos) * dh;
    dst[d] = o1;
    dst[d + half] = o2;
  }
}

void launch_f32_qkv_rope(const float* C, float* q, float* kc, float* vc,
                         const int* prefix_len, const float2* rope, int M, int T, int S_cap,
                         int nq, int dh, cudaStream_t s) {
  if (M <= 0) return;
  launch_pdl(f32_qkv_rope_kernel, dim3(M), dim3(128), 0, s, C, q, kc, vc, prefix_len, rope, T,
             S_cap, nq, dh);
}

// C [M, 2F] = [gate | up] -> out [M, F] = gelu_tanh(gate) * up.
__global__ void f32_geglu_kernel(const float* __restrict__ C, float* __restrict__ out,
                                 long long n, int F) {
  pdl_trigger();
  pdl_wait();
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x) {
    const long long m = i / F, f = i % F;
    out[i] = gelu_tanh_f(C[m * 2 * F + f]) * C[m * 2 * F + F + f];
  }
}

void launch_f32_geglu(const float* C, float* out, int M, int F, cudaStream_t s) {
  if (M <= 0) return;
  launch_pdl(f32_geglu_kernel, dim3(304), dim3(256), 0, s, C, out, (long long)M * F, F);
}

// One CTA per (token row, head): softmax over the row's visible keys only.
__global__ void f32_attention_kernel(const float* __restrict__ q, const float* __restrict__ kc,
                                     const float* __restrict__ vc,
                                     const int* __restrict__ prefix_len,
                                     const int* __restrict__ pad_tokens, int block_diag,
                                     const int* __restrict__ prefix_src,
                                     float* __restrict__ out, int T, int H, int nq, int dh,
                                     int S_cap) {
  extern __shared__ float sm[];  // [dh] query, then [limit] scores
  const int m = blockIdx.x, head = blockIdx.y;
  const int r = m / T, t = m % T;
  pdl_trigger();
  pdl_wait();
  const int P = prefix_len[r];
  const int limit = attn_key_limit(P, t, H);
  // action keys below P + lo are padding (cold start) or, block-diagonal, other chunks
  const int pad = pad_tokens ? pad_tokens[r] : 0;
  const int lo = P + (block_diag ? max(pad, (t / H) * H) : pad);
  float* sq = sm;
  float* sc = sm + dh;
  const float* qrow = q + ((size_t)m * nq + head) * dh;
  for (int d = threadIdx.x; d < dh; d += blockDim.x) sq[d] = qrow[d];
  __syncthreads();
  const float scale = rsqrtf((float)dh);
  const float* K = kc + (size_t)r * S_cap * dh;
  const float* V = vc + (size_t)r * S_cap * dh;
  // a request that shares another's prefix reads the prefix keys from its rows
  const int src = prefix_src ? prefix_src[r] : r;
  const float* Ks = kc + (size_t)src * S_cap * dh;
  const float* Vs = vc + (size_t)src * S_cap * dh;
  for (int s = threadIdx.x; s < limit; s += blockDim.x) {
    const float* krow = (s < P ? Ks : K) + (size_t)s * dh;
    float acc = 0.f;
    for (int d = 0; d < dh; ++d) acc = fmaf(sq[d], krow[d], acc);
    sc[s] = (s < P || s >= lo) ? acc * scale : -INFINITY;
  }
  __syncthreads();
  __shared__ float red[32];
  float mx = -INFINITY;
  for (int s = threadIdx.x; s < limit; s += blockDim.x) mx = fmaxf(mx, sc[s]);
  mx = warp_max(mx);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
  __syncthreads();
  mx = -INFINITY;
  for (int w = 0; w < (int)(blockDim.x >> 5); ++w) mx = fmaxf(mx, red[w]);
  __syncthreads();
  float sum = 0.f;
  for (int s = threadIdx.x; s < limit; s += blockDim.x) {
    const float p = mx > -INFINITY ? expf(sc[s] - mx) : 0.f;  // no visible key: zeros
    sc[s] = p;
    sum += p;
  }
  sum = warp_sum(sum);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = sum;
  __syncthreads();
  sum = 0.f;
  for (int w = 0; w < (int)(blockDim.x >> 5); ++w) sum += red[w];
  const float inv = sum > 0.f ? 1.f / sum : 0.f;
  float* orow = out + ((size_t)m * nq + head) * dh;
  for (int d = threadIdx.x; d < dh; d += blockDim.x) {
    float acc = 0.f;
    for (int s = 0; s < limit; ++s) acc = fmaf(sc[s], (s < P ? Vs : V)[(size_t)s * dh + d], acc);
    orow[d] = acc * inv;
  }
}

void launch_f32_attention(const float* q, const float* kc, const float* vc,
                          const int* prefix_len, const int* pad_tokens, int block_diag,
                          const int* prefix_src, float* out, int B, int T, int H, int nq, int dh,
                          int S_cap, int max_keys, cudaStream_t s) {
  if (B * T <= 0) return;
  dim3 grid(B * T, nq);
  const size_t smem = sizeof(float) * (dh + max_keys);
  launch_pdl(f32_attention_kernel, grid, dim3(128), smem, s, q, kc, vc, prefix_len, pad_tokens,
             block_diag, prefix_src, out, T, H, nq, dh, S_cap);
}

}  // namespace fva
