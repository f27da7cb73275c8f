// Internal interface between the host library (fva_api.cu) and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace fva {

// Number of leading keys of [prefix ; action tokens] that action token t of a
// request with prefix length P attends to under the chunk-wise causal mask
// (own chunk bidirectional, earlier chunks fully, later chunks never).
__host__ __device__ __forceinline__ int attn_key_limit(int P, int t, int H) {
  return P + (t / H + 1) * H;
}

// Shapes of one step (all in elements).
struct StepDims {
  int B;       // active batch
  int Bmax;    // allocated batch
  int K, H, T; // chunks, tokens per chunk, K*H
  int A, W, nq, dh, Dq, F, L;
  int S_cap;   // KV rows per request and layer: max_prefix + T
  int N_mod;   // FiLM outputs per chunk: L*6W + 2W
  float eps;
  int n_sms;   // SMs of the device (launch-shape choices; 0: unknown)
};

// FiLM slice offsets inside one row of `mod` [B*K, N_mod].
__host__ __device__ __forceinline__ int mod_off(int l, int which, int W) {
  // which: 0 s1, 1 b1, 2 g1, 3 s2, 4 b2, 5 g2
  return l * 6 * W + which * W;
}
__host__ __device__ __forceinline__ int modf_off(int L, int which, int W) {
  // which: 0 sF, 1 bF
  return L * 6 * W + which * W;
}

// Sets the text fva_last_error() returns on the calling thread (fva_api.cu).
void set_last_error(const char* msg);

// ---------------------------------------------------------------- rowwise.cu
// act_bf16 selects the activation type (bf16 when true, else fp32).
// freq[j] = (hi, lo) two-float split of 2 / p_j, j < W/2 (see temb_kernel).
void launch_temb(const float* tau, const float2* freq, int rows, int W, void* out,
                 bool act_bf16, cudaStream_t s);

void launch_embed_norm(const StepDims& d, const float* buffer, const float* w_in_t,
                       const float* b_in, const float* mod, float* h, void* y, bool act_bf16,
                       int n_sms, cudaStream_t s);

// h += gate * sum_z part[z];  y = rmsnorm(h) * (1 + scale) + shift.
void launch_resid_norm(const StepDims& d, float* h, const void* part, bool part_bf16,
                       int n_parts, long long part_stride, const float* mod, int gate_off,
                       int scale_off, int shift_off, void* y, bool act_bf16, cudaStream_t s);

// Final residual + final FiLM RMSNorm (fp32 y_F into yF [B*K*H, W]), then
// out-projection, Euler update, emit, roll and tail (two launches).  w_out_t is
// W_out transposed, [W, A] fp32.  final_init sets the second kernel's
// shared-memory limit for these dimensions (once per handle).
cudaError_t final_init(const StepDims& d);
void launch_final_norm(const StepDims& d, float* h, const void* part, bool part_bf16,
                       int n_parts, long long part_stride, const float* mod, float* yF,
                       cudaStream_t s);
void launch_velocity_euler(const StepDims& d, const float* yF, const float* w_out_t,
                           const float* b_out, const float* dt, float* buffer, float* out_chunk,
                           float* vel_out, const float* fresh, unsigned long long seed,
                           const unsigned long long* step_idx, cudaStream_t s);

// out = silu(in W^T + bias), bf16 [M, K] x [N, K] -> bf16 [M, N]; K a multiple of 8.
// gemv_init sets the shared-memory limit for K (once per handle).
cudaError_t gemv_init(int K);
void launch_gemv_silu(const void* in, const void* w, const float* bias, void* out, int M, int N,
                      int K, cudaStream_t s);

// (cos, sin) of position x frequency for RoPE, fp32 and rounded to fp16 pairs.
void launch_rope_table(float2* table, uint32_t* table_h, int n_pos, int dh, float theta,
                       cudaStream_t s);

void launch_to_f32(const void* src, bool src_bf16, float* dst, long long n, cudaStream_t s);

// Gather action-token K or V of one layer into a dense [B*T, dh] fp32 array.
void launch_gather_action_kv(const void* kv_layer, bool act_bf16, const int* prefix_len,
                             int B, int T, int S_cap, int dh, float* dst, cudaStream_t s);

void launch_mask_table(const int* prefix_len, int B, int T, int H, int* key_limit,
                       cudaStream_t s);

// The step's parameter block (tau, dt, step index, padding tokens: `floats` values)
// from ring slot *ctr % ring of the pinned host ring `ring_host` (its device
// address) into `dst`; then ++*ctr.  The first kernel of every step.  With temb
// (bf16 [temb_rows, W]) it also writes the timestep embeddings of the block's first
// temb_rows values (freq as for launch_temb).
void launch_fetch_params(const float* ring_host, int floats, int ring, int* ctr, float* dst,
                         void* temb, int temb_rows, int W, const float2* freq, cudaStream_t s);

// y = the bf16 GeGLU epilogue's GELU of x (fp32 in and out).
void launch_geglu_gelu(const float* x, float* y, long long n, cudaStream_t s);


// ---------------------------------------------------------------- tc_gemm.cu
enum GemmMode {
  GEMM_BIAS_F32 = 0,      // out f32 = acc + bias
  GEMM_BIAS_SILU_BF16 = 1,// out bf16 = silu(acc + bias)
  GEMM_PARTIAL_F32 = 2,   // out f32 [split] = acc (split-K partial plane)
  GEMM_QKV_ROPE = 3,      // RoPE, q -> q buffer, k/v -> KV workspace (permuted weights)
  GEMM_GEGLU = 4,         // out bf16 = gelu(gate) * up (interleaved weights)
  GEMM_PARTIAL_BF16 = 5,  // out bf16 [split] = acc (split-K partial plane)
};

struct GemmEpi {
  void* out;
  const float* bias;
  int ldo;
  long long split_stride;
  // GEMM_QKV_ROPE
  void* q;
  void* kc;             // layer's [Bmax, S_cap, dh]
  void* vc;
  const int* prefix_len;
  const float2* rope;   // [n_pos, dh/2] (cos, sin)
  const uint32_t* rope_h;  // the same table as fp16 (cos, sin) pairs
  int T, S_cap, nq, dh;
  int* err;
  // rows of the A box (the activation tile) the kernel waits for: 0 = 128; fewer (a
  // multiple of 16) when every row fits them (the MMA still reads 128 rows; the rows
  // past the box are never stored)
  int a_rows;
  // optional L2 prefetch issued by the first CTA before its dependency wait:
  // pf_count ranges of pf_bytes (multiples of 16) at pf_base + i * pf_stride floats
  const float* pf_base;
  int pf_count, pf_bytes;
  long long pf_stride;
};

// Column tiles of the FiLM projection carried by the QKV or gate/up projection's
// launch: extra CTAs (grid.y >= y0, numbered (y - y0) * grid.x + x) each compute one
// kFilmTile-wide tile tile0 + f of out[rows, :] = a b^T + bias (the GEMM_BIAS_F32
// epilogue, the same arithmetic as the FiLM kernel's), on the SMs the projection
// leaves idle.
constexpr int kFilmTile = 64;
struct FilmTiles {
  CUtensorMap a;       // condition rows [rows, K], 16-row boxes
  CUtensorMap b;       // FiLM weights [N_mod, K], kFilmTile-row boxes
  float* out;          // modulation [rows, ldo]
  const float* bias;
  int ldo;
  int rows;            // at most 16
  int pre_stages;      // weight stages requested before the dependency wait (>= 1)
  int tile0, tiles;    // tiles 0: none
  int y0;              // set by the launcher
};

// Tile widths used for each GEMM of the step (the weight layouts depend on them).
constexpr int kBnQKV = 128;
constexpr int kBnGU = 256;
// QKV and gate/up tile width when every row fits one row tile (B*K*H <= 128):
// with so few rows the wide tiles leave most SMs idle.
constexpr int kBnSmall = 64;
constexpr int kBnResid = 128;
constexpr int kBnTime = 64;
constexpr int kBnFilm = 128;

// Prepare kernel attributes (max dynamic shared memory); call once per device.
cudaError_t tc_gemm_init();

// C = A[M, K] * B[N, K]^T on tcgen05 with the given epilogue.
// K must be a multiple of 64 and N of bn; M is any positive size.
cudaError_t launch_tc_gemm(int bn, int mode, const CUtensorMap* a, const CUtensorMap* b,
                           const GemmEpi& ep, int M, int N, int K, int splits,
                           cudaStream_t s);

// Persistent form for many tiles: min(grid, tiles) CTAs walk the (row tile,
// column tile) grid with two TMEM accumulators, no split-K.  bn/mode:
// (kBnQKV, QKV_ROPE), (kBnGU, GEGLU), (kBnResid, PARTIAL_BF16).
cudaError_t launch_tc_gemm_persist(int bn, int mode, const CUtensorMap* a, const CUtensorMap* b,
                                   const GemmEpi& ep, int M, int N, int K, int grid,
                                   cudaStream_t s);

// A QKV (GEMM_QKV_ROPE) or gate/up (GEMM_GEGLU) projection, per-tile form with one
// K split, together with FiLM column tiles (FilmTiles) in one launch.
cudaError_t launch_tc_gemm_film(int bn, int mode, const CUtensorMap* a, const CUtensorMap* b,
                                const GemmEpi& ep, int M, int N, int K, const FilmTiles& film,
                                cudaStream_t s);

// FiLM column tiles alone (one CTA per tile, the FilmTiles path of the launch
// above); K as for the condition rows.
cudaError_t launch_tc_film_tiles(const FilmTiles& film, int K, int* err, cudaStream_t s);

// Persistent weight-streaming form of (kBnFilm, BIAS_F32) for M <= 16 rows: at
// most `grid` CTAs (two per SM: pass twice the SM count) walk the N / kBnFilm
// column tiles.
cudaError_t launch_tc_gemm_stream(const CUtensorMap* a, const CUtensorMap* b, const GemmEpi& ep,
                                  int M, int N, int K, int grid, cudaStream_t s);

// ---------------------------------------------------------------- tc_attention.cu
struct AttnArgs {
  const int* prefix_len;
  void* out;            // bf16 [Bmax*T*nq, 256]
  void* part_o;         // bf16 [B*tiles, max_splits, 128, 256]: per-split O / l
  float2* part_ml;      // [B*tiles, max_splits, 128]
  int T, H, nq, S_cap, tiles_per_req, max_splits;
  int blocks_per_split;  // 64-key blocks per split, 1..4 (0: 4)
  int kv_row0;          // first KV row of this layer in the 2D view
  float scale_log2;     // log2(e) / sqrt(dh)
  int* err;
  // Action keys a row sees start at P + lo: lo = pad_tokens[r] (cold-start
  // padding; nullptr = 0), and under the block-diagonal mask at least the row's
  // own chunk start.
  const int* pad_tokens;
  int block_diag;
  // Key blocks wholly inside request r's prefix are read from the KV rows of
  // request prefix_src[r] (a shared prefix); nullptr: every request its own.
  const int* prefix_src;
};

constexpr int kAttnKeysPerSplit = 256;
constexpr int kAttnKeyBlock = 64;

// Largest cluster of the attention's cluster form (one cluster of CTAs per query
// tile, the tile's key blocks dealt out evenly, at most kAttnMaxBlocksPerCta each).
constexpr int kAttnMaxClusterSplits = 8;
constexpr int kAttnMaxBlocksPerCta = 4;

cudaError_t tc_attention_init();
// How many clusters of `splits` attention CTAs the device can hold at once (0: the
// cluster form cannot run with that many splits).
int attn_cluster_capacity(int splits);
// Attention kernel.  cluster: each query tile is one cluster of a.max_splits CTAs
// (<= kAttnMaxClusterSplits) that share the tile's key blocks and combine their
// results inside the cluster; otherwise fixed splits of a.blocks_per_split blocks, and
// launch_attn_merge then combines them from a.part_o / a.part_ml (it launches
// nothing when no tile can have more than one split).
cudaError_t launch_attn_merge(const AttnArgs& a, int B, cudaStream_t s);
cudaError_t launch_tc_attention(const CUtensorMap* q, const CUtensorMap* k,
                                const CUtensorMap* v, const AttnArgs& a, int B,
                                cudaStream_t s, bool cluster);

// ---------------------------------------------------------------- simt_f32.cu
// C[M, N] = A[M, K] (lda) * B[N, K]^T, fp32 on CUDA cores.
void launch_f32_gemm(const float* A, int lda, const float* B, float* C, int ldc, int M, int N,
                     int K, cudaStream_t s);
void launch_f32_bias_act(const float* C, const float* bias, float* out, int M, int N,
                         bool silu, cudaStream_t s);
void launch_f32_qkv_rope(const float* C, float* q, float* kc, float* vc,
                         const int* prefix_len, const float2* rope, int M, int T, int S_cap,
                         int nq, int dh, cudaStream_t s);
void launch_f32_geglu(const float* C, float* out, int M, int F, cudaStream_t s);
// prefix_src: per request, the request whose KV rows hold its prefix keys
// (nullptr: its own).
void launch_f32_attention(const float* q, const float* kc, const float* vc,
                          const int* prefix_len, const int* pad_tokens, int block_diag,
                          const int* prefix_src, float* out, int B, int T, int H, int nq, int dh,
                          int S_cap, int max_keys, cudaStream_t s);

}  // namespace fva
