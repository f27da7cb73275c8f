// Host side of libfva: the C ABI declared in include/fva.h.
//
// Owns weights (re-laid-out for the kernels at load time), the per-layer prefix +
// action K/V workspace, activations and scratch; validates every call on the host;
// enqueues the step (§3.2, Algorithm 1) as a fixed sequence of kernels and, by
// default, replays it as a CUDA graph (one graph per batch size / buffer pair).
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "common.cuh"
#include "fva.h"
#include "kernels.h"

using namespace fva;

namespace {

thread_local std::string g_last_error;

fva_status fail(fva_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return st;
}

#define CUDA_TRY(expr)                                                                   \
  do {                                                                                   \
    cudaError_t e_ = (expr);                                                             \
    if (e_ != cudaSuccess)                                                               \
      return fail(e_ == cudaErrorMemoryAllocation ? FVA_ERR_OOM : FVA_ERR_CUDA,          \
                  "%s failed: %s (%s:%d)", #expr, cudaGetErrorString(e_), __FILE__,      \
                  __LINE__);                                                             \
  } while (0)

inline float bf16_to_f32(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  std::memcpy(&f, &u, 4);
  return f;
}

struct DeviceGuard {
  int prev = -1;
  explicit DeviceGuard(int dev) {
    cudaGetDevice(&prev);
    if (prev != dev) cudaSetDevice(dev);
  }
  ~DeviceGuard() {
    int cur;
    if (cudaGetDevice(&cur) == cudaSuccess && cur != prev && prev >= 0) cudaSetDevice(prev);
  }
};

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

fva_status get_encoder() {
  if (g_encode) return FVA_OK;
  cudaDriverEntryPointQueryResult q;
  void* fn = nullptr;
  cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                   cudaEnableDefault, &q);
  if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn)
    return fail(FVA_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
  g_encode = (PFN_cuTensorMapEncodeTiled_v12000)fn;
  return FVA_OK;
}

// 2D bf16 row-major [rows, cols] tensor; box = box_rows x 64 columns, 128-byte swizzle.
fva_status make_map(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols,
                    uint32_t box_rows) {
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS)
    return fail(FVA_ERR_CUDA, "cuTensorMapEncodeTiled(rows=%llu cols=%llu box=%u) failed: %d",
                (unsigned long long)rows, (unsigned long long)cols, box_rows, (int)r);
  return FVA_OK;
}

struct LayerW {
  void* w_qkv = nullptr;  // [Dq + 2 dh, W]
  void* w_o = nullptr;    // [W, Dq]
  void* w_gu = nullptr;   // [2F, W]
  void* w_d = nullptr;    // [W, F]
  CUtensorMap m_qkv, m_o, m_gu, m_d;
};

struct GraphEntry {
  int batch;
  float* buffer;
  float* out;
  bool fresh;
  bool reuse_film;
  bool serial_film;
  cudaGraphExec_t exec;
  uint64_t last_use;
};

int choose_splits(int tiles, int kblocks) {
  int best = 1;
  for (int s : {2, 4, 8})
    if (kblocks % s == 0 && kblocks / s >= 4 && tiles * s <= 160) best = s;
  return best;
}

}  // namespace

struct fva_handle {
  fva_config cfg;
  int device = 0;
  bool bf16 = true;
  size_t act = 2;  // bytes per activation / weight element
  int W, nq, dh, Dq, F, A, K, H, T, L, Bmax, Pmax, S_cap, N_qkv, N_mod, BKmax, Mmax;
  int tiles_per_req = 0, attn_max_splits = 0, attn_bps = 4;
  // CTAs per cluster of the attention's cluster form (0: the global form, whose key
  // splits the merge kernel combines; always so with FVA_FLAG_NO_ATTN_CLUSTER)
  int attn_ncl = 0;
  // attn_cluster_capacity by split count (-1: not asked yet)
  int cluster_cap[kAttnMaxClusterSplits + 1] = {-1, -1, -1, -1, -1, -1, -1, -1, -1};
  static_assert(kAttnMaxClusterSplits == 8, "initialiser of cluster_cap");
  int n_sms = 0;
  int bn_qkv = kBnQKV, bn_gu = kBnGU;  // tile widths of the QKV and gate/up weight layouts
  // persistent GEMMs where a projection has at least two tiles per SM
  // (FVA_FLAG_NO_PERSISTENT_GEMM: off)
  bool persist_on = true;

  std::vector<void*> allocs;
  // weights
  void* warena = nullptr;
  size_t warena_bytes = 0;
  float *w_in_t = nullptr, *b_in = nullptr, *b_t1 = nullptr, *b_t2 = nullptr, *b_mod = nullptr;
  float *w_out_t = nullptr, *b_out = nullptr;  // w_out_t: [W, A]
  void *w_t1 = nullptr, *w_t2 = nullptr, *w_mod = nullptr;
  std::vector<LayerW> layers;
  CUtensorMap m_wt1, m_wt2, m_wmod;
  CUtensorMap m_wmod_q;  // FiLM weights in kFilmTile-row boxes (FiLM tiles in projections)
  bool weights_loaded = false;
  // prefix / KV workspace
  void *kc = nullptr, *vc = nullptr;
  int* prefix_len_dev = nullptr;
  int* prefix_src_dev = nullptr;  // [Bmax]: request whose rows hold the prefix keys
  std::vector<int> prefix_src;    // host copy
  std::vector<int> layer_len;  // [Bmax * L], -1 = never set
  float2* rope = nullptr;
  uint32_t* rope_h = nullptr;  // fp16 copy for the bf16 QKV epilogue
  float2* temb_freq = nullptr;  // [W/2] two-float split of 2 / p_j
  // activations / scratch
  void *temb = nullptr, *t1 = nullptr, *cond = nullptr, *y = nullptr, *q = nullptr;
  void *attn = nullptr, *mlp = nullptr;
  float *mod = nullptr, *h = nullptr, *part = nullptr, *c32 = nullptr, *vel = nullptr;
  float* yF = nullptr;  // [Mmax, W] fp32 output of the final FiLM RMSNorm
  float* fresh = nullptr;
  __nv_bfloat16* att_part_o = nullptr;
  float2* att_part_ml = nullptr;
  int* err_dev = nullptr;
  CUtensorMap m_temb, m_t1, m_cond, m_y, m_attn, m_mlp, m_q, m_k, m_v;
  CUtensorMap m_cond16;  // cond with 16-row boxes (streaming FiLM GEMM)
  // Fewer than 128 rows (Mmax < 128, the paper's own buffer shapes): the QKV and
  // gate/up projections read y through boxes of y_box = Mmax rounded up to 16 rows
  // (FVA_FLAG_FULL_A_BOX: 128-row boxes); 0 = 128-row boxes
  int y_box = 0;
  CUtensorMap m_ybox;
  // per-step parameters: [tau BKmax | dt BKmax | step u64]
  float* params_dev = nullptr;
  float* params_host = nullptr;  // pinned ring [FVA_PARAM_RING][params_floats]
  float* params_host_dev = nullptr;  // the ring's device address (mapped pinned memory)
  int* ring_ctr = nullptr;  // device: slot the next step's fetch kernel reads
  bool fetch_enqueued = false;  // enqueue_step queued the parameter fetch
  int params_floats = 0;
  cudaEvent_t ring_ev[FVA_PARAM_RING] = {};
  bool ring_used[FVA_PARAM_RING] = {};
  int ring_pos = 0;
  uint64_t step_index = 0;
  // asynchronous error word polling
  int* err_host = nullptr;
  cudaEvent_t err_ev = nullptr;
  bool err_pending = false;
  uint64_t polls = 0;
  // profiling graph (fva_step_profile): events between kernels
  std::vector<cudaEvent_t> prof_events;
  cudaGraphExec_t prof_exec = nullptr;
  int prof_batch = 0;
  float *prof_buf = nullptr, *prof_out = nullptr;
  std::vector<int> prof_kind, prof_layer;
  // graphs
  cudaStream_t cap_stream = nullptr;
  std::vector<GraphEntry> graphs;
  uint64_t use_clock = 0;
  // the FiLM modulation in `mod` / `cond` was computed for these noise levels
  bool film_valid = false;
  int film_batch = 0;
  std::vector<float> film_tau;

  float* tau_dev() const { return params_dev; }
  // padding tokens (K - n_valid) * H per request of the current step
  int* pad_dev() const { return reinterpret_cast<int*>(params_dev + 2 * BKmax + 2); }
  float* dt_dev() const { return params_dev + BKmax; }
  unsigned long long* step_dev() const {
    return reinterpret_cast<unsigned long long*>(params_dev + 2 * BKmax);
  }
};

namespace {

// Cluster size of the attention's cluster form for `tiles` query tiles of at most
// `nkb` 64-key blocks each, or 0 for the global form (splits of `global_bps` blocks
// and the merge kernel): the largest n <= 8 (and <= nkb) whose clusters the device
// holds all at once and that leaves every CTA fewer blocks than the global form's
// splits.  Clusters in a second wave would wait for whole groups of SMs, and every
// CTA of a cluster stays resident until its tile is combined; the combination
// through distributed shared memory costs about as much as the merge kernel, so
// the cluster form pays only with shorter CTAs.
int attn_cluster_size(fva_handle* h, long long tiles, int nkb, int global_bps) {
  if (h->cfg.flags & FVA_FLAG_NO_ATTN_CLUSTER) return 0;
  for (int n = std::min(kAttnMaxClusterSplits, nkb); n >= 2; --n) {
    const int blocks = (nkb + n - 1) / n;  // fewer CTAs: more blocks each
    if (blocks > kAttnMaxBlocksPerCta || blocks >= global_bps) break;
    if (h->cluster_cap[n] < 0) h->cluster_cap[n] = attn_cluster_capacity(n);
    if (h->cluster_cap[n] >= tiles) return n;
  }
  return 0;
}

fva_status dev_alloc(fva_handle* h, void** p, size_t bytes) {
  if (bytes == 0) bytes = 256;
  cudaError_t e = cudaMalloc(p, bytes);
  if (e != cudaSuccess) {
    *p = nullptr;
    cudaGetLastError();
    return fail(FVA_ERR_OOM, "cudaMalloc(%zu) failed: %s", bytes, cudaGetErrorString(e));
  }
  h->allocs.push_back(*p);
  e = cudaMemset(*p, 0, bytes);
  if (e != cudaSuccess) return fail(FVA_ERR_CUDA, "cudaMemset failed: %s", cudaGetErrorString(e));
  return FVA_OK;
}

template <typename T>
fva_status dalloc(fva_handle* h, T** p, size_t count, size_t elem = sizeof(T)) {
  void* v = nullptr;
  fva_status st = dev_alloc(h, &v, count * elem);
  *p = (T*)v;
  return st;
}

void release(fva_handle* h) {
  if (!h) return;
  cudaDeviceSynchronize();
  for (auto& g : h->graphs) cudaGraphExecDestroy(g.exec);
  h->graphs.clear();
  if (h->prof_exec) cudaGraphExecDestroy(h->prof_exec);
  h->prof_exec = nullptr;
  for (auto e : h->prof_events) cudaEventDestroy(e);
  h->prof_events.clear();
  for (void* p : h->allocs) cudaFree(p);
  h->allocs.clear();
  if (h->warena) cudaFree(h->warena);
  if (h->params_host) cudaFreeHost(h->params_host);
  if (h->err_host) cudaFreeHost(h->err_host);
  for (auto& e : h->ring_ev)
    if (e) cudaEventDestroy(e);
  if (h->err_ev) cudaEventDestroy(h->err_ev);
  if (h->cap_stream) cudaStreamDestroy(h->cap_stream);
  cudaGetLastError();
}

fva_status validate_config(const fva_config* c) {
  if (!c) return fail(FVA_ERR_INVALID_ARG, "config is NULL");
  if (c->abi_version != FVA_ABI_VERSION)
    return fail(FVA_ERR_INVALID_ARG, "abi_version %d != %d", c->abi_version, FVA_ABI_VERSION);
  if (c->dtype != FVA_FP32 && c->dtype != FVA_BF16)
    return fail(FVA_ERR_INVALID_ARG, "dtype %d is not FVA_FP32 or FVA_BF16", c->dtype);
  if (c->n_layers < 1 || c->width < 8 || c->n_q_heads < 1 || c->head_dim < 2 ||
      c->mlp_dim < 1 || c->action_dim < 1 || c->n_chunks < 1 || c->chunk_tokens < 1 ||
      c->max_batch < 1 || c->max_prefix < 0)
    return fail(FVA_ERR_INVALID_ARG, "non-positive dimension in config");
  if (c->n_kv_heads != 1)
    return fail(FVA_ERR_UNSUPPORTED, "n_kv_heads must be 1 (multi-query attention)");
  if (c->head_dim % 2 || c->width % 4)
    return fail(FVA_ERR_INVALID_ARG, "head_dim must be even and width a multiple of 4");
  if (!(c->rms_eps > 0.f) || !(c->rope_theta >= 0.f) || !(c->t_min_period > 0.f) ||
      !(c->t_max_period >= c->t_min_period) || !std::isfinite(c->t_max_period) ||
      !std::isfinite(c->rope_theta))
    return fail(FVA_ERR_INVALID_ARG, "bad rms_eps / rope_theta / timestep periods");
  if (c->action_dim > 128) return fail(FVA_ERR_UNSUPPORTED, "action_dim > 128");
  if (c->flags & ~(FVA_FLAG_NO_GRAPH | FVA_FLAG_BLOCK_DIAGONAL | FVA_FLAG_NO_PERSISTENT_GEMM |
                   FVA_FLAG_NO_ATTN_CLUSTER | FVA_FLAG_FULL_A_BOX))
    return fail(FVA_ERR_INVALID_ARG, "unknown flags 0x%x", c->flags);
  const long long T = (long long)c->n_chunks * c->chunk_tokens;
  if (T * c->max_batch > (1LL << 24) || c->max_prefix > (1 << 20) || c->n_layers > 1024)
    return fail(FVA_ERR_UNSUPPORTED, "sizes too large");
  if (c->dtype == FVA_BF16) {
    if (c->head_dim != 256) return fail(FVA_ERR_UNSUPPORTED, "bf16 kernels need head_dim 256");
    if (128 % c->n_q_heads != 0 || c->n_q_heads > 16)
      return fail(FVA_ERR_UNSUPPORTED, "bf16 kernels need n_q_heads in {1,2,4,8,16}");
    if (c->width % 128 || c->mlp_dim % 128)
      return fail(FVA_ERR_UNSUPPORTED, "bf16 kernels need width and mlp_dim multiples of 128");
    const long long keys = c->max_prefix + T;
    if ((keys + kAttnKeysPerSplit - 1) / kAttnKeysPerSplit > 32)
      return fail(FVA_ERR_UNSUPPORTED, "max_prefix + K*H above 8192 keys");
    if ((long long)c->n_layers * c->max_batch * (c->max_prefix + T) >= (1LL << 31))
      return fail(FVA_ERR_UNSUPPORTED, "KV workspace rows exceed 2^31");
  } else {
    if (c->head_dim > 256) return fail(FVA_ERR_UNSUPPORTED, "fp32 kernels need head_dim <= 256");
    if ((c->head_dim + c->max_prefix + T) * 4 > 48 * 1024)
      return fail(FVA_ERR_UNSUPPORTED, "fp32 attention: max_prefix + K*H too large");
  }
  return FVA_OK;
}

}  // namespace

// =============================================================================
// create / destroy
// =============================================================================
extern "C" int32_t fva_num_weights(const fva_config* cfg) {
  if (!cfg || cfg->n_layers < 1) return 0;
  return 6 + 11 * cfg->n_layers + 4;
}

extern "C" fva_status fva_weight_shape(const fva_config* c, int32_t index, int64_t* rows,
                                       int64_t* cols) {
  if (!c || !rows || !cols) return fail(FVA_ERR_INVALID_ARG, "NULL argument");
  fva_status st = validate_config(c);
  if (st != FVA_OK) return st;
  const int64_t W = c->width, A = c->action_dim, F = c->mlp_dim, dh = c->head_dim;
  const int64_t Dq = (int64_t)c->n_q_heads * dh;
  const int n = fva_num_weights(c);
  if (index < 0 || index >= n) return fail(FVA_ERR_INVALID_ARG, "weight index %d out of range", index);
  int64_t r = 1, k = 1;
  if (index < 6) {
    const int64_t s[6][2] = {{W, A}, {1, W}, {W, W}, {1, W}, {W, W}, {1, W}};
    r = s[index][0];
    k = s[index][1];
  } else if (index < 6 + 11 * c->n_layers) {
    const int j = (index - 6) % 11;
    const int64_t s[11][2] = {{3 * W, W}, {1, 3 * W}, {3 * W, W}, {1, 3 * W}, {Dq, W}, {dh, W},
                              {dh, W},    {W, Dq},    {F, W},     {F, W},     {W, F}};
    r = s[j][0];
    k = s[j][1];
  } else {
    const int j = index - 6 - 11 * c->n_layers;
    const int64_t s[4][2] = {{2 * W, W}, {1, 2 * W}, {A, W}, {1, A}};
    r = s[j][0];
    k = s[j][1];
  }
  *rows = r;
  *cols = k;
  return FVA_OK;
}

static fva_status create_impl(const fva_config* cfg, fva_handle* h) {
  const fva_config& c = *cfg;
  h->cfg = c;
  h->bf16 = c.dtype == FVA_BF16;
  h->act = h->bf16 ? 2 : 4;
  h->W = c.width;
  h->nq = c.n_q_heads;
  h->dh = c.head_dim;
  h->Dq = c.n_q_heads * c.head_dim;
  h->F = c.mlp_dim;
  h->A = c.action_dim;
  h->K = c.n_chunks;
  h->H = c.chunk_tokens;
  h->T = h->K * h->H;
  h->L = c.n_layers;
  h->Bmax = c.max_batch;
  h->Pmax = c.max_prefix;
  h->S_cap = h->Pmax + h->T;
  h->N_qkv = h->Dq + 2 * h->dh;
  h->N_mod = h->L * 6 * h->W + 2 * h->W;
  h->BKmax = ((h->Bmax * h->K) + 1) & ~1;  // even, keeps the u64 step word aligned
  h->Mmax = h->Bmax * h->T;
  h->layers.resize(h->L);
  h->layer_len.assign((size_t)h->Bmax * h->L, -1);
  h->prefix_src.resize(h->Bmax);
  for (int r = 0; r < h->Bmax; ++r) h->prefix_src[r] = r;
  CUDA_TRY(cudaGetDevice(&h->device));
  fva_status st;
  if (h->bf16) {
    if ((st = get_encoder()) != FVA_OK) return st;
    CUDA_TRY(tc_gemm_init());
    CUDA_TRY(tc_attention_init());
    if (h->W > 4096) return fail(FVA_ERR_UNSUPPORTED, "bf16 kernels need width <= 4096");
    CUDA_TRY(gemv_init(h->W));
    CUDA_TRY(cudaDeviceGetAttribute(&h->n_sms, cudaDevAttrMultiProcessorCount, h->device));
  }
  const size_t a = h->act;
  const size_t kv_elems = (size_t)h->L * h->Bmax * h->S_cap * h->dh;
  if ((st = dalloc(h, &h->kc, kv_elems, a)) || (st = dalloc(h, &h->vc, kv_elems, a)) ||
      (st = dalloc(h, &h->prefix_len_dev, h->Bmax)) ||
      (st = dalloc(h, &h->prefix_src_dev, h->Bmax)) ||
      (st = dalloc(h, &h->rope, (size_t)h->S_cap * (h->dh / 2))) ||
      (st = dalloc(h, &h->rope_h, (size_t)h->S_cap * (h->dh / 2))) ||
      (st = dalloc(h, &h->temb, (size_t)h->BKmax * h->W, a)) ||
      (st = dalloc(h, &h->t1, (size_t)h->BKmax * h->W, a)) ||
      (st = dalloc(h, &h->cond, (size_t)h->BKmax * h->W, a)) ||
      (st = dalloc(h, &h->mod, (size_t)h->BKmax * h->N_mod)) ||
      (st = dalloc(h, &h->h, (size_t)h->Mmax * h->W)) ||
      (st = dalloc(h, &h->y, (size_t)h->Mmax * h->W, a)) ||
      (st = dalloc(h, &h->q, (size_t)h->Mmax * h->Dq, a)) ||
      (st = dalloc(h, &h->attn, (size_t)h->Mmax * h->Dq, a)) ||
      (st = dalloc(h, &h->mlp, (size_t)h->Mmax * h->F, a)) ||
      (st = dalloc(h, &h->vel, (size_t)h->Mmax * h->A)) ||
      (st = dalloc(h, &h->yF, (size_t)h->Mmax * h->W)) ||
      (st = dalloc(h, &h->fresh, (size_t)h->Bmax * h->H * h->A)) ||
      (st = dalloc(h, &h->err_dev, 1)))
    return st;
  // split-K partial planes: enough for the largest split count any batch size uses
  size_t part_elems = (size_t)h->Mmax * h->W;
  if (h->bf16) {
    for (int B = 1; B <= h->Bmax; ++B) {
      const int M = B * h->T, tiles = ((M + 127) / 128) * (h->W / kBnResid);
      const int s = std::max(choose_splits(tiles, h->Dq / 64), choose_splits(tiles, h->F / 64));
      part_elems = std::max(part_elems, (size_t)s * M * h->W);
    }
  }
  if (h->bf16) {
    if (h->Mmax <= 128) {  // one row tile: narrower QKV and gate/up tiles
      h->bn_qkv = kBnSmall;
      h->bn_gu = kBnSmall;
    }
    h->persist_on = !(c.flags & FVA_FLAG_NO_PERSISTENT_GEMM);
  }
  if ((st = dalloc(h, &h->part, part_elems))) return st;
  if (!h->bf16) {
    const size_t c32 = std::max({(size_t)h->Mmax * std::max(h->N_qkv, 2 * h->F),
                                 (size_t)h->BKmax * h->N_mod, (size_t)h->BKmax * h->W});
    if ((st = dalloc(h, &h->c32, c32))) return st;
  }
  if (h->bf16) {
    h->tiles_per_req = (h->T * h->nq + 127) / 128;
    // 64-key blocks per split: the largest of 4, 2, 1 that still gives about half
    // as many CTAs as SMs (few query tiles: short splits), at most 32 splits
    const int nkb_max = (h->S_cap + 63) / 64;
    h->attn_bps = 4;
    while (h->attn_bps > 1 &&
           (long long)h->tiles_per_req * h->Bmax * ((nkb_max + h->attn_bps - 1) / h->attn_bps) <
               std::max(1, h->n_sms / 2))
      h->attn_bps /= 2;
    while ((nkb_max + h->attn_bps - 1) / h->attn_bps > 32 && h->attn_bps < 4) h->attn_bps *= 2;
    h->attn_max_splits = (nkb_max + h->attn_bps - 1) / h->attn_bps;
    h->attn_ncl = attn_cluster_size(h, (long long)h->Bmax * h->tiles_per_req, nkb_max, h->attn_bps);
    const size_t tiles = (size_t)h->Bmax * h->tiles_per_req;
    if ((st = dalloc(h, &h->att_part_o, tiles * h->attn_max_splits * 128 * 256)) ||
        (st = dalloc(h, &h->att_part_ml, tiles * h->attn_max_splits * 128)))
      return st;
  }
  h->params_floats = 2 * h->BKmax + 2 + h->Bmax;
  if ((st = dalloc(h, &h->params_dev, h->params_floats))) return st;
  CUDA_TRY(cudaMallocHost((void**)&h->params_host,
                          sizeof(float) * h->params_floats * FVA_PARAM_RING));
  CUDA_TRY(cudaHostGetDevicePointer((void**)&h->params_host_dev, h->params_host, 0));
  if ((st = dalloc(h, &h->ring_ctr, 1))) return st;
  CUDA_TRY(cudaMallocHost((void**)&h->err_host, sizeof(int)));
  *h->err_host = 0;
  for (auto& e : h->ring_ev) CUDA_TRY(cudaEventCreateWithFlags(&e, cudaEventDisableTiming));
  CUDA_TRY(cudaEventCreateWithFlags(&h->err_ev, cudaEventDisableTiming));
  CUDA_TRY(cudaStreamCreateWithFlags(&h->cap_stream, cudaStreamNonBlocking));
  {
    StepDims d{};
    d.K = h->K;
    d.A = h->A;
    d.W = h->W;
    if (sizeof(float) * ((size_t)18 * d.K * d.A + (size_t)(d.K + d.A) * 4) > 200 * 1024)
      return fail(FVA_ERR_UNSUPPORTED, "n_chunks * action_dim too large for the final kernel");
    CUDA_TRY(final_init(d));
  }
  launch_rope_table(h->rope, h->rope_h, h->S_cap, h->dh, c.rope_theta, 0);
  CUDA_TRY(cudaGetLastError());
  {
    // 2 / p_j in half turns per unit tau, p_j = t_min (t_max / t_min)^(j / (W/2 - 1))
    const int half = h->W / 2;
    std::vector<float2> fq(half);
    for (int j = 0; j < half; ++j) {
      const double period = (double)c.t_min_period *
                            std::pow((double)c.t_max_period / (double)c.t_min_period,
                                     half > 1 ? (double)j / (double)(half - 1) : 0.0);
      const double v = 2.0 / period;
      const float hi = (float)v;
      fq[j] = make_float2(hi, (float)(v - (double)hi));
    }
    if ((st = dalloc(h, &h->temb_freq, half))) return st;
    CUDA_TRY(cudaMemcpy(h->temb_freq, fq.data(), sizeof(float2) * half, cudaMemcpyHostToDevice));
  }
  if (h->bf16) {
    const uint64_t M = h->Mmax, BK = h->BKmax;
    if ((st = make_map(&h->m_temb, h->temb, BK, h->W, 128)) ||
        (st = make_map(&h->m_t1, h->t1, BK, h->W, 128)) ||
        (st = make_map(&h->m_cond, h->cond, BK, h->W, 128)) ||
        (st = make_map(&h->m_cond16, h->cond, BK, h->W, 16)) ||
        (st = make_map(&h->m_y, h->y, M, h->W, 128)) ||

        (st = make_map(&h->m_attn, h->attn, M, h->Dq, 128)) ||
        (st = make_map(&h->m_mlp, h->mlp, M, h->F, 128)) ||
        (st = make_map(&h->m_q, h->q, M * h->nq, h->dh, 128)) ||
        (st = make_map(&h->m_k, h->kc, (uint64_t)h->L * h->Bmax * h->S_cap, h->dh, 64)) ||
        (st = make_map(&h->m_v, h->vc, (uint64_t)h->L * h->Bmax * h->S_cap, h->dh, 64)))
      return st;
    if (M < 128 && !(h->cfg.flags & FVA_FLAG_FULL_A_BOX)) {
      h->y_box = (int)((M + 15) / 16 * 16);
      if ((st = make_map(&h->m_ybox, h->y, M, h->W, h->y_box))) return st;
    }
  }
  CUDA_TRY(cudaDeviceSynchronize());
  return FVA_OK;
}

extern "C" fva_status fva_create(const fva_config* cfg, fva_handle** out) {
  if (!out) return fail(FVA_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  fva_status st = validate_config(cfg);
  if (st != FVA_OK) return st;
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess || ndev == 0) {
    cudaGetLastError();
    return fail(FVA_ERR_CUDA, "no CUDA device");
  }
  fva_handle* h = new (std::nothrow) fva_handle();
  if (!h) return fail(FVA_ERR_OOM, "host allocation failed");
  st = create_impl(cfg, h);
  if (st != FVA_OK) {
    std::string msg = g_last_error;
    release(h);
    delete h;
    g_last_error = msg;
    return st;
  }
  *out = h;
  return FVA_OK;
}

extern "C" void fva_destroy(fva_handle* h) {
  if (!h) return;
  DeviceGuard g(h->device);
  release(h);
  delete h;
}

extern "C" const char* fva_last_error(void) { return g_last_error.c_str(); }

void fva::set_last_error(const char* msg) { g_last_error = msg; }

// =============================================================================
// weights
// =============================================================================
namespace {

// Host copy of tensor i as fp32 values.
fva_status fetch(const fva_handle* h, const void* src, size_t n, bool on_device,
                 std::vector<float>& out) {
  out.resize(n);
  if (h->bf16) {
    std::vector<uint16_t> tmp(n);
    if (on_device)
      CUDA_TRY(cudaMemcpy(tmp.data(), src, n * 2, cudaMemcpyDeviceToHost));
    else
      std::memcpy(tmp.data(), src, n * 2);
    for (size_t i = 0; i < n; ++i) out[i] = bf16_to_f32(tmp[i]);
  } else {
    if (on_device)
      CUDA_TRY(cudaMemcpy(out.data(), src, n * 4, cudaMemcpyDeviceToHost));
    else
      std::memcpy(out.data(), src, n * 4);
  }
  return FVA_OK;
}

uint16_t f32_to_bf16_exact(float f) {  // values came from bf16, so truncation is exact
  uint32_t u;
  std::memcpy(&u, &f, 4);
  return (uint16_t)(u >> 16);
}

// Append rows (each `cols` values) to a weight image in the activation dtype.
void push_rows(const fva_handle* h, std::vector<uint8_t>& img, const float* rows, size_t n) {
  const size_t off = img.size();
  img.resize(off + n * h->act);
  if (h->bf16) {
    uint16_t* d = (uint16_t*)(img.data() + off);
    for (size_t i = 0; i < n; ++i) d[i] = f32_to_bf16_exact(rows[i]);
  } else {
    std::memcpy(img.data() + off, rows, n * 4);
  }
}

void align_img(std::vector<uint8_t>& img) { img.resize((img.size() + 1023) & ~size_t(1023)); }

}  // namespace

extern "C" fva_status fva_load_weights(fva_handle* h, const void* const* tensors,
                                       int32_t n_tensors, int32_t on_device) {
  if (!h || !tensors) return fail(FVA_ERR_INVALID_ARG, "NULL argument");
  const int n = fva_num_weights(&h->cfg);
  if (n_tensors != n)
    return fail(FVA_ERR_INVALID_ARG, "expected %d tensors, got %d", n, n_tensors);
  for (int i = 0; i < n; ++i)
    if (!tensors[i]) return fail(FVA_ERR_INVALID_ARG, "tensor %d is NULL", i);
  DeviceGuard guard(h->device);
  CUDA_TRY(cudaDeviceSynchronize());
  const int W = h->W, A = h->A, F = h->F, dh = h->dh, Dq = h->Dq, L = h->L;
  std::vector<std::vector<float>> t(n);
  for (int i = 0; i < n; ++i) {
    int64_t r, c;
    fva_weight_shape(&h->cfg, i, &r, &c);
    fva_status st = fetch(h, tensors[i], (size_t)(r * c), on_device != 0, t[i]);
    if (st != FVA_OK) return st;
  }
  auto li = [&](int l, int j) -> std::vector<float>& { return t[6 + 11 * l + j]; };
  const int fin = 6 + 11 * L;

  // fp32 small tensors: in-projection (transposed to [A, W]), biases, out-projection.
  std::vector<float> f32img;
  auto f32_off = [&](const float* p, size_t cnt) {
    size_t o = f32img.size();
    f32img.insert(f32img.end(), p, p + cnt);
    f32img.resize((f32img.size() + 255) & ~size_t(255));
    return o;
  };
  std::vector<float> w_in_t((size_t)A * W);
  for (int w = 0; w < W; ++w)
    for (int a = 0; a < A; ++a) w_in_t[(size_t)a * W + w] = t[0][(size_t)w * A + a];
  std::vector<float> b_mod;
  b_mod.reserve(h->N_mod);
  for (int l = 0; l < L; ++l) {
    b_mod.insert(b_mod.end(), li(l, 1).begin(), li(l, 1).end());
    b_mod.insert(b_mod.end(), li(l, 3).begin(), li(l, 3).end());
  }
  b_mod.insert(b_mod.end(), t[fin + 1].begin(), t[fin + 1].end());
  const size_t o_win = f32_off(w_in_t.data(), w_in_t.size());
  const size_t o_bin = f32_off(t[1].data(), W);
  const size_t o_bt1 = f32_off(t[3].data(), W);
  const size_t o_bt2 = f32_off(t[5].data(), W);
  const size_t o_bmod = f32_off(b_mod.data(), b_mod.size());
  std::vector<float> w_out_t((size_t)W * A);  // [W, A]
  for (int a2 = 0; a2 < A; ++a2)
    for (int w = 0; w < W; ++w) w_out_t[(size_t)w * A + a2] = t[fin + 2][(size_t)a2 * W + w];
  const size_t o_wout = f32_off(w_out_t.data(), (size_t)A * W);
  const size_t o_bout = f32_off(t[fin + 3].data(), A);

  // matrices in the activation dtype, laid out for the kernels.
  std::vector<uint8_t> img;
  img.reserve(((size_t)L * (h->N_qkv * W + W * Dq + 2 * F * W + W * F) + h->N_mod * W +
               2 * W * W) * h->act + 1024 * (4 * L + 8));
  auto place = [&](const float* rows, size_t cnt) {
    align_img(img);
    size_t o = img.size();
    push_rows(h, img, rows, cnt);
    return o;
  };
  const size_t o_wt1 = place(t[2].data(), (size_t)W * W);
  const size_t o_wt2 = place(t[4].data(), (size_t)W * W);
  std::vector<float> wmod;
  wmod.reserve((size_t)h->N_mod * W);
  for (int l = 0; l < L; ++l) {
    wmod.insert(wmod.end(), li(l, 0).begin(), li(l, 0).end());
    wmod.insert(wmod.end(), li(l, 2).begin(), li(l, 2).end());
  }
  wmod.insert(wmod.end(), t[fin].begin(), t[fin].end());
  const size_t o_wmod = place(wmod.data(), wmod.size());
  std::vector<size_t> o_qkv(L), o_o(L), o_gu(L), o_d(L);
  std::vector<float> qkv((size_t)h->N_qkv * W), gu((size_t)2 * F * W);
  for (int l = 0; l < L; ++l) {
    // original rows: [q heads (Dq) | k (dh) | v (dh)]
    auto src_row = [&](int n) -> const float* {
      if (n < Dq) return li(l, 4).data() + (size_t)n * W;
      if (n < Dq + dh) return li(l, 5).data() + (size_t)(n - Dq) * W;
      return li(l, 6).data() + (size_t)(n - Dq - dh) * W;
    };
    for (int n2 = 0; n2 < h->N_qkv; ++n2) {
      int src = n2;
      if (h->bf16) {  // rotate-half partners side by side inside each QKV tile
        const int bq = h->bn_qkv;
        const int half = bq / 2, seg = n2 / dh, within = n2 % dh;
        const int tj = within / bq, c = within % bq;
        const int d = c < half ? tj * half + c : tj * half + (c - half) + dh / 2;
        src = seg * dh + d;
      }
      std::memcpy(qkv.data() + (size_t)n2 * W, src_row(src), sizeof(float) * W);
    }
    for (int n2 = 0; n2 < 2 * F; ++n2) {
      const float* s;
      if (h->bf16) {  // gate rows then matching up rows inside each gate/up tile
        const int bg = h->bn_gu;
        const int half = bg / 2, j = n2 / bg, c = n2 % bg;
        const int f = j * half + (c < half ? c : c - half);
        s = (c < half ? li(l, 8) : li(l, 9)).data() + (size_t)f * W;
      } else {
        s = (n2 < F ? li(l, 8).data() + (size_t)n2 * W : li(l, 9).data() + (size_t)(n2 - F) * W);
      }
      std::memcpy(gu.data() + (size_t)n2 * W, s, sizeof(float) * W);
    }
    o_qkv[l] = place(qkv.data(), qkv.size());
    o_o[l] = place(li(l, 7).data(), (size_t)W * Dq);
    o_gu[l] = place(gu.data(), gu.size());
    o_d[l] = place(li(l, 10).data(), (size_t)W * F);
  }
  align_img(img);
  const size_t f32_base = img.size();
  img.resize(f32_base + f32img.size() * 4);
  std::memcpy(img.data() + f32_base, f32img.data(), f32img.size() * 4);

  // upload into a fresh arena (replacing any previous weights)
  for (auto& g : h->graphs) cudaGraphExecDestroy(g.exec);
  h->graphs.clear();
  if (h->prof_exec) cudaGraphExecDestroy(h->prof_exec);
  h->prof_exec = nullptr;
  if (h->warena) cudaFree(h->warena);
  h->warena = nullptr;
  h->weights_loaded = false;
  h->film_valid = false;
  void* arena = nullptr;
  cudaError_t e = cudaMalloc(&arena, img.size());
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(FVA_ERR_OOM, "weight arena cudaMalloc(%zu) failed", img.size());
  }
  h->warena = arena;
  h->warena_bytes = img.size();
  CUDA_TRY(cudaMemcpy(arena, img.data(), img.size(), cudaMemcpyHostToDevice));
  uint8_t* base = (uint8_t*)arena;
  float* fb = (float*)(base + f32_base);
  h->w_in_t = fb + o_win;
  h->b_in = fb + o_bin;
  h->b_t1 = fb + o_bt1;
  h->b_t2 = fb + o_bt2;
  h->b_mod = fb + o_bmod;
  h->w_out_t = fb + o_wout;
  h->b_out = fb + o_bout;
  h->w_t1 = base + o_wt1;
  h->w_t2 = base + o_wt2;
  h->w_mod = base + o_wmod;
  for (int l = 0; l < L; ++l) {
    LayerW& lw = h->layers[l];
    lw.w_qkv = base + o_qkv[l];
    lw.w_o = base + o_o[l];
    lw.w_gu = base + o_gu[l];
    lw.w_d = base + o_d[l];
    if (h->bf16) {
      fva_status st;
      if ((st = make_map(&lw.m_qkv, lw.w_qkv, h->N_qkv, W, h->bn_qkv)) ||
          (st = make_map(&lw.m_o, lw.w_o, W, Dq, kBnResid)) ||
          (st = make_map(&lw.m_gu, lw.w_gu, 2 * F, W, h->bn_gu)) ||
          (st = make_map(&lw.m_d, lw.w_d, W, F, kBnResid)))
        return st;
    }
  }
  if (h->bf16) {
    fva_status st;
    if ((st = make_map(&h->m_wt1, h->w_t1, W, W, kBnTime)) ||
        (st = make_map(&h->m_wt2, h->w_t2, W, W, kBnTime)) ||
        (st = make_map(&h->m_wmod, h->w_mod, h->N_mod, W, kBnFilm)) ||
        (st = make_map(&h->m_wmod_q, h->w_mod, h->N_mod, W, kFilmTile)))
      return st;
  }
  h->weights_loaded = true;
  return FVA_OK;
}

// =============================================================================
// prefix K/V
// =============================================================================
namespace {
__global__ void set_len_kernel(int* dst, int v) { *dst = v; }
__global__ void set_share_kernel(int* len, int* src, int r, int v, int s) {
  len[r] = v;
  src[r] = s;
}

// Request r's prefix was replaced: requests that shared it lose the share (their
// steps report a missing prefix until they are set or shared again), and r itself
// reads its own rows again.
void drop_shares_of(fva_handle* h, int r, cudaStream_t s) {
  for (int q = 0; q < h->Bmax; ++q)
    if (q != r && h->prefix_src[q] == r) {
      h->prefix_src[q] = q;
      for (int l = 0; l < h->L; ++l) h->layer_len[(size_t)q * h->L + l] = -1;
      set_share_kernel<<<1, 1, 0, s>>>(h->prefix_len_dev, h->prefix_src_dev, q, 0, q);
    }
  h->prefix_src[r] = r;
}
}  // namespace

extern "C" fva_status fva_set_prefix_kv(fva_handle* h, int32_t request, int32_t layer,
                                        const void* k, const void* v, int32_t len,
                                        int32_t on_device, fva_stream stream) {
  if (!h) return fail(FVA_ERR_INVALID_ARG, "handle is NULL");
  if (request < 0 || request >= h->Bmax)
    return fail(FVA_ERR_INVALID_ARG, "request %d outside [0, %d)", request, h->Bmax);
  if (layer < -1 || layer >= h->L)
    return fail(FVA_ERR_INVALID_ARG, "layer %d outside [-1, %d)", layer, h->L);
  if (len < 0 || len > h->Pmax)
    return fail(FVA_ERR_INVALID_ARG, "prefix length %d outside [0, %d]", len, h->Pmax);
  if (len > 0 && (!k || !v)) return fail(FVA_ERR_INVALID_ARG, "k or v is NULL");
  DeviceGuard guard(h->device);
  cudaStream_t s = (cudaStream_t)stream;
  drop_shares_of(h, request, s);
  const size_t row = (size_t)h->dh * h->act, bytes = (size_t)len * row;
  const cudaMemcpyKind kind = on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
  const int l0 = layer < 0 ? 0 : layer, l1 = layer < 0 ? h->L : layer + 1;
  for (int l = l0; l < l1; ++l) {
    const size_t dst = ((size_t)l * h->Bmax + request) * h->S_cap * row;
    const size_t src = layer < 0 ? (size_t)l * bytes : 0;
    if (bytes) {
      CUDA_TRY(cudaMemcpyAsync((uint8_t*)h->kc + dst, (const uint8_t*)k + src, bytes, kind, s));
      CUDA_TRY(cudaMemcpyAsync((uint8_t*)h->vc + dst, (const uint8_t*)v + src, bytes, kind, s));
    }
    h->layer_len[(size_t)request * h->L + l] = len;
  }
  set_share_kernel<<<1, 1, 0, s>>>(h->prefix_len_dev, h->prefix_src_dev, request, len, request);
  CUDA_TRY(cudaGetLastError());
  return FVA_OK;
}

extern "C" fva_status fva_share_prefix_kv(fva_handle* h, int32_t request, int32_t src_request,
                                          fva_stream stream) {
  if (!h) return fail(FVA_ERR_INVALID_ARG, "handle is NULL");
  if (request < 0 || request >= h->Bmax || src_request < 0 || src_request >= h->Bmax)
    return fail(FVA_ERR_INVALID_ARG, "request %d / src_request %d outside [0, %d)", request,
                src_request, h->Bmax);
  if (request == src_request) return fail(FVA_ERR_INVALID_ARG, "a request cannot share itself");
  if (h->prefix_src[src_request] != src_request)
    return fail(FVA_ERR_STATE, "request %d itself shares another request's prefix", src_request);
  const int len = h->layer_len[(size_t)src_request * h->L];
  for (int l = 0; l < h->L; ++l)
    if (len < 0 || h->layer_len[(size_t)src_request * h->L + l] != len)
      return fail(FVA_ERR_STATE, "request %d has no complete prefix K/V", src_request);
  DeviceGuard guard(h->device);
  cudaStream_t s = (cudaStream_t)stream;
  drop_shares_of(h, request, s);
  // the 64-key block that straddles the prefix end also holds action keys, so it
  // is read from this request's rows: copy the prefix tail there
  const int tail0 = h->bf16 ? (len / 64) * 64 : len;
  const size_t row = (size_t)h->dh * h->act;
  for (int l = 0; l < h->L; ++l) {
    const size_t src = (((size_t)l * h->Bmax + src_request) * h->S_cap + tail0) * row;
    const size_t dst = (((size_t)l * h->Bmax + request) * h->S_cap + tail0) * row;
    if (len > tail0) {
      CUDA_TRY(cudaMemcpyAsync((uint8_t*)h->kc + dst, (const uint8_t*)h->kc + src,
                               (size_t)(len - tail0) * row, cudaMemcpyDeviceToDevice, s));
      CUDA_TRY(cudaMemcpyAsync((uint8_t*)h->vc + dst, (const uint8_t*)h->vc + src,
                               (size_t)(len - tail0) * row, cudaMemcpyDeviceToDevice, s));
    }
    h->layer_len[(size_t)request * h->L + l] = len;
  }
  h->prefix_src[request] = src_request;
  set_share_kernel<<<1, 1, 0, s>>>(h->prefix_len_dev, h->prefix_src_dev, request, len,
                                   src_request);
  CUDA_TRY(cudaGetLastError());
  return FVA_OK;
}

// =============================================================================
// the step
// =============================================================================
namespace {

struct StepTrace {
  int layer = -1;
  float* out = nullptr;
  bool reuse_film = false;  // skip the timestep embedding, time MLP and FiLM projection
  bool serial_film = false; // every layer's FiLM modulation before the first layer
};

// Event before every launch (kernel profiling mode of fva_step_profile).  The
// events come from a pool owned by the handle and are recorded while the
// profiling graph is captured, so every replay re-records them between kernels.
struct StepProfile {
  std::vector<cudaEvent_t>* pool = nullptr;
  size_t used = 0;
  std::vector<int> kind, layer;
  cudaError_t err = cudaSuccess;
  void mark(int k, int l, cudaStream_t s) {
    if (used == pool->size()) {
      cudaEvent_t e;
      cudaError_t r = cudaEventCreate(&e);
      if (r != cudaSuccess) {
        err = r;
        return;
      }
      pool->push_back(e);
    }
    // an external record is captured as an event-record node that every replay re-records
    cudaError_t r = cudaEventRecordWithFlags((*pool)[used], s, cudaEventRecordExternal);
    if (r != cudaSuccess) {
      err = r;
      return;
    }
    ++used;
    kind.push_back(k);
    layer.push_back(l);
  }
};

fva_status enqueue_step(fva_handle* h, int B, float* buffer, float* out_chunk, bool use_fresh,
                        const StepTrace& tr, cudaStream_t s, StepProfile* prof = nullptr) {
  auto mark = [&](int kind, int layer) {
    if (prof) prof->mark(kind, layer, s);
  };
  StepDims d;
  d.B = B;
  d.Bmax = h->Bmax;
  d.K = h->K;
  d.H = h->H;
  d.T = h->T;
  d.A = h->A;
  d.W = h->W;
  d.nq = h->nq;
  d.dh = h->dh;
  d.Dq = h->Dq;
  d.F = h->F;
  d.L = h->L;
  d.S_cap = h->S_cap;
  d.N_mod = h->N_mod;
  d.eps = h->cfg.rms_eps;
  d.n_sms = h->n_sms;
  const int M = B * h->T, BK = B * h->K, W = h->W, F = h->F, Dq = h->Dq, L = h->L;
  const bool bf = h->bf16;
  const size_t a = h->act;
  const size_t kv_layer = (size_t)h->Bmax * h->S_cap * h->dh;  // elements per layer

  // trace bookkeeping: offsets (floats) of each traced tensor
  const size_t MW = (size_t)M * W;
  float* tp = tr.out;
  auto tr_at = [&](size_t off) { return tp + off; };
  const size_t o_hin = 0, o_y1 = o_hin + MW, o_q = o_y1 + MW, o_k = o_q + (size_t)M * Dq,
               o_v = o_k + (size_t)M * h->dh, o_att = o_v + (size_t)M * h->dh,
               o_hmid = o_att + (size_t)M * Dq, o_y2 = o_hmid + MW, o_mlp = o_y2 + MW,
               o_hout = o_mlp + (size_t)M * F, o_cond = o_hout + MW;
  auto copy_h = [&](size_t off) {
    return cudaMemcpyAsync(tr_at(off), h->h, MW * 4, cudaMemcpyDeviceToDevice, s);
  };


  // ---- this step's tau, dt, step index and padding counts from its ring slot (with
  // the timestep embeddings when the time MLP runs as the GEMV)
  const bool gemv = bf && BK <= 32;
  mark(FVA_K_PARAMS, -1);
  launch_fetch_params(h->params_host_dev, h->params_floats, FVA_PARAM_RING, h->ring_ctr,
                      h->params_dev, gemv && !tr.reuse_film ? h->temb : nullptr, BK, W,
                      h->temb_freq, s);
  CUDA_TRY(cudaGetLastError());
  h->fetch_enqueued = true;

  // ---- per-chunk FiLM condition and modulation (App. A.4); reused from the previous
  // step when the host saw identical noise levels (FVA_STEP_REUSE_FILM)
  // a projection with at least two tiles per SM and no K-split runs persistent, so
  // each tile's epilogue overlaps the next tile's MMAs
  auto gemm = [&](int bn, int mode, const CUtensorMap* ma, const CUtensorMap* mb,
                  const GemmEpi& e, int Mr, int N, int Kd, int splits) {
    const long long tiles = (long long)((Mr + 127) / 128) * (N / bn);
    if (h->persist_on && splits == 1 && h->n_sms > 0 && tiles >= 2LL * h->n_sms)
      return launch_tc_gemm_persist(bn, mode, ma, mb, e, Mr, N, Kd, h->n_sms, s);
    return launch_tc_gemm(bn, mode, ma, mb, e, Mr, N, Kd, splits, s);
  };
  // The FiLM modulation rides in the QKV and gate/up projections' launches (extra
  // CTAs of kFilmTile columns on the SMs they leave idle): a layer's columns are
  // [scale1 shift1 | gate1 scale2 shift2 | gate2] and its norms read them in that
  // order, the first pair in the norm before its QKV projection, the next three
  // after its attention, the last after its MLP.  So only layer 0's (scale1,
  // shift1) are computed before the first layer, and layer l's launches compute
  // the next 6W columns: its QKV launch at least (gate1, scale2, shift2) and as many
  // more as it has idle SMs for, its gate/up launch the rest (gate2 and layer l+1's
  // first pair, the last layer's the final norm's pair), each complete by stream
  // order before a norm reads it.  Needs the per-tile QKV form, at most 16
  // condition rows and W <= 1024; not when profiling kernel by kernel or tracing,
  // which keep the FiLM projection a kernel of its own.
  const int m_tiles_q = (M + 127) / 128;
  const int qkv_ctas = m_tiles_q * (h->N_qkv / h->bn_qkv);
  const int gu_ctas = m_tiles_q * (2 * F / h->bn_gu);
  const bool qkv_persist = h->persist_on && h->n_sms > 0 && qkv_ctas >= 2 * h->n_sms;
  const bool gu_persist = h->persist_on && h->n_sms > 0 && gu_ctas >= 2 * h->n_sms;
  const bool film_fold = bf && BK <= 16 && !tr.reuse_film && !tr.serial_film && !prof &&
                         tr.layer < 0 && !qkv_persist && W % kFilmTile == 0 && W <= 1024;
  const int film_group = 6 * W / kFilmTile;  // tiles computed by each layer's launches
  int film_gu = 0;                           // of which in the gate/up launch
  if (film_fold && !gu_persist) {
    const int film_q_min = 3 * W / kFilmTile;
    const int q = std::max(film_q_min, std::min(film_group, h->n_sms - qkv_ctas));
    film_gu = std::min(film_group - q, std::max(0, h->n_sms - gu_ctas));
  }
  const int film_q = film_group - film_gu;
  // FiLM columns [c0, c0 + n) as kFilmTile-wide tiles
  auto film_tiles = [&](int c0, int n) {
    FilmTiles ft{};
    ft.a = h->m_cond16;
    ft.b = h->m_wmod_q;
    ft.out = h->mod;
    ft.bias = h->b_mod;
    ft.ldo = h->N_mod;
    ft.rows = BK;
    ft.pre_stages = 4;
    ft.tile0 = c0 / kFilmTile;
    ft.tiles = n / kFilmTile;
    return ft;
  };
  GemmEpi ep{};
  ep.err = h->err_dev;
  if (!tr.reuse_film) {
    // a few rows (bf16): the parameter fetch wrote the timestep embeddings;
    // otherwise they are a kernel of their own
    if (!gemv) {
      mark(FVA_K_TIMESTEP_EMBED, -1);
      launch_temb(h->tau_dev(), h->temb_freq, BK, W, h->temb, bf, s);
    }
    if (bf) {
      // a few rows: one warp per output column (GEMV); more: the tensor-core GEMM
      // (the GEMV walks its rows 16 at a time)
      if (gemv) {
        mark(FVA_K_TIME_MLP, -1);
        launch_gemv_silu(h->temb, h->w_t1, h->b_t1, h->t1, BK, W, W, s);
        mark(FVA_K_TIME_MLP, -1);
        launch_gemv_silu(h->t1, h->w_t2, h->b_t2, h->cond, BK, W, W, s);
      } else {
        GemmEpi et{};
        et.err = h->err_dev;
        et.out = h->t1;
        et.bias = h->b_t1;
        et.ldo = W;
        mark(FVA_K_TIME_MLP, -1);
        CUDA_TRY(launch_tc_gemm(kBnTime, GEMM_BIAS_SILU_BF16, &h->m_temb, &h->m_wt1, et, BK, W, W, 1, s));
        et.out = h->cond;
        et.bias = h->b_t2;
        mark(FVA_K_TIME_MLP, -1);
        CUDA_TRY(launch_tc_gemm(kBnTime, GEMM_BIAS_SILU_BF16, &h->m_t1, &h->m_wt2, et, BK, W, W, 1, s));
      }
      ep.out = h->mod;
      ep.bias = h->b_mod;
      ep.ldo = h->N_mod;
      mark(FVA_K_FILM, -1);
      if (film_fold) {
        FilmTiles f0 = film_tiles(0, 2 * W);
        f0.pre_stages = W / 64;  // alone after the time MLP: every stage that fits
        CUDA_TRY(launch_tc_film_tiles(f0, W, h->err_dev, s));
      }
      else
        CUDA_TRY(BK <= 16 ? launch_tc_gemm_stream(&h->m_cond16, &h->m_wmod, ep, BK, h->N_mod, W,
                                                  2 * h->n_sms, s)
                           : gemm(kBnFilm, GEMM_BIAS_F32, &h->m_cond, &h->m_wmod, ep, BK,
                                  h->N_mod, W, 1));
    } else {
      launch_f32_gemm((float*)h->temb, W, (float*)h->w_t1, h->c32, W, BK, W, W, s);
      launch_f32_bias_act(h->c32, h->b_t1, (float*)h->t1, BK, W, true, s);
      launch_f32_gemm((float*)h->t1, W, (float*)h->w_t2, h->c32, W, BK, W, W, s);
      launch_f32_bias_act(h->c32, h->b_t2, (float*)h->cond, BK, W, true, s);
      launch_f32_gemm((float*)h->cond, W, (float*)h->w_mod, h->c32, h->N_mod, BK, h->N_mod, W, s);
      launch_f32_bias_act(h->c32, h->b_mod, h->mod, BK, h->N_mod, false, s);
    }
  }
  if (tr.layer >= 0) launch_to_f32(h->cond, bf, tr_at(o_cond), (long long)BK * W, s);

  // ---- action in-projection + layer 0 norm 1
  mark(FVA_K_EMBED_NORM, -1);
  launch_embed_norm(d, buffer, h->w_in_t, h->b_in, h->mod, h->h, h->y, bf, h->n_sms, s);

  const int m_tiles = (M + 127) / 128;
  const int sp_o = bf ? choose_splits(m_tiles * (W / kBnResid), Dq / 64) : 1;
  const int sp_d = bf ? choose_splits(m_tiles * (W / kBnResid), F / 64) : 1;
  const long long pstride = (long long)M * W;

  for (int l = 0; l < L; ++l) {
    const LayerW& lw = h->layers[l];
    void* kc_l = (uint8_t*)h->kc + (size_t)l * kv_layer * a;
    void* vc_l = (uint8_t*)h->vc + (size_t)l * kv_layer * a;
    const bool trace = tr.layer == l;
    if (trace) {
      CUDA_TRY(copy_h(o_hin));
      launch_to_f32(h->y, bf, tr_at(o_y1), (long long)MW, s);
    }
    // QKV projection + RoPE + KV append
    if (bf) {
      ep = GemmEpi{};
      ep.err = h->err_dev;
      ep.q = h->q;
      ep.kc = kc_l;
      ep.vc = vc_l;
      ep.prefix_len = h->prefix_len_dev;
      ep.rope = h->rope;
      ep.rope_h = h->rope_h;
      ep.T = h->T;
      ep.S_cap = h->S_cap;
      ep.nq = h->nq;
      ep.dh = h->dh;
      // this layer's FiLM modulation rows (scale, shift, gate of both norms, 6W
      // floats per chunk), written at the start of the step and long evicted from
      // L2 by the weights streamed since: L2 fetches them while the QKV projection
      // runs, ahead of the layer's two residual + norm kernels
      ep.pf_base = h->mod + mod_off(l, 0, W);
      ep.pf_count = BK;
      ep.pf_bytes = 6 * W * (int)sizeof(float);
      ep.pf_stride = h->N_mod;
      mark(FVA_K_QKV, l);
      ep.a_rows = h->y_box;
      if (film_fold) {
        CUDA_TRY(launch_tc_gemm_film(h->bn_qkv, GEMM_QKV_ROPE, h->y_box ? &h->m_ybox : &h->m_y,
                                     &lw.m_qkv, ep, M, h->N_qkv, W,
                                     film_tiles(6 * W * l + 2 * W, film_q * kFilmTile), s));
      } else {
        CUDA_TRY(gemm(h->bn_qkv, GEMM_QKV_ROPE, h->y_box ? &h->m_ybox : &h->m_y, &lw.m_qkv, ep,
                      M, h->N_qkv, W, 1));
      }
    } else {
      launch_f32_gemm((float*)h->y, W, (float*)lw.w_qkv, h->c32, h->N_qkv, M, h->N_qkv, W, s);
      launch_f32_qkv_rope(h->c32, (float*)h->q, (float*)kc_l, (float*)vc_l, h->prefix_len_dev,
                          h->rope, M, h->T, h->S_cap, h->nq, h->dh, s);
    }
    if (trace) {
      launch_to_f32(h->q, bf, tr_at(o_q), (long long)M * Dq, s);
      launch_gather_action_kv(kc_l, bf, h->prefix_len_dev, B, h->T, h->S_cap, h->dh, tr_at(o_k), s);
      launch_gather_action_kv(vc_l, bf, h->prefix_len_dev, B, h->T, h->S_cap, h->dh, tr_at(o_v), s);
    }
    // chunk-causal attention
    if (bf) {
      AttnArgs aa{};
      aa.prefix_len = h->prefix_len_dev;
      aa.out = h->attn;
      aa.part_o = h->att_part_o;
      aa.part_ml = h->att_part_ml;
      aa.T = h->T;
      aa.H = h->H;
      aa.nq = h->nq;
      aa.S_cap = h->S_cap;
      aa.tiles_per_req = h->tiles_per_req;
      aa.max_splits = h->attn_ncl > 0 ? h->attn_ncl : h->attn_max_splits;
      aa.blocks_per_split = h->attn_bps;
      aa.kv_row0 = l * h->Bmax * h->S_cap;
      aa.scale_log2 = 1.4426950408889634f / std::sqrt((float)h->dh);
      aa.err = h->err_dev;
      aa.pad_tokens = h->pad_dev();
      aa.block_diag = (h->cfg.flags & FVA_FLAG_BLOCK_DIAGONAL) ? 1 : 0;
      aa.prefix_src = h->prefix_src_dev;
      mark(FVA_K_ATTENTION, l);
      CUDA_TRY(launch_tc_attention(&h->m_q, &h->m_k, &h->m_v, aa, B, s, h->attn_ncl > 0));
      if (aa.max_splits > 1 && h->attn_ncl == 0) {
        mark(FVA_K_ATTN_MERGE, l);
        CUDA_TRY(launch_attn_merge(aa, B, s));
      }
    } else {
      launch_f32_attention((float*)h->q, (float*)kc_l, (float*)vc_l, h->prefix_len_dev,
                           h->pad_dev(), (h->cfg.flags & FVA_FLAG_BLOCK_DIAGONAL) ? 1 : 0,
                           h->prefix_src_dev, (float*)h->attn, B, h->T, h->H, h->nq, h->dh, h->S_cap, h->S_cap, s);
    }
    if (trace) launch_to_f32(h->attn, bf, tr_at(o_att), (long long)M * Dq, s);
    // output projection (split-K partials) -> gated residual + norm 2
    if (bf) {
      ep = GemmEpi{};
      ep.err = h->err_dev;
      ep.out = h->part;
      ep.ldo = W;
      ep.split_stride = pstride;
      mark(FVA_K_OUT_PROJ, l);
      CUDA_TRY(gemm(kBnResid, GEMM_PARTIAL_BF16, &h->m_attn, &lw.m_o, ep, M, W, Dq, sp_o));
    } else {
      launch_f32_gemm((float*)h->attn, Dq, (float*)lw.w_o, h->part, W, M, W, Dq, s);
    }
    mark(FVA_K_RESID_NORM, l);
    launch_resid_norm(d, h->h, h->part, bf, sp_o, pstride, h->mod, mod_off(l, 2, W),
                      mod_off(l, 3, W), mod_off(l, 4, W), h->y, bf, s);
    if (trace) {
      CUDA_TRY(copy_h(o_hmid));
      launch_to_f32(h->y, bf, tr_at(o_y2), (long long)MW, s);
    }
    // gated MLP
    if (bf) {
      ep = GemmEpi{};
      ep.err = h->err_dev;
      ep.out = h->mlp;
      ep.ldo = F;
      mark(FVA_K_GATE_UP, l);
      ep.a_rows = h->y_box;
      if (film_fold && film_gu > 0)
        CUDA_TRY(launch_tc_gemm_film(
            h->bn_gu, GEMM_GEGLU, h->y_box ? &h->m_ybox : &h->m_y, &lw.m_gu, ep, M, 2 * F, W,
            film_tiles(6 * W * l + 2 * W + film_q * kFilmTile, film_gu * kFilmTile), s));
      else
        CUDA_TRY(gemm(h->bn_gu, GEMM_GEGLU, h->y_box ? &h->m_ybox : &h->m_y, &lw.m_gu, ep, M,
                      2 * F, W, 1));
      ep.a_rows = 0;
      ep.out = h->part;
      ep.ldo = W;
      ep.split_stride = pstride;
      mark(FVA_K_DOWN, l);
      CUDA_TRY(gemm(kBnResid, GEMM_PARTIAL_BF16, &h->m_mlp, &lw.m_d, ep, M, W, F, sp_d));
    } else {
      launch_f32_gemm((float*)h->y, W, (float*)lw.w_gu, h->c32, 2 * F, M, 2 * F, W, s);
      launch_f32_geglu(h->c32, (float*)h->mlp, M, F, s);
      launch_f32_gemm((float*)h->mlp, F, (float*)lw.w_d, h->part, W, M, W, F, s);
    }
    if (trace) launch_to_f32(h->mlp, bf, tr_at(o_mlp), (long long)M * F, s);
    if (l + 1 < L) {
      mark(FVA_K_RESID_NORM, l);
      launch_resid_norm(d, h->h, h->part, bf, sp_d, pstride, h->mod, mod_off(l, 5, W),
                        mod_off(l + 1, 0, W), mod_off(l + 1, 1, W), h->y, bf, s);
      if (trace) CUDA_TRY(copy_h(o_hout));
    }
  }
  // ---- final norm, out-projection, Euler update, emit, roll, tail
  {
    mark(FVA_K_FINAL, -1);
    launch_final_norm(d, h->h, h->part, bf, sp_d, pstride, h->mod, h->yF, s);
  }
  mark(FVA_K_VELOCITY, -1);
  launch_velocity_euler(d, h->yF, h->w_out_t, h->b_out, h->dt_dev(), buffer, out_chunk, h->vel,
                        use_fresh ? h->fresh : nullptr, h->cfg.noise_seed, h->step_dev(), s);
  if (tr.layer == L - 1) CUDA_TRY(copy_h(o_hout));
  mark(FVA_K_COUNT, -1);
  CUDA_TRY(cudaGetLastError());
  if (prof && prof->err != cudaSuccess)
    return fail(FVA_ERR_CUDA, "profiling event failed: %s", cudaGetErrorString(prof->err));
  return FVA_OK;
}

// Reports the device error word once it has been read back, and clears it so that
// the calls after the reported one run normally.  `s` is the calling step's stream.
fva_status check_async_error(fva_handle* h, cudaStream_t s) {
  if (h->err_pending && cudaEventQuery(h->err_ev) == cudaSuccess) {
    h->err_pending = false;
    const int code = *h->err_host;
    if (code != 0) {
      *h->err_host = 0;
      CUDA_TRY(cudaMemsetAsync(h->err_dev, 0, sizeof(int), s));
    }
    if (code == 4 /* KERR_BAD_SHAPE */)
      return fail(FVA_ERR_INVALID_ARG, "an earlier kernel saw a device size beyond its bound");
    if (code != 0)
      return fail(FVA_ERR_TIMEOUT, "a kernel of an earlier step gave up a bounded wait (code %d)",
                  code);
  }
  cudaError_t e = cudaPeekAtLastError();
  if (e != cudaSuccess && e != cudaErrorNotReady) {
    cudaGetLastError();
    return fail(FVA_ERR_CUDA, "earlier CUDA error: %s", cudaGetErrorString(e));
  }
  return FVA_OK;
}

// The step using ring slot `slot` is queued (its parameter fetch with it): the slot
// may be written again once the stream has passed this point.
void advance_ring(fva_handle* h, int slot, cudaStream_t s) {
  h->ring_pos = (h->ring_pos + 1) % FVA_PARAM_RING;
  if (cudaEventRecord(h->ring_ev[slot], s) == cudaSuccess) {
    h->ring_used[slot] = true;
  } else {
    cudaGetLastError();
    cudaStreamSynchronize(s);  // no event: the slot is free once the stream is idle
    cudaGetLastError();
    h->ring_used[slot] = false;
  }
}

fva_status get_graph(fva_handle* h, int B, float* buffer, float* out, bool fresh, bool reuse_film,
                     bool serial_film, cudaGraphExec_t* exec) {
  for (auto& g : h->graphs)
    if (g.batch == B && g.buffer == buffer && g.out == out && g.fresh == fresh &&
        g.reuse_film == reuse_film && g.serial_film == serial_film) {
      g.last_use = ++h->use_clock;
      *exec = g.exec;
      return FVA_OK;
    }
  if (h->graphs.size() >= 8) {
    auto it = std::min_element(h->graphs.begin(), h->graphs.end(),
                               [](const GraphEntry& x, const GraphEntry& y) {
                                 return x.last_use < y.last_use;
                               });
    cudaGraphExecDestroy(it->exec);
    h->graphs.erase(it);
  }
  cudaGraph_t graph;
  CUDA_TRY(cudaStreamBeginCapture(h->cap_stream, cudaStreamCaptureModeThreadLocal));
  StepTrace tr;
  tr.reuse_film = reuse_film;
  tr.serial_film = serial_film;
  fva_status st = enqueue_step(h, B, buffer, out, fresh, tr, h->cap_stream);
  cudaError_t e = cudaStreamEndCapture(h->cap_stream, &graph);
  if (st != FVA_OK) {
    if (e == cudaSuccess) cudaGraphDestroy(graph);
    return st;
  }
  CUDA_TRY(e);
  cudaGraphExec_t ge;
  e = cudaGraphInstantiate(&ge, graph, 0);
  cudaGraphDestroy(graph);
  CUDA_TRY(e);
  h->graphs.push_back(GraphEntry{B, buffer, out, fresh, reuse_film, serial_film, ge,
                                 ++h->use_clock});
  *exec = ge;
  return FVA_OK;
}

}  // namespace

extern "C" int64_t fva_trace_floats(const fva_handle* h, int32_t batch) {
  if (!h || batch < 1 || batch > h->Bmax) return 0;
  const int64_t M = (int64_t)batch * h->T;
  return M * (5LL * h->W + 2LL * h->Dq + 2LL * h->dh + h->F) + (int64_t)batch * h->K * h->W;
}

// A pointer the step's kernels dereference: device memory of the handle's device, or
// pinned host memory mapped at the same address (the kernels then read and write it
// over the host link).  Pageable host memory is refused before any launch.
static fva_status check_step_ptr(fva_handle* h, const void* p, const char* what) {
  cudaPointerAttributes at{};
  cudaError_t e = cudaPointerGetAttributes(&at, p);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(FVA_ERR_INVALID_ARG, "%s: cudaPointerGetAttributes failed: %s", what,
                cudaGetErrorString(e));
  }
  const bool device = (at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged) &&
                      at.device == h->device;
  const bool mapped_host = at.type == cudaMemoryTypeHost && at.devicePointer == p;
  if (!device && !mapped_host)
    return fail(FVA_ERR_INVALID_ARG,
                "%s must be memory of device %d or pinned host memory mapped at the same "
                "address (cudaHostAlloc / cudaHostRegister), not pageable host memory",
                what, h->device);
  return FVA_OK;
}

static fva_status step_impl(fva_handle* h, float* buffer, const float* noise_levels,
                            float* out_chunk, int32_t batch, const fva_step_opts* opts,
                            fva_stream stream, StepProfile* prof) {
  if (!h) return fail(FVA_ERR_INVALID_ARG, "handle is NULL");
  if (!buffer || !noise_levels || !out_chunk)
    return fail(FVA_ERR_INVALID_ARG, "buffer, noise_levels and out_chunk must be non-NULL");
  if (batch < 1 || batch > h->Bmax)
    return fail(FVA_ERR_INVALID_ARG, "batch %d outside [1, %d]", batch, h->Bmax);
  if (opts && opts->trace_layer >= h->L)
    return fail(FVA_ERR_INVALID_ARG, "trace_layer %d >= n_layers", opts->trace_layer);
  if (opts && opts->trace_layer >= 0 && !opts->trace_out)
    return fail(FVA_ERR_INVALID_ARG, "trace_out is NULL");
  if (opts && (opts->flags & ~(FVA_STEP_REUSE_FILM | FVA_STEP_SERIAL_FILM)))
    return fail(FVA_ERR_INVALID_ARG, "unknown step flags 0x%x", opts->flags);
  if (opts && opts->n_valid)
    for (int r = 0; r < batch; ++r)
      if (opts->n_valid[r] < 1 || opts->n_valid[r] > h->K)
        return fail(FVA_ERR_INVALID_ARG, "n_valid[%d] = %d outside [1, %d]", r,
                    opts->n_valid[r], h->K);
  for (int r = 0; r < batch; ++r) {
    float prev = 0.f;
    for (int k = 0; k < h->K; ++k) {
      const float t = noise_levels[(size_t)r * h->K + k];
      if (!(t > prev) || !(t <= 1.f))
        return fail(FVA_ERR_INVALID_ARG,
                    "noise_levels[%d][%d] = %g: need 0 < tau_1 < ... < tau_K <= 1", r, k, t);
      prev = t;
    }
  }
  if (!h->weights_loaded) return fail(FVA_ERR_STATE, "weights are not loaded");
  for (int r = 0; r < batch; ++r) {
    const int l0 = h->layer_len[(size_t)r * h->L];
    for (int l = 0; l < h->L; ++l) {
      const int v = h->layer_len[(size_t)r * h->L + l];
      if (v < 0) return fail(FVA_ERR_STATE, "request %d has no prefix K/V for layer %d", r, l);
      if (v != l0)
        return fail(FVA_ERR_STATE, "request %d: prefix length differs across layers", r);
    }
  }
  DeviceGuard guard(h->device);
  fva_status st;
  if ((st = check_step_ptr(h, buffer, "buffer")) != FVA_OK ||
      (st = check_step_ptr(h, out_chunk, "out_chunk")) != FVA_OK ||
      (opts && opts->trace_layer >= 0 &&
       (st = check_step_ptr(h, opts->trace_out, "trace_out")) != FVA_OK))
    return st;
  cudaStream_t s = (cudaStream_t)stream;
  st = check_async_error(h, s);
  if (st != FVA_OK) return st;

  // stage tau, dt and the step index in the next slot of the pinned ring; the
  // step's first kernel reads that slot (its device-side counter follows the host's
  // ring position: both advance once per queued step)
  const int slot = h->ring_pos;
  if (h->ring_used[slot]) CUDA_TRY(cudaEventSynchronize(h->ring_ev[slot]));
  float* ph = h->params_host + (size_t)slot * h->params_floats;
  for (int r = 0; r < batch; ++r)
    for (int k = 0; k < h->K; ++k) {
      const size_t i = (size_t)r * h->K + k;
      const float t = noise_levels[i];
      const float prev = k ? noise_levels[i - 1] : 0.f;
      ph[i] = t;
      ph[h->BKmax + i] = prev - t;  // fp32 dt_k = tau_{k-1} - tau_k
    }
  const unsigned long long step = h->step_index++;
  std::memcpy(ph + 2 * h->BKmax, &step, sizeof(step));
  int* pad = reinterpret_cast<int*>(ph + 2 * h->BKmax + 2);
  for (int r = 0; r < h->Bmax; ++r)
    pad[r] = (opts && opts->n_valid && r < batch) ? (h->K - opts->n_valid[r]) * h->H : 0;

  const bool fresh = opts && opts->fresh_noise;
  const bool serial_film = opts && (opts->flags & FVA_STEP_SERIAL_FILM);
  // the previous step's FiLM modulation is reused only for the same batch and
  // bit-identical noise levels
  const size_t n_tau = (size_t)batch * h->K;
  const bool reuse_film = opts && (opts->flags & FVA_STEP_REUSE_FILM) && !prof && h->film_valid &&
                          h->film_batch == batch && h->film_tau.size() == n_tau &&
                          std::memcmp(h->film_tau.data(), noise_levels, n_tau * sizeof(float)) == 0;
  if (fresh)
    CUDA_TRY(cudaMemcpyAsync(h->fresh, opts->fresh_noise,
                             sizeof(float) * batch * h->H * h->A, cudaMemcpyDeviceToDevice, s));
  if (prof) {
    if (!h->prof_exec || h->prof_batch != batch || h->prof_buf != buffer ||
        h->prof_out != out_chunk) {
      if (h->prof_exec) cudaGraphExecDestroy(h->prof_exec);
      h->prof_exec = nullptr;
      prof->pool = &h->prof_events;
      cudaGraph_t graph;
      CUDA_TRY(cudaStreamBeginCapture(h->cap_stream, cudaStreamCaptureModeThreadLocal));
      st = enqueue_step(h, batch, buffer, out_chunk, fresh, StepTrace{}, h->cap_stream, prof);
      cudaError_t e = cudaStreamEndCapture(h->cap_stream, &graph);
      if (st != FVA_OK) {
        if (e == cudaSuccess) cudaGraphDestroy(graph);
        return st;
      }
      CUDA_TRY(e);
      e = cudaGraphInstantiate(&h->prof_exec, graph, 0);
      cudaGraphDestroy(graph);
      CUDA_TRY(e);
      h->prof_batch = batch;
      h->prof_buf = buffer;
      h->prof_out = out_chunk;
      h->prof_kind = prof->kind;
      h->prof_layer = prof->layer;
    }
    prof->pool = &h->prof_events;
    prof->used = h->prof_kind.size();
    prof->kind = h->prof_kind;
    prof->layer = h->prof_layer;
    CUDA_TRY(cudaGraphLaunch(h->prof_exec, s));
    advance_ring(h, slot, s);
  } else if ((opts && opts->trace_layer >= 0) || (h->cfg.flags & FVA_FLAG_NO_GRAPH)) {
    StepTrace tr;
    tr.reuse_film = reuse_film;
    tr.serial_film = serial_film;
    if (opts && opts->trace_layer >= 0) {
      tr.layer = opts->trace_layer;
      tr.out = opts->trace_out;
    }
    h->fetch_enqueued = false;
    st = enqueue_step(h, batch, buffer, out_chunk, fresh, tr, s);
    if (h->fetch_enqueued) advance_ring(h, slot, s);
    if (st != FVA_OK) return st;
  } else {
    cudaGraphExec_t exec;
    if ((st = get_graph(h, batch, buffer, out_chunk, fresh, reuse_film, serial_film, &exec)) !=
        FVA_OK)
      return st;
    CUDA_TRY(cudaGraphLaunch(exec, s));
    advance_ring(h, slot, s);
  }
  if (!reuse_film) {
    h->film_valid = true;
    h->film_batch = batch;
    h->film_tau.assign(noise_levels, noise_levels + n_tau);
  }
  if (opts && opts->velocity_out)
    CUDA_TRY(cudaMemcpyAsync(opts->velocity_out, h->vel,
                             sizeof(float) * batch * h->T * h->A, cudaMemcpyDeviceToDevice, s));
  if (!h->err_pending && (h->polls++ % 16) == 0) {
    CUDA_TRY(cudaMemcpyAsync(h->err_host, h->err_dev, sizeof(int), cudaMemcpyDeviceToHost, s));
    CUDA_TRY(cudaEventRecord(h->err_ev, s));
    h->err_pending = true;
  }
  return FVA_OK;
}

extern "C" fva_status fva_step_ex(fva_handle* h, float* buffer, const float* noise_levels,
                                  float* out_chunk, int32_t batch, const fva_step_opts* opts,
                                  fva_stream stream) {
  return step_impl(h, buffer, noise_levels, out_chunk, batch, opts, stream, nullptr);
}

extern "C" fva_status fva_step(fva_handle* h, float* buffer, const float* noise_levels,
                               float* out_chunk, int32_t batch, fva_stream stream) {
  return step_impl(h, buffer, noise_levels, out_chunk, batch, nullptr, stream, nullptr);
}

extern "C" fva_status fva_step_profile(fva_handle* h, float* buffer, const float* noise_levels,
                                       float* out_chunk, int32_t batch, fva_kernel_time* records,
                                       int32_t max_records, int32_t* n_records,
                                       fva_stream stream) {
  if (!records || !n_records) return fail(FVA_ERR_INVALID_ARG, "records / n_records is NULL");
  *n_records = 0;
  if (h) {
    const int needed = 6 + 8 * h->L;
    if (max_records < needed)
      return fail(FVA_ERR_INVALID_ARG, "max_records %d < %d launches", max_records, needed);
  }
  StepProfile prof;
  fva_status st = step_impl(h, buffer, noise_levels, out_chunk, batch, nullptr, stream, &prof);
  if (st != FVA_OK) return st;
  DeviceGuard guard(h->device);
  CUDA_TRY(cudaStreamSynchronize((cudaStream_t)stream));
  const int n = (int)prof.used - 1;
  if (n > max_records) return fail(FVA_ERR_INVALID_ARG, "max_records %d < %d", max_records, n);
  for (int i = 0; i < n; ++i) {
    float ms = 0.f;
    CUDA_TRY(cudaEventElapsedTime(&ms, h->prof_events[i], h->prof_events[i + 1]));
    records[i].kind = prof.kind[i];
    records[i].layer = prof.layer[i];
    records[i].microseconds = ms * 1000.f;
  }
  *n_records = n;
  return FVA_OK;
}

extern "C" fva_status fva_set_step_index(fva_handle* h, uint64_t step) {
  if (!h) return fail(FVA_ERR_INVALID_ARG, "handle is NULL");
  h->step_index = step;
  return FVA_OK;
}

extern "C" fva_status fva_get_step_index(const fva_handle* h, uint64_t* step) {
  if (!h || !step) return fail(FVA_ERR_INVALID_ARG, "NULL argument");
  *step = h->step_index;
  return FVA_OK;
}

extern "C" fva_status fva_mask_table(fva_handle* h, int32_t batch, int32_t* key_limit,
                                     fva_stream stream) {
  if (!h || !key_limit) return fail(FVA_ERR_INVALID_ARG, "NULL argument");
  if (batch < 1 || batch > h->Bmax)
    return fail(FVA_ERR_INVALID_ARG, "batch %d outside [1, %d]", batch, h->Bmax);
  DeviceGuard guard(h->device);
  launch_mask_table(h->prefix_len_dev, batch, h->T, h->H, key_limit, (cudaStream_t)stream);
  CUDA_TRY(cudaGetLastError());
  return FVA_OK;
}

extern "C" fva_status fva_geglu_gelu(const float* x, float* y, int64_t n, fva_stream stream) {
  if (n < 0 || (n > 0 && (!x || !y))) return fail(FVA_ERR_INVALID_ARG, "bad x / y / n");
  launch_geglu_gelu(x, y, n, (cudaStream_t)stream);
  CUDA_TRY(cudaGetLastError());
  return FVA_OK;
}

// =============================================================================
// bounded-wait check
// =============================================================================
namespace {
// One thread waits on an mbarrier that nothing arrives at, with a wall-clock limit
// of limit_ns: when the limit passes it records KERR_WAIT_SYNC in *err and returns,
// the same path every bounded wait of the library's kernels takes.
__global__ void stall_kernel(int* err, unsigned long long limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  fence_barrier_init();
  mbar_wait_ns(&bar, 0, err, KERR_WAIT_SYNC, limit_ns);
}
}  // namespace

extern "C" fva_status fva_check_bounded_wait(fva_handle* h, int32_t limit_us, fva_stream stream) {
  if (!h) return fail(FVA_ERR_INVALID_ARG, "handle is NULL");
  if (limit_us < 1 || limit_us > 1000000)
    return fail(FVA_ERR_INVALID_ARG, "limit_us %d outside [1, 1000000]", limit_us);
  DeviceGuard guard(h->device);
  cudaStream_t s = (cudaStream_t)stream;
  stall_kernel<<<1, 32, 0, s>>>(h->err_dev, (unsigned long long)limit_us * 1000ull);
  CUDA_TRY(cudaGetLastError());
  // read the error word back behind it (replacing any read-back still pending: this
  // one also sees what an earlier one would), so the next call reports it once the
  // stream has passed this point
  CUDA_TRY(cudaMemcpyAsync(h->err_host, h->err_dev, sizeof(int), cudaMemcpyDeviceToHost, s));
  CUDA_TRY(cudaEventRecord(h->err_ev, s));
  h->err_pending = true;
  return FVA_OK;
}

// =============================================================================
// isolated chunk-causal attention on caller buffers
// =============================================================================
extern "C" fva_status fva_chunk_attention(fva_handle* h, const void* q, const void* k,
                                          const void* v, const int32_t* prefix_len,
                                          int32_t batch, int32_t kv_rows, void* out,
                                          fva_stream stream) {
  if (!h || !q || !k || !v || !prefix_len || !out) return fail(FVA_ERR_INVALID_ARG, "NULL argument");
  if (!h->bf16) return fail(FVA_ERR_UNSUPPORTED, "fva_chunk_attention needs a bf16 handle");
  if (batch < 1 || batch > h->Bmax)
    return fail(FVA_ERR_INVALID_ARG, "batch %d outside [1, %d]", batch, h->Bmax);
  if (kv_rows < h->T || kv_rows > h->S_cap)
    return fail(FVA_ERR_INVALID_ARG, "kv_rows %d outside [K*H, max_prefix + K*H] = [%d, %d]",
                kv_rows, h->T, h->S_cap);
  for (const void* p : {q, k, v, (const void*)out})
    if (reinterpret_cast<uintptr_t>(p) % 16)
      return fail(FVA_ERR_INVALID_ARG, "q, k, v and out must be 16-byte aligned");
  DeviceGuard guard(h->device);
  fva_status st;
  CUtensorMap mq, mk, mv;
  if ((st = make_map(&mq, q, (uint64_t)batch * h->T * h->nq, h->dh, 128)) ||
      (st = make_map(&mk, k, (uint64_t)batch * kv_rows, h->dh, 64)) ||
      (st = make_map(&mv, v, (uint64_t)batch * kv_rows, h->dh, 64)))
    return st;
  AttnArgs aa{};
  aa.prefix_len = prefix_len;
  aa.out = out;
  aa.part_o = h->att_part_o;
  aa.part_ml = h->att_part_ml;
  aa.T = h->T;
  aa.H = h->H;
  aa.nq = h->nq;
  aa.S_cap = kv_rows;
  aa.tiles_per_req = h->tiles_per_req;
  aa.max_splits = (kv_rows + kAttnKeysPerSplit - 1) / kAttnKeysPerSplit;
  aa.blocks_per_split = kAttnKeysPerSplit / kAttnKeyBlock;
  aa.kv_row0 = 0;
  aa.scale_log2 = 1.4426950408889634f / std::sqrt((float)h->dh);
  aa.err = h->err_dev;
  const int ncl = attn_cluster_size(h, (long long)batch * h->tiles_per_req, (kv_rows + 63) / 64,
                                    aa.blocks_per_split);
  const bool cluster = ncl > 0;
  if (cluster) aa.max_splits = ncl;
  CUDA_TRY(launch_tc_attention(&mq, &mk, &mv, aa, batch, (cudaStream_t)stream, cluster));
  if (!cluster) CUDA_TRY(launch_attn_merge(aa, batch, (cudaStream_t)stream));
  return FVA_OK;
}
