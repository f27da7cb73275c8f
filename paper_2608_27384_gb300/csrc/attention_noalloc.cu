// fva_chunk_attention_noalloc: the chunk-causal attention of fva_chunk_attention for
// callers that must not allocate device memory.
//
// Who needs it: a robot-side controller runs the decoder inside a fixed-period
// control loop, and cudaMalloc / cudaFree may synchronise the whole device and
// take an unbounded time, which such a loop cannot afford; other hosts hand all
// device memory to their own pool at start-up, so any allocation a library makes
// later fails.  This entry point needs no handle (fva_create allocates) and calls
// no allocating routine: the attention's split-KV scratch lives in a fixed
// file-scope device array instead.
//
// The array is kNoAllocSlots partial tiles (128 rows x 256 bf16 each, plus their
// row max / sum as fp32 pairs): 16 MiB + 256 KiB, held by every GPU that loads
// libfva until the process exits.  A call needs batch * ceil(K*H*nq / 128) * ceil(kv_rows / 256)
// slots; larger calls are rejected.
#include <cudaTypedefs.h>

#include <cstdio>
#include <mutex>

#include "common.cuh"
#include "fva.h"
#include "kernels.h"

namespace fva {
namespace {

constexpr int kNoAllocSlots = 256;
constexpr int kRowsPerSlot = 128;
constexpr int kDH = 256;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) bf16 g_part_o[(size_t)kNoAllocSlots * kRowsPerSlot * kDH];
static __device__ __align__(256) float2 g_part_ml[(size_t)kNoAllocSlots * kRowsPerSlot];

struct DeviceScratch {
  std::once_flag once;
  cudaError_t status = cudaErrorNotReady;
  bf16* part_o = nullptr;
  float2* part_ml = nullptr;
};
DeviceScratch g_dev[kMaxDevices];
std::once_flag g_encoder_once;
PFN_cuTensorMapEncodeTiled_v12000 g_encode_fn = nullptr;

fva_status set_error(fva_status st, const char* msg) {
  set_last_error(msg);
  return st;
}

// Device addresses of the scratch arrays, looked up once per device with that
// device current (host code cannot use the array names as device addresses).
void init_device(DeviceScratch& d) {
  d.status = cudaGetSymbolAddress((void**)&d.part_o, g_part_o);
  if (d.status == cudaSuccess) d.status = cudaGetSymbolAddress((void**)&d.part_ml, g_part_ml);
  if (d.status == cudaSuccess) d.status = tc_attention_init();
}

bool encode(CUtensorMap* m, const void* ptr, uint64_t rows, uint32_t box_rows) {
  cuuint64_t dims[2] = {kDH, rows};
  cuuint64_t strides[1] = {kDH * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return g_encode_fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides,
                     box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace
}  // namespace fva

using namespace fva;

extern "C" fva_status fva_chunk_attention_noalloc(const void* q, const void* k, const void* v,
                                                  const int32_t* prefix_len, int32_t batch,
                                                  int32_t n_chunks, int32_t chunk_tokens,
                                                  int32_t n_q_heads, int32_t head_dim,
                                                  int32_t kv_rows, void* out,
                                                  fva_stream stream) {
  if (!q || !k || !v || !prefix_len || !out) return set_error(FVA_ERR_INVALID_ARG, "NULL argument");
  if (head_dim != kDH) return set_error(FVA_ERR_UNSUPPORTED, "head_dim must be 256");
  if (n_q_heads < 1 || n_q_heads > 16 || 128 % n_q_heads)
    return set_error(FVA_ERR_UNSUPPORTED, "n_q_heads must be 1, 2, 4, 8 or 16");
  if (batch < 1 || n_chunks < 1 || chunk_tokens < 1)
    return set_error(FVA_ERR_INVALID_ARG, "batch, n_chunks and chunk_tokens must be positive");
  const long long T = (long long)n_chunks * chunk_tokens;
  if (kv_rows < T || T * n_q_heads * batch >= (1LL << 31) || (long long)batch * kv_rows >= (1LL << 31))
    return set_error(FVA_ERR_INVALID_ARG, "kv_rows below K*H or sizes beyond 2^31 rows");
  for (const void* p : {q, k, v, (const void*)out})
    if (reinterpret_cast<uintptr_t>(p) % 16)
      return set_error(FVA_ERR_INVALID_ARG, "q, k, v and out must be 16-byte aligned");
  const long long tiles = (T * n_q_heads + 127) / 128;
  const long long splits = (kv_rows + kAttnKeysPerSplit - 1) / kAttnKeysPerSplit;
  if (splits > 32 || batch * tiles * splits > kNoAllocSlots)
    return set_error(FVA_ERR_INVALID_ARG,
                     "call needs more than the 256 fixed scratch slots "
                     "(batch * ceil(K*H*nq/128) * ceil(kv_rows/256))");
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    cudaGetLastError();
    return set_error(FVA_ERR_CUDA, "no usable current CUDA device");
  }
  DeviceScratch& ds = g_dev[dev];
  std::call_once(ds.once, [&ds] { init_device(ds); });
  if (ds.status != cudaSuccess)
    return set_error(FVA_ERR_CUDA, "looking up the fixed scratch on this device failed");
  std::call_once(g_encoder_once, [] {
    cudaDriverEntryPointQueryResult res;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &res) == cudaSuccess &&
        res == cudaDriverEntryPointSuccess)
      g_encode_fn = (PFN_cuTensorMapEncodeTiled_v12000)fn;
  });
  if (!g_encode_fn) return set_error(FVA_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
  CUtensorMap mq, mk, mv;
  if (!encode(&mq, q, (uint64_t)batch * T * n_q_heads, 128) ||
      !encode(&mk, k, (uint64_t)batch * kv_rows, 64) || !encode(&mv, v, (uint64_t)batch * kv_rows, 64))
    return set_error(FVA_ERR_CUDA, "tensor map encoding failed");
  AttnArgs a{};
  a.prefix_len = prefix_len;
  a.out = out;
  a.part_o = ds.part_o;
  a.part_ml = ds.part_ml;
  a.T = (int)T;
  a.H = chunk_tokens;
  a.nq = n_q_heads;
  a.S_cap = kv_rows;
  a.tiles_per_req = (int)tiles;
  a.blocks_per_split = kAttnKeysPerSplit / kAttnKeyBlock;
  a.max_splits = (int)splits;
  a.kv_row0 = 0;
  a.scale_log2 = 1.4426950408889634f / 16.0f;  // log2(e) / sqrt(256)
  a.err = nullptr;
  cudaError_t e = launch_tc_attention(&mq, &mk, &mv, a, batch, (cudaStream_t)stream, false);
  if (e == cudaSuccess) e = launch_attn_merge(a, batch, (cudaStream_t)stream);
  if (e != cudaSuccess) return set_error(FVA_ERR_CUDA, cudaGetErrorString(e));
  return FVA_OK;
}
