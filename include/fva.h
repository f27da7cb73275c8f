/*
 * fva.h -- C ABI of the FlashVLA streaming action-decode library (libfva.so).
 *
 * FlashVLA (arXiv 2608.27384) decodes robot action chunks as a stream: a buffer of
 * K action chunks, each H tokens of A action dimensions, holds the chunks at
 * staggered noise levels tau_1 < ... < tau_K (§3.1, Eq. 2).  One forward pass of the
 * flow-matching action expert, under a chunk-wise causal mask (§3.1), yields a
 * velocity for every chunk; every chunk takes one Euler step toward its
 * front neighbour's level (Eq. 1), the head chunk -- now clean -- is emitted as
 * the executable action chunk, the others shift forward and fresh N(0, I) noise
 * is pushed at the tail (§3.2, Algorithm 1, steady streaming).
 *
 * Everything on that path runs in this library's own CUDA kernels for sm_103a
 * (GB300).  The library owns the weights, the cached prefix K/V and every
 * workspace; the caller owns the streaming buffer, the output chunk and the
 * CUDA stream.
 *
 * Conventions for every function:
 *   - Return FVA_OK or an error code; no C++ exception crosses this boundary.
 *   - Argument and state errors are detected on the host before any GPU work is
 *     queued and leave every buffer untouched; fva_last_error() describes the
 *     most recent error of the calling thread.
 *   - Device pointers are plain CUDA device addresses on the device that was
 *     current when fva_create ran; host pointers are ordinary host memory.
 *   - Asynchronous CUDA faults surface as FVA_ERR_CUDA from a later call.
 *   - A handle must not be used by two threads at once, nor on two streams whose
 *     work can overlap: every queued call of a handle shares its parameter block,
 *     workspaces and scratch, so the calls of one handle must be ordered on the
 *     GPU (one stream per handle, or streams the caller orders with events).
 *   - Every wait inside the library's kernels is bounded (2 s of GPU wall clock):
 *     a kernel that gives up records a code in the handle's error word and
 *     finishes without faulting; a later call returns FVA_ERR_TIMEOUT once (the
 *     word is then cleared) and the calls after it run normally.
 */
#ifndef FVA_H_
#define FVA_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define FVA_ABI_VERSION 1

/* A CUDA stream (layout-compatible with cudaStream_t; NULL = legacy default stream). */
typedef struct CUstream_st* fva_stream;

typedef enum fva_status {
  FVA_OK = 0,
  FVA_ERR_INVALID_ARG = 1,  /* bad pointer, size, shape or value                      */
  FVA_ERR_STATE = 2,        /* call out of order (e.g. step before weights / prefix) */
  FVA_ERR_OOM = 3,          /* device or pinned-host allocation failed              */
  FVA_ERR_CUDA = 4,         /* a CUDA runtime/driver call or a kernel failed        */
  FVA_ERR_UNSUPPORTED = 5,  /* shape outside what the kernels of this dtype support */
  FVA_ERR_TIMEOUT = 6       /* a kernel gave up a bounded wait (reported next call) */
} fva_status;

typedef enum fva_dtype {
  FVA_FP32 = 0,  /* weights, activations and GEMMs in fp32 (CUDA-core path)            */
  FVA_BF16 = 1   /* bf16 weights/activations, fp32 accumulate (tcgen05 tensor cores)   */
} fva_dtype;

/* fva_config.flags */
#define FVA_FLAG_NO_GRAPH 1u  /* launch the step kernel by kernel instead of replaying a CUDA graph */
/* Block-diagonal mask: every chunk attends to the prefix and to itself only (the
 * no-causal ablation of the paper's App. A.3) instead of the chunk-causal mask of
 * Sec. 3.1. */
#define FVA_FLAG_BLOCK_DIAGONAL 2u
/* bf16: run every projection as one launch of per-tile CTAs, never in the persistent
 * form (one CTA per SM walking several output tiles with two TMEM accumulators) that
 * is otherwise used where a projection has at least two output tiles per SM (large
 * batches).  Both forms give bit-identical results. */
#define FVA_FLAG_NO_PERSISTENT_GEMM 4u
/* bf16: split the attention's keys into fixed-size pieces whose results a second
 * kernel combines through global scratch, never into a thread-block cluster per query
 * tile that combines them in distributed shared memory (the form otherwise used when
 * every query tile's cluster fits on the GPU at once).  Each split's result is rounded
 * to bf16 before the combination, so the two forms agree to that rounding, and bit for
 * bit when they cut the keys at the same places. */
#define FVA_FLAG_NO_ATTN_CLUSTER 8u
/* bf16, fewer than 128 rows in the step (max_batch * K * H < 128, e.g. the paper's
 * 4 x 10, 4 x 20 and 5 x 10 buffers): the QKV and gate/up projections load their
 * activation tile through 128-row boxes, mostly zero padding, instead of boxes of the
 * row count rounded up to 16 (the MMA still runs 128 rows; the rows past the box are
 * never stored).  Both give bit-identical results. */
#define FVA_FLAG_FULL_A_BOX 16u

/*
 * Shape and numerics of the action expert and of the streaming buffer.
 *
 * The expert (App. A.4 of the paper: FiLM scale/shift/gate from the per-chunk
 * timestep embedding; dimensions of a pi0.5-style expert) is: in-projection A->W;
 * n_layers x [FiLM-modulated RMSNorm, MQA attention (n_q_heads query heads of
 * head_dim, one KV head) with rotate-half RoPE, gated residual, FiLM-modulated
 * RMSNorm, tanh-GELU gated MLP of mlp_dim, gated residual]; final FiLM-modulated
 * RMSNorm; out-projection W->A.
 *
 * bf16 kernels support: head_dim == 256, n_q_heads in {1,2,4,8,16}, width and
 * mlp_dim multiples of 128, action_dim <= 128.  fp32 kernels: any even head_dim
 * <= 256, width a multiple of 4 (>= 8), action_dim <= 128.
 */
typedef struct fva_config {
  int32_t abi_version;   /* must be FVA_ABI_VERSION                                  */
  int32_t dtype;         /* fva_dtype                                                */
  int32_t n_layers;      /* L                                                        */
  int32_t width;         /* W, residual width                                        */
  int32_t n_q_heads;     /* nq                                                       */
  int32_t n_kv_heads;    /* must be 1 (multi-query attention)                        */
  int32_t head_dim;      /* dh                                                       */
  int32_t mlp_dim;       /* F                                                        */
  int32_t action_dim;    /* A                                                        */
  int32_t n_chunks;      /* K, buffer length (the paper's N)                         */
  int32_t chunk_tokens;  /* H, tokens per chunk (the paper's chunk size C)           */
  int32_t max_batch;     /* largest batch (independent requests) passed to fva_step */
  int32_t max_prefix;    /* largest prefix length passed to fva_set_prefix_kv       */
  uint32_t flags;        /* FVA_FLAG_*                                               */
  float rms_eps;         /* RMSNorm epsilon (> 0)                                    */
  float rope_theta;      /* RoPE base; 0 disables RoPE                               */
  float t_min_period;    /* shortest period of the sinusoidal timestep embedding     */
  float t_max_period;    /* longest period                                           */
  uint64_t noise_seed;   /* Philox key of the tail noise drawn by fva_step           */
} fva_config;

typedef struct fva_handle fva_handle;

/*
 * Create a decoder on the current CUDA device: validates cfg, allocates every
 * device buffer for max_batch requests (weights, prefix/action K/V workspace,
 * activations, scratch) and zero-fills them.  *out receives the handle.
 * Errors: INVALID_ARG (bad field), UNSUPPORTED (shape outside the dtype's
 * kernels), OOM, CUDA.  Nothing is allocated when an error is returned.  No
 * environment variable is read.
 */
fva_status fva_create(const fva_config* cfg, fva_handle** out);

/* Release every resource of h (NULL is a no-op).  Synchronises the device first. */
void fva_destroy(fva_handle* h);

/* Number of tensors fva_load_weights expects for cfg (0 if cfg is invalid). */
int32_t fva_num_weights(const fva_config* cfg);

/*
 * Shape [rows, cols] (row-major, cols contiguous; vectors have rows == 1) of
 * tensor `index` in the fva_load_weights order:
 *   0 w_in [W, A]      1 b_in [W]      2 w_t1 [W, W]   3 b_t1 [W]
 *   4 w_t2 [W, W]      5 b_t2 [W]
 *   then for each layer l (base 6 + 11 l):
 *     +0 w_mod1 [3W, W]  +1 b_mod1 [3W]   (scale | shift | gate, before attention)
 *     +2 w_mod2 [3W, W]  +3 b_mod2 [3W]   (scale | shift | gate, before the MLP)
 *     +4 w_q [nq dh, W]  +5 w_k [dh, W]   +6 w_v [dh, W]   +7 w_o [W, nq dh]
 *     +8 w_gate [F, W]   +9 w_up [F, W]   +10 w_down [W, F]
 *   then w_modf [2W, W], b_modf [2W] (scale | shift of the final norm),
 *   w_out [A, W], b_out [A].
 * Every matrix maps its input (cols) to its output (rows): y = x M^T + b.
 */
fva_status fva_weight_shape(const fva_config* cfg, int32_t index, int64_t* rows, int64_t* cols);

/*
 * Copy all weights into the library (the caller's arrays are not retained).
 * tensors[i] points to tensor i above, element type = cfg.dtype (fp32, or bf16
 * as raw uint16 bit patterns); on_device != 0 means device pointers, else host.
 * May be called again to replace the weights.  Synchronous.
 * Errors: INVALID_ARG (n_tensors != fva_num_weights, NULL entry), CUDA.
 */
fva_status fva_load_weights(fva_handle* h, const void* const* tensors, int32_t n_tensors,
                            int32_t on_device);

/*
 * Install the cached VLM prefix keys/values of one observation for `request`
 * (§3.1: every action token attends to the observation's prefix K/V).
 * layer >= 0: k and v are [len, head_dim] for that layer; layer == -1: k and v
 * are [n_layers, len, head_dim] for all layers.  Element type = cfg.dtype.  K is
 * taken as already rotated by RoPE at positions 0..len-1; action token t of the
 * request then sits at position len + t.  on_device selects device vs host
 * pointers.  Copies are queued on `stream`; the caller's arrays may be reused
 * once the stream reaches this point.  0 <= len <= max_prefix.  Every layer of a
 * request must have the same len before fva_step uses that request.
 */
fva_status fva_set_prefix_kv(fva_handle* h, int32_t request, int32_t layer, const void* k,
                             const void* v, int32_t len, int32_t on_device, fva_stream stream);

/*
 * Let `request` use the prefix K/V of `src_request` (every layer, same length)
 * without a copy of it: the attention reads the shared prefix keys and values from
 * src_request's rows.  Only the prefix rows past the last multiple of 64 (fewer than
 * 64 per layer; the whole prefix on an fp32 handle is still read from the source)
 * are copied into request's rows, because the attention's 64-key block that
 * straddles the prefix end also holds request's own action keys.  This is the
 * packed multi-buffer forward of the paper (§3.3, App. A.4): N buffer
 * configurations of one observation, separated by the mask and reading one prefix.
 * The share lasts until either request's prefix is set again: setting
 * src_request's prefix (fva_set_prefix_kv) drops the share, and request's next
 * step then returns FVA_ERR_STATE until it is set or shared again.  Queued on
 * `stream`.  Errors: INVALID_ARG (request out of range or equal to src_request),
 * STATE (src_request has no complete prefix, or itself shares one), CUDA.
 */
fva_status fva_share_prefix_kv(fva_handle* h, int32_t request, int32_t src_request,
                               fva_stream stream);

/*
 * One steady-streaming step (§3.2, Algorithm 1; Eq. 1 and 2) for `batch`
 * independent requests, queued on `stream`; returns without waiting.
 *   buffer       fp32 [batch, K, H, A], slot 0 = cleanest chunk; updated in place
 *                to [x'_2, ..., x'_K, z] where x'_k = x_k + dt_k v_k.
 *   noise_levels host fp32 [batch, K]: tau_1 < ... < tau_K, each in (0, 1], per
 *                request (read before the call returns).  dt_k = tau_{k-1} - tau_k
 *                with tau_0 = 0, computed in fp32.
 *   out_chunk    fp32 [batch, H, A]: the emitted clean chunk x'_1.
 *   batch        1 .. max_batch.
 * buffer and out_chunk are device memory, or pinned host memory mapped at the same
 * address (cudaHostAlloc / cudaMallocHost, or cudaHostRegister with the mapped flag,
 * on a unified-address system): the step's kernels then read the buffer from and
 * write the buffer and the chunk to host memory themselves, over the host link
 * (NVLink-C2C on Grace), without a copy on the stream.  Pageable host memory is
 * refused (INVALID_ARG) before anything is queued.
 * The tail chunk z is drawn from Philox4x32-10 (key noise_seed, counter =
 * (element/4, request, step index)) with Box-Muller; the step index starts at 0 and
 * increases by one per call.  No allocation and no host synchronisation happen
 * inside (except waiting for the parameter ring slot used `FVA_PARAM_RING` calls
 * earlier).  Errors: INVALID_ARG (NULL, batch, non-increasing or out-of-range
 * tau), STATE (no weights, a request without a complete prefix), TIMEOUT / CUDA
 * (an earlier step failed on the GPU).
 */
fva_status fva_step(fva_handle* h, float* buffer, const float* noise_levels, float* out_chunk,
                    int32_t batch, fva_stream stream);

#define FVA_PARAM_RING 8

/* fva_step_opts.flags.  REUSE_FILM: the FiLM modulation (timestep embedding, time
 * MLP and every layer's scale / shift / gate) depends on the noise levels only, and
 * in steady streaming those are the same every step (§3.2).  With this flag the
 * modulation computed by the previous step on this handle is reused instead of
 * recomputed, provided that step ran with the same batch and bit-identical
 * noise_levels (and the weights were not reloaded since); otherwise it is computed
 * as usual.  Results are identical either way. */
#define FVA_STEP_REUSE_FILM 1u

/* fva_step_opts.flags.  SERIAL_FILM: compute every layer's FiLM modulation in one
 * projection before the first layer.  By default (bf16, at most 16 chunk rows, the
 * per-tile QKV projection) only layer 0's (scale, shift) pair is computed up front
 * and each layer's QKV projection launch computes the next 6W modulation columns
 * in extra CTAs on the SMs it leaves idle, before any norm reads them.  Results are
 * bit-identical either way; the flag exists for comparison. */
#define FVA_STEP_SERIAL_FILM 2u

/* Extra inputs / outputs of fva_step_ex (zero-initialise; every field optional). */
typedef struct fva_step_opts {
  const float* fresh_noise;  /* device fp32 [batch, H, A]: tail chunk to push instead of Philox */
  float* velocity_out;       /* device fp32 [batch, K, H, A]: receives v                        */
  int32_t trace_layer;       /* >= 0: write that layer's intermediates to trace_out            */
  uint32_t flags;            /* FVA_STEP_* below                                               */
  float* trace_out;          /* device fp32, fva_trace_floats(h, batch) floats; see below      */
  const int32_t* n_valid;    /* host int32 [batch], each in 1..K: real chunks per request      */
} fva_step_opts;

/*
 * fva_step with options.
 *
 * Cold start (Sec. 3.2, Algorithm 1): with n_valid set, request r holds n_valid[r]
 * real chunks in slots K - n_valid[r] .. K-1 and padding in the cleaner slots
 * before them.  Padding tokens are never attention keys, so the real chunks
 * move as if the padding were absent; the padding slots' velocities, the
 * emitted chunk while it is padding and the padding slots of the updated buffer
 * are meaningless (the caller executes its default action instead).  The roll
 * and the tail push are those of a steady step (the queue keeps its length), so
 * Algorithm 1 is: buffer = [pad, ..., pad, z]; K-1 steps with n_valid = 1 .. K-1;
 * then steady steps (n_valid NULL or K).  A query without any visible key (a
 * padding token of a request with no prefix) gets a zero attention output.
 * INVALID_ARG if an entry is outside 1..K.
 *
 * With trace_layer >= 0 the step runs kernel by kernel
 * (no graph) and, for M = batch*K*H rows, writes fp32 copies of that layer's
 * tensors to trace_out back to back in this order:
 *   h_in [M, W], y1 [M, W], q [M, nq dh] (after RoPE), k [M, dh] (after RoPE),
 *   v [M, dh], attn [M, nq dh], h_mid [M, W], y2 [M, W], mlp [M, F], h_out [M, W],
 *   cond [batch*K, W] (per-chunk timestep condition).
 */
fva_status fva_step_ex(fva_handle* h, float* buffer, const float* noise_levels, float* out_chunk,
                       int32_t batch, const fva_step_opts* opts, fva_stream stream);

/* Floats needed by trace_out for `batch` (see fva_step_ex). */
int64_t fva_trace_floats(const fva_handle* h, int32_t batch);

/* Step index used for the next call's tail noise (checkpoint / resume of a stream). */
fva_status fva_set_step_index(fva_handle* h, uint64_t step);
fva_status fva_get_step_index(const fva_handle* h, uint64_t* step);

/*
 * The chunk-causal mask as the attention kernel applies it (§3.1): for each
 * request r < batch and action token t < K*H, key_limit[r*K*H + t] receives the
 * number of leading keys of [prefix_r ; action tokens of r] that the token
 * attends to, P_r + (floor(t/H) + 1) H.  key_limit is a device int32 array.
 */
fva_status fva_mask_table(fva_handle* h, int32_t batch, int32_t* key_limit, fva_stream stream);

/*
 * The chunk-wise causal multi-query attention of one expert layer (§3.1), as the
 * step computes it, on caller-owned buffers (bf16 handles only):
 *   q           device bf16 [batch*K*H*nq, head_dim]; row (r*K*H + t)*nq + head is
 *               head `head` of action token t of request r (RoPE already applied).
 *   k, v        device bf16 [batch, kv_rows, head_dim]: request r's keys/values in
 *               the order [prefix_r ; action tokens 0..K*H-1].
 *   prefix_len  device int32 [batch]: P_r, with P_r + K*H <= kv_rows.
 *   out         device bf16 [batch*K*H*nq, head_dim] (same row order as q).
 * Token t attends to the first P_r + (floor(t/H) + 1) H keys of its request;
 * softmax scale 1/sqrt(head_dim).  Uses the handle's split-KV scratch, so calls
 * on one handle must not overlap on the GPU.  Requires 1 <= batch <= max_batch and
 * kv_rows <= max_prefix + K*H, and 16-byte aligned pointers.  Errors: INVALID_ARG,
 * UNSUPPORTED (fp32 handle), CUDA.  A device P_r that breaks 0 <= P_r and
 * P_r + K*H <= kv_rows cannot be seen on the host: the kernel leaves request r's
 * rows unwritten and the next fva_step on the handle returns FVA_ERR_INVALID_ARG.
 */

/*
 * The tanh-form GELU exactly as the bf16 gate/up epilogue evaluates it, before the
 * product with the up branch and the bf16 rounding (the fp32 dtype uses a separate,
 * full-precision form): y[i] = 0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3))) with
 * tanh from the PTX tanh.approx.f32 instruction, whose absolute error bound makes
 * |y - GELU(x)| <= |x| 2^-12.  x and y are device fp32 arrays of n >= 0 elements.
 * Errors: INVALID_ARG, CUDA.
 */
fva_status fva_geglu_gelu(const float* x, float* y, int64_t n, fva_stream stream);
fva_status fva_chunk_attention(fva_handle* h, const void* q, const void* k, const void* v,
                               const int32_t* prefix_len, int32_t batch, int32_t kv_rows,
                               void* out, fva_stream stream);

/*
 * fva_chunk_attention without any device allocation and without a handle.  The
 * paper has no counterpart: this exists for callers that cannot allocate device
 * memory -- a controller running the decoder in a fixed-period loop, where
 * cudaMalloc / cudaFree may synchronise the device for an unbounded time, or a
 * host that gives all device memory to its own pool at start-up.
 *
 * Same inputs, output, kernel and mask as fva_chunk_attention, with the shapes
 * passed explicitly (head_dim must be 256, n_q_heads one of 1, 2, 4, 8, 16).  Its
 * key splits are always 256 keys, while a handle may use shorter ones, so the two
 * can differ by bf16 rounding.  The split-KV
 * scratch is a fixed array inside the library: 256 slots of 128 x 256 bf16 plus
 * row statistics (16 MiB + 256 KiB), kept by every GPU that loads the library
 * until the process exits.  A call needs
 *   batch * ceil(K*H*n_q_heads / 128) * ceil(kv_rows / 256)
 * slots (and ceil(kv_rows / 256) <= 32); larger calls return FVA_ERR_INVALID_ARG.
 * The first call on a device looks up the array's device address (and sets the
 * kernel attributes) with that device current; make that first call before any
 * stream capture.  Every call uses the same array, which keeps the last call's
 * contents (nothing in it needs to start at zero): calls that overlap on the GPU,
 * from any thread or stream, race.  Device-side problems (a prefix length P_r with
 * P_r + K*H > kv_rows, or P_r < 0) leave request r's rows unwritten and are not
 * reported.
 * Calls no cudaMalloc, cudaFree or other allocating routine.
 */
fva_status fva_chunk_attention_noalloc(const void* q, const void* k, const void* v,
                                       const int32_t* prefix_len, int32_t batch,
                                       int32_t n_chunks, int32_t chunk_tokens,
                                       int32_t n_q_heads, int32_t head_dim, int32_t kv_rows,
                                       void* out, fva_stream stream);

/*
 * Test hook of the bounded waits (no counterpart in the paper).  Queues on
 * `stream` one kernel whose only wait can never complete: after limit_us
 * (1 .. 1000000) microseconds of GPU wall clock it records a timeout code in the
 * handle's error word and returns, as every bounded wait of the library does.
 * The first fva_step / fva_step_ex issued after the stream has passed that point
 * (e.g. after synchronising it) returns FVA_ERR_TIMEOUT without queuing work;
 * the step after that runs normally.  Errors: INVALID_ARG, CUDA.
 */
fva_status fva_check_bounded_wait(fva_handle* h, int32_t limit_us, fva_stream stream);

/* Kernels of one step, as reported by fva_step_profile. */
typedef enum fva_kernel_kind {
  FVA_K_TIMESTEP_EMBED = 0,  /* sinusoidal embedding of every chunk's tau             */
  FVA_K_TIME_MLP = 1,        /* one of the two SiLU linear layers of the condition   */
  FVA_K_FILM = 2,            /* FiLM projections of every layer (one GEMM)           */
  FVA_K_EMBED_NORM = 3,      /* action in-projection + layer-0 FiLM RMSNorm          */
  FVA_K_QKV = 4,             /* packed QKV projection + RoPE + KV append             */
  FVA_K_ATTENTION = 5,       /* chunk-causal MQA over prefix + action keys           */
  FVA_K_OUT_PROJ = 6,        /* attention output projection (split-K partials)       */
  FVA_K_RESID_NORM = 7,      /* split-K reduction + gated residual + FiLM RMSNorm    */
  FVA_K_GATE_UP = 8,         /* packed gate/up projection + tanh-GELU gating         */
  FVA_K_DOWN = 9,            /* MLP down projection (split-K partials)               */
  FVA_K_FINAL = 10,          /* last gated residual + final FiLM RMSNorm (fp32 out)  */
  FVA_K_ATTN_MERGE = 11,     /* combination of the attention's key splits            */
  FVA_K_VELOCITY = 12,       /* out-projection + Euler + emit + roll + tail          */
  FVA_K_PARAMS = 13,         /* the step's tau, dt, step index from the pinned ring   */
  FVA_K_COUNT = 14
} fva_kernel_kind;

typedef struct fva_kernel_time {
  int32_t kind;        /* fva_kernel_kind                                    */
  int32_t layer;       /* expert layer, or -1                                */
  float microseconds;  /* CUDA-event time from this launch to the next one   */
} fva_kernel_time;

/*
 * One step exactly like fva_step (same kernels, same results, advances the step
 * index), replayed from a separately captured CUDA graph that has an event node
 * before every kernel and after the last (the events serialise the kernels, so
 * the overlap programmatic dependent launch gives the normal step is lost).
 * Waits for the stream, then writes one record per launch, in launch order, to
 * records[0 .. *n_records); each duration spans from the launch's event to the
 * next one.  Errors: as fva_step, plus INVALID_ARG when max_records is smaller
 * than the number of launches.
 */
fva_status fva_step_profile(fva_handle* h, float* buffer, const float* noise_levels,
                            float* out_chunk, int32_t batch, fva_kernel_time* records,
                            int32_t max_records, int32_t* n_records, fva_stream stream);

/* Description of the calling thread's most recent error ("" if none). */
const char* fva_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* FVA_H_ */
