// The part of an action-expert layer that follows attention, as one persistent
// kernel: output projection, gated residual and FiLM-modulated norm 2, gate/up
// projection with tanh-GELU gating, down projection, gated residual, and then
// the next layer's modulated norm 1 and QKV projection (RoPE, KV append) or, on
// the last layer, the final modulated norm (App. A.4 block structure; Sec. 3.2
// packs the step into few GPU programs).
//
// The host builds a task list in stage order: output-projection tiles, norm-2
// row groups, gate/up tiles, down tiles, norm row groups, QKV tiles.  CTA c runs
// tasks c, c + G, c + 2G, ... in order (G CTAs, one per SM, all resident).  A
// task waits until a counter of its 128-row tile reaches a target; counters are
// raised by the tasks it depends on, and every such task has a smaller index.
// The smallest unfinished task therefore always has its inputs, and its CTA has
// finished everything before it, so the kernel cannot deadlock.  Row tiles are
// independent outside attention, so tile 0 can be in its MLP while tile 3 is
// still in its output projection.
//
// Roles of the 320 threads of a CTA:
//   warp 0     TMA producer.  For each GEMM task it first requests the weight (B)
//              tiles of the first ring slots (weights never depend on other
//              tasks), then waits for the task's counter and requests the
//              activation (A) tiles: the weights of the next task stream in while
//              the CTA still works on the previous one.
//   warp 1     TMEM owner (two 256-column fp32 accumulators, so the epilogue of
//              one tile overlaps the MMAs of the next) and tcgen05.mma issuer.
//   warps 2-9  GEMM epilogues (TMEM -> registers -> coalesced stores; two warps
//              per TMEM lane quarter, each taking half of the tile's columns) and
//              the norm row groups (two warps per row); they raise the task's
//              counter.  An SM stores far slower than it loads, and one warp
//              alone is latency-bound, so the epilogue gets eight warps.
// Every wait is bounded.  When one gives up, the kernel records an error code,
// every later wait returns at once, and the kernel drains its own copies and
// MMAs before it releases TMEM and exits.
#include <algorithm>
#include <cstring>

#include "common.cuh"
#include "gemm_epilogue.cuh"
#include "kernels.h"

namespace fva {
namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kEpiWarps = 8;
constexpr int kThreads = 64 + 32 * kEpiWarps;
constexpr int kNormRows = kEpiWarps / 2;  // rows of one norm task (two warps per row)
constexpr int kStages = 4;
constexpr int kABytes = kBM * kBK * 2;            // 16 KB
constexpr int kSlotBytes = kABytes + 256 * kBK * 2;  // A + B for tiles up to 256 wide
constexpr int kAccCols = 256;
constexpr int kTmemCols = 2 * kAccCols;
constexpr int kEpiStageBytes = 32 * 80;           // per epilogue warp: 32 rows x 64 bytes
constexpr int kBarBytes = 256;
constexpr int kSmemBytes =
    1024 /*alignment*/ + kStages * kSlotBytes + kEpiWarps * kEpiStageBytes + kBarBytes;
constexpr int KERR_WAIT_DEP = 5;  // a task waited too long for a counter
// Tile widths: the split-K projections write fp32 partial tiles, and an SM
// stores far slower than it loads, so they use narrow tiles (more CTAs share
// the stores); gate/up uses the 256-wide tile its weight interleave is built for.
constexpr int kBnO = 128, kBnD = 128, kBnQ = 128;  // gate/up: kBnGU (weight interleave)

// GEMM operation of a task kind: 0 out-proj, 1 gate/up, 2 down, 3 QKV; -1 norm.
__device__ __forceinline__ int gemm_op(int kind) {
  switch (kind) {
    case BK_OUT_PROJ: return 0;
    case BK_GATE_UP: return 1;
    case BK_DOWN: return 2;
    case BK_QKV: return 3;
    default: return -1;
  }
}

struct BlockParams {
  CUtensorMap a[4];
  CUtensorMap b[4];
  int b_box[4];
  int bn[4];
  int kb_per_split[4];
  GemmEpi epi[4];
  BlockNorm norm[2];
  int M, T, K, H, W, N_mod;
  float eps;
  const BlockTask* tasks;
  int n_tasks;
  unsigned* ctr;
  int* err;
};

__device__ __forceinline__ bool aborted(const int* err) {
  return *reinterpret_cast<const volatile int*>(err) != 0;
}

// Bounded mbarrier wait that also gives up as soon as any wait of the kernel has.
__device__ __forceinline__ bool bk_wait(uint64_t* bar, uint32_t parity, int* err, int code) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = globaltimer_ns();
  uint32_t n = 0;
  while (!mbar_try_wait(bar, parity)) {
    if ((++n & 255u) == 0u) {
      if (aborted(err)) return false;
      if (globaltimer_ns() - t0 > kWaitLimitNs) {
        report_error(err, code);
        return false;
      }
    }
  }
  return true;
}

__device__ __forceinline__ unsigned ld_relaxed(const unsigned* p) {
  unsigned v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void fence_acquire_gpu() {
  asm volatile("fence.acq_rel.gpu;" ::: "memory");
}

__device__ __forceinline__ void red_release_add(unsigned* p, unsigned v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Orders this thread's generic-proxy global accesses with its async-proxy (TMA)
// ones: writers issue it before raising a counter, the TMA producer after
// observing one.
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

__device__ __forceinline__ void epi_bar_sync() {
  asm volatile("bar.sync 1, %0;" ::"r"(kEpiWarps * 32) : "memory");
}

// Spins with relaxed loads and orders what follows with one fence once the
// counter has reached the target.
__device__ bool wait_counter(const unsigned* c, unsigned target, int* err) {
  if (ld_relaxed(c) >= target) {
    fence_acquire_gpu();
    return true;
  }
  const unsigned long long t0 = globaltimer_ns();
  uint32_t n = 0;
  while (ld_relaxed(c) < target) {
    __nanosleep(32);
    if ((++n & 63u) == 0u) {
      if (aborted(err)) return false;
      if (globaltimer_ns() - t0 > kWaitLimitNs) {
        report_error(err, KERR_WAIT_DEP);
        return false;
      }
    }
  }
  fence_acquire_gpu();
  return true;
}

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Half `hf` of row m of  h += gate * sum_z part[z];  y = rmsnorm(h)(1 + scale) + shift,
// by one warp (the other half by its partner warp; sums of squares meet in
// red[8]).  Lane holds columns ((hf*vh + v)*32 + lane)*4 .. +3, v < vh = W / 256
// (at most 4).
// Partials and h were written by other CTAs of this kernel: read through L2.
// Every load of the half row is in flight at once; partials are summed in split
// order.
__device__ __forceinline__ void norm_task(const BlockNorm& nm, const BlockParams& p, int m,
                                          bool active, int hf, int slot, float* red, int lane) {
  constexpr int VH = 4;
  const int vh = p.W >> 8;
  float4 hv[VH];
  float ss = 0.f;
  const float* mrow = nullptr;
  const size_t base = (size_t)m * p.W;
  if (active) {
    const int r = m / p.T, c = (m - r * p.T) / p.H;
    mrow = nm.mod + (size_t)(r * p.K + c) * p.N_mod;
    const float4* p0 = reinterpret_cast<const float4*>(nm.part + base);
    const long long ps = nm.part_stride / 4;
    const int np = nm.n_parts;
    float4* h4 = reinterpret_cast<float4*>(nm.h + base);
    float4 acc[VH], x1[VH], x2[VH], x3[VH];
#pragma unroll
    for (int v = 0; v < VH; ++v) {
      if (v >= vh) break;
      const int o = (hf * vh + v) * 32 + lane;
      acc[v] = __ldcg(p0 + o);
      if (np > 1) x1[v] = __ldcg(p0 + ps + o);
      if (np > 2) x2[v] = __ldcg(p0 + 2 * ps + o);
      if (np > 3) x3[v] = __ldcg(p0 + 3 * ps + o);
      hv[v] = __ldcg(h4 + o);
    }
#pragma unroll
    for (int v = 0; v < VH; ++v) {
      if (v >= vh) break;
      if (np > 1) { acc[v].x += x1[v].x; acc[v].y += x1[v].y; acc[v].z += x1[v].z; acc[v].w += x1[v].w; }
      if (np > 2) { acc[v].x += x2[v].x; acc[v].y += x2[v].y; acc[v].z += x2[v].z; acc[v].w += x2[v].w; }
      if (np > 3) { acc[v].x += x3[v].x; acc[v].y += x3[v].y; acc[v].z += x3[v].z; acc[v].w += x3[v].w; }
    }
    for (int z = 4; z < np; ++z)
#pragma unroll
      for (int v = 0; v < VH; ++v) {
        if (v >= vh) break;
        const float4 q = __ldcg(p0 + z * ps + (hf * vh + v) * 32 + lane);
        acc[v].x += q.x; acc[v].y += q.y; acc[v].z += q.z; acc[v].w += q.w;
      }
#pragma unroll
    for (int v = 0; v < VH; ++v) {
      if (v >= vh) break;
      const int o = (hf * vh + v) * 32 + lane;
      const float4 g = __ldg(reinterpret_cast<const float4*>(mrow + nm.gate_off) + o);
      hv[v].x = fmaf(g.x, acc[v].x, hv[v].x);
      hv[v].y = fmaf(g.y, acc[v].y, hv[v].y);
      hv[v].z = fmaf(g.z, acc[v].z, hv[v].z);
      hv[v].w = fmaf(g.w, acc[v].w, hv[v].w);
      __stcg(h4 + o, hv[v]);
      ss += hv[v].x * hv[v].x + hv[v].y * hv[v].y + hv[v].z * hv[v].z + hv[v].w * hv[v].w;
    }
    ss = warp_sum_f(ss);
    if (lane == 0) red[hf * kNormRows + slot] = ss;
  }
  epi_bar_sync();
  if (active) {
    const float tot = red[slot] + red[kNormRows + slot];
    const float rn = rsqrtf(tot / (float)p.W + p.eps);
#pragma unroll
    for (int v = 0; v < VH; ++v) {
      if (v >= vh) break;
      const int o = (hf * vh + v) * 32 + lane;
      const float4 sc = __ldg(reinterpret_cast<const float4*>(mrow + nm.scale_off) + o);
      const float4 sh = __ldg(reinterpret_cast<const float4*>(mrow + nm.shift_off) + o);
      const float y0 = hv[v].x * rn * (1.f + sc.x) + sh.x, y1 = hv[v].y * rn * (1.f + sc.y) + sh.y,
                  y2 = hv[v].z * rn * (1.f + sc.z) + sh.z, y3 = hv[v].w * rn * (1.f + sc.w) + sh.w;
      if (nm.y_f32) {
        __stcg(reinterpret_cast<float4*>((float*)nm.y + base) + o, make_float4(y0, y1, y2, y3));
      } else {
        __nv_bfloat162 lo = __floats2bfloat162_rn(y0, y1), hi = __floats2bfloat162_rn(y2, y3);
        uint2 u;
        u.x = *reinterpret_cast<uint32_t*>(&lo);
        u.y = *reinterpret_cast<uint32_t*>(&hi);
        __stcg(reinterpret_cast<uint2*>((bf16*)nm.y + base) + o, u);
      }
    }
  }
}

// ---- GEMM epilogues: one output row per thread, this warp's half `hf` of the
// tile's columns, stored through the warp's 32 x 64-byte stage.

// split-K partial plane (fp32), tile kBnO wide
__device__ __forceinline__ void epi_partial(const GemmEpi& ep, uint32_t trow, int m, bool ok,
                                            int n0, int split, int hf, uint8_t* stage, int lane) {
  constexpr int kCols = kBnO / 2;
  uint32_t v[kCols];
  tmem_ld32_nowait(trow + hf * kCols, *reinterpret_cast<uint32_t(*)[32]>(&v[0]));
  tmem_ld32_nowait(trow + hf * kCols + 32, *reinterpret_cast<uint32_t(*)[32]>(&v[32]));
  tmem_ld_wait();
  float* dst = ok ? (float*)ep.out + split * ep.split_stride + (size_t)m * ep.ldo + n0 +
                        hf * kCols
                  : nullptr;
#pragma unroll
  for (int c = 0; c < kCols; c += 16) {
    uint4 u[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) u[i] = make_uint4(v[c + 4 * i], v[c + 4 * i + 1], v[c + 4 * i + 2], v[c + 4 * i + 3]);
    warp_store_rows<64>(stage, u, dst ? dst + c : nullptr, lane);
  }
}

// gelu_tanh(gate) * up (bf16): tile columns [0, 128) gate, [128, 256) up; this
// warp makes outputs [64 hf, 64 hf + 64) of the tile's 128
__device__ __forceinline__ void epi_geglu(const GemmEpi& ep, uint32_t trow, int m, bool ok,
                                          int n0, int hf, uint8_t* stage, int lane) {
  constexpr int half = kBnGU / 2;
#pragma unroll 1
  for (int c = hf * 64; c < hf * 64 + 64; c += 32) {
    uint32_t g[32], u[32];
    tmem_ld32_nowait(trow + c, g);
    tmem_ld32_nowait(trow + half + c, u);
    tmem_ld_wait();
    float o[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) o[i] = gelu_tanh_bf16out(__uint_as_float(g[i])) * __uint_as_float(u[i]);
    uint4 pk[4];
    pack_bf16x32(o, pk);
    warp_store_rows<64>(stage, pk, ok ? (bf16*)ep.out + (size_t)m * ep.ldo + n0 / 2 + c : nullptr,
                        lane);
  }
}

// RoPE + q / KV-workspace scatter (weights permuted so that tile column c < 64
// holds head dim d = tj*64 + c of its segment and column c + 64 the rotate-half
// partner d + dh/2); this warp takes pairs [32 hf, 32 hf + 32).  cs points at the
// (cos, sin) pairs of the row's position and these pairs (nullptr: no rotation).
__device__ __forceinline__ void qkv_rope_pos(const GemmEpi& ep, int m, bool ok, int& r, int& pos) {
  r = 0;
  pos = 0;
  if (ok) {
    r = m / ep.T;
    pos = __ldg(ep.prefix_len + r) + (m - r * ep.T);
  }
}

__device__ __forceinline__ void epi_qkv(const GemmEpi& ep, uint32_t trow, int m, bool ok, int n0,
                                        int hf, const float4* cs, uint8_t* stage, int lane) {
  constexpr int half = kBnQ / 2;
  const int dh = ep.dh, seg = n0 / dh, tj = (n0 % dh) / kBnQ;
  int r, pos;
  qkv_rope_pos(ep, m, ok, r, pos);
  bf16* dst;
  if (seg < ep.nq)
    dst = (bf16*)ep.q + (size_t)m * ep.nq * dh + seg * dh;
  else
    dst = (bf16*)(seg == ep.nq ? ep.kc : ep.vc) + ((size_t)r * ep.S_cap + pos) * dh;
  const bool rotate = cs != nullptr;  // q and k heads of valid rows
  const int c = hf * 32;
  uint4 p1[4], p2[4];
#pragma unroll
  for (int q16 = 0; q16 < 2; ++q16) {  // 16 pairs at a time keeps registers low
    uint32_t a[16], b[16];
    tmem_ld16_nowait(trow + c + q16 * 16, a);
    tmem_ld16_nowait(trow + half + c + q16 * 16, b);
    tmem_ld_wait();
    float x1[16], x2[16];
#pragma unroll
    for (int i = 0; i < 16; i += 2) {
      const float a0 = __uint_as_float(a[i]), b0 = __uint_as_float(b[i]);
      const float a1 = __uint_as_float(a[i + 1]), b1 = __uint_as_float(b[i + 1]);
      if (rotate) {
        const float4 q = __ldg(cs + q16 * 8 + i / 2);
        x1[i] = a0 * q.x - b0 * q.y;
        x2[i] = b0 * q.x + a0 * q.y;
        x1[i + 1] = a1 * q.z - b1 * q.w;
        x2[i + 1] = b1 * q.z + a1 * q.w;
      } else {
        x1[i] = a0; x2[i] = b0; x1[i + 1] = a1; x2[i + 1] = b1;
      }
    }
    p1[2 * q16] = pack_bf16x8(&x1[0]);
    p1[2 * q16 + 1] = pack_bf16x8(&x1[8]);
    p2[2 * q16] = pack_bf16x8(&x2[0]);
    p2[2 * q16 + 1] = pack_bf16x8(&x2[8]);
  }
  const int d0 = tj * half + c;
  warp_store_rows<64>(stage, p1, ok ? dst + d0 : nullptr, lane);
  warp_store_rows<64>(stage, p2, ok ? dst + d0 + dh / 2 : nullptr, lane);
}

__device__ __forceinline__ BlockTask load_task(const BlockTask* tasks, int j) {
  const uint4 u = __ldg(reinterpret_cast<const uint4*>(tasks) + j);
  BlockTask t;
  t.kind = (uint16_t)(u.x & 0xffffu);
  t.m = (uint16_t)(u.x >> 16);
  t.n = (uint16_t)(u.y & 0xffffu);
  t.split = (uint16_t)(u.y >> 16);
  t.wait_ctr = (uint16_t)(u.z & 0xffffu);
  t.wait_target = (uint16_t)(u.z >> 16);
  t.done_ctr = (uint16_t)(u.w & 0xffffu);
  t.pad = 0;
  return t;
}

__global__ void __launch_bounds__(kThreads, 1) block_kernel(const __grid_constant__ BlockParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* epi_stage = smem + kStages * kSlotBytes;
  uint64_t* bars = (uint64_t*)(epi_stage + kEpiWarps * kEpiStageBytes);
  uint64_t* full = bars;                  // [kStages]
  uint64_t* empty = bars + kStages;       // [kStages]
  uint64_t* acc_full = bars + 2 * kStages;      // [2]
  uint64_t* acc_empty = bars + 2 * kStages + 2; // [2]
  uint64_t* drain = bars + 2 * kStages + 4;
  uint32_t* tmem_slot = (uint32_t*)(bars + 2 * kStages + 5);
  float* red = (float*)(bars + 2 * kStages + 6);  // [2][kNormRows] norm sums of squares

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], kEpiWarps);
    }
    mbar_init(drain, 1);
    fence_barrier_init();
    for (int i = 0; i < 4; ++i) {
      tma_prefetch_desc(&p.a[i]);
      tma_prefetch_desc(&p.b[i]);
    }
  }
  // One CTA per SM (shared memory), and no other tcgen05 kernel of the library
  // can share the SM with it, so the 512-column allocation never waits.
  if (warp == 1) tmem_alloc(tmem_slot, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();
  const int G = gridDim.x;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer
      uint32_t it = 0;  // ring stages issued so far
      bool ok = true, waited = false;
      for (int j = blockIdx.x; ok && j < p.n_tasks; j += G) {
        const BlockTask t = load_task(p.tasks, j);
        const int op = gemm_op(t.kind);
        if (op < 0) continue;
        const int bn = p.bn[op], nkb = p.kb_per_split[op], kb0 = t.split * nkb;
        const int m0 = t.m * kBM, n0 = t.n * bn, box = p.b_box[op];
        const uint32_t bytes = kABytes + bn * kBK * 2;
        const CUtensorMap* ma = &p.a[op];
        const CUtensorMap* mb = &p.b[op];
        const int pre = min(nkb, kStages);
        int nb = 0;
        for (; nb < pre; ++nb) {  // weights first
          const uint32_t st = (it + nb) % kStages, use = (it + nb) / kStages;
          if (!bk_wait(&empty[st], (use & 1u) ^ 1u, p.err, KERR_WAIT_MMA)) {
            ok = false;
            break;
          }
          uint8_t* slot = smem + st * kSlotBytes;
          mbar_arrive_expect_tx(&full[st], bytes);
          for (int r = 0; r < bn; r += box)
            tma_load_2d(slot + kABytes + r * 128, mb, (kb0 + nb) * kBK, n0 + r, &full[st]);
        }
        if (!waited) {  // activations of earlier kernels are read from here on
          pdl_wait();
          waited = true;
        }
        if (ok && t.wait_ctr != kNoCounter) ok = wait_counter(p.ctr + t.wait_ctr, t.wait_target, p.err);
        fence_proxy_async_global();
        // A of the stages whose B is on its way, even after a failed wait, so
        // every armed stage completes
        for (int i = 0; i < nb; ++i) {
          const uint32_t st = (it + i) % kStages;
          tma_load_2d(smem + st * kSlotBytes, ma, (kb0 + i) * kBK, m0, &full[st]);
        }
        it += nb;
        if (!ok || nb < pre) {
          ok = false;
          break;
        }
        for (int i = pre; i < nkb; ++i) {
          const uint32_t st = it % kStages, use = it / kStages;
          if (!bk_wait(&empty[st], (use & 1u) ^ 1u, p.err, KERR_WAIT_MMA)) {
            ok = false;
            break;
          }
          uint8_t* slot = smem + st * kSlotBytes;
          mbar_arrive_expect_tx(&full[st], bytes);
          tma_load_2d(slot, ma, (kb0 + i) * kBK, m0, &full[st]);
          for (int r = 0; r < bn; r += box)
            tma_load_2d(slot + kABytes + r * 128, mb, (kb0 + i) * kBK, n0 + r, &full[st]);
          ++it;
        }
      }
      if (!waited) pdl_wait();
      // drain: the last stage issued on each slot has landed before the CTA exits
      for (uint32_t k = 0; k < (uint32_t)kStages && k < it; ++k) {
        const uint32_t i = it - 1 - k;
        mbar_wait(&full[i % kStages], (i / kStages) & 1u, nullptr, 0);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer
      constexpr uint32_t idesc128 = umma_idesc_bf16(kBM, 128, false);
      constexpr uint32_t idesc256 = umma_idesc_bf16(kBM, 256, false);
      pdl_wait();
      uint32_t it = 0, acc = 0;
      bool ok = true;
      for (int j = blockIdx.x; ok && j < p.n_tasks; j += G) {
        const BlockTask t = load_task(p.tasks, j);
        const int op = gemm_op(t.kind);
        if (op < 0) continue;
        const int bn = p.bn[op], nkb = p.kb_per_split[op];
        const uint32_t buf = acc & 1u, use = acc >> 1;
        if (!bk_wait(&acc_empty[buf], (use & 1u) ^ 1u, p.err, KERR_WAIT_SYNC)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + buf * kAccCols;
        const uint32_t idesc = bn == 256 ? idesc256 : idesc128;
        for (int i = 0; i < nkb; ++i, ++it) {
          const uint32_t st = it % kStages;
          if (!bk_wait(&full[st], (it / kStages) & 1u, p.err, KERR_WAIT_TMA)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + st * kSlotBytes);
          const uint32_t sb = sa + kABytes;
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk) {
            const uint64_t ad = umma_desc_sw128(sa + kk * 32, 16, 1024);
            const uint64_t bd = umma_desc_sw128(sb + kk * 32, 16, 1024);
            umma_bf16(d, ad, bd, idesc, (i > 0 || kk > 0) ? 1u : 0u);
          }
          umma_commit(&empty[st]);
        }
        if (!ok) break;
        umma_commit(&acc_full[buf]);
        ++acc;
      }
      // every MMA issued by this thread completes before TMEM is released
      umma_commit(drain);
      mbar_wait(drain, 0, nullptr, 0);
    }
  } else {
    // ---------------- epilogues and norm row groups
    const int ew = warp - 2;
    const int quarter = warp & 3;  // TMEM lanes this warp may read
    const int hf = ew >> 2;        // half of the tile's columns (norm: half of the row)
    const int row = quarter * 32 + lane;
    uint8_t* stage = epi_stage + ew * kEpiStageBytes;
    pdl_wait();
    uint32_t acc = 0;
    bool ok = true;
    for (int j = blockIdx.x; j < p.n_tasks; j += G) {
      const BlockTask t = load_task(p.tasks, j);
      const int op = gemm_op(t.kind);
      if (op >= 0) {
        const uint32_t buf = acc & 1u, use = acc >> 1;
        const int m = t.m * kBM + row, n0 = t.n * p.bn[op];
        const bool okr = m < p.M;
        // RoPE (cos, sin) of this row's position: a constant table, pulled into
        // L1 before the accumulator is ready
        const float4* cs4 = nullptr;
        if (op == 3) {
          const GemmEpi& eq = p.epi[3];
          const int seg = n0 / eq.dh, tj = (n0 % eq.dh) / kBnQ;
          if (okr && seg <= eq.nq) {
            int r, pos;
            qkv_rope_pos(eq, m, okr, r, pos);
            cs4 = reinterpret_cast<const float4*>(eq.rope + (size_t)pos * (eq.dh / 2) +
                                                  tj * (kBnQ / 2) + hf * 32);
            asm volatile("prefetch.global.L1 [%0];" ::"l"(cs4));
            asm volatile("prefetch.global.L1 [%0];" ::"l"(cs4 + 8));
          }
        }
        if (ok) ok = __all_sync(0xffffffffu, bk_wait(&acc_full[buf], use & 1u, p.err, KERR_WAIT_MMA));
        if (ok) {
          tc_fence_after();
          const uint32_t trow = tmem + buf * kAccCols + ((uint32_t)(quarter * 32) << 16);
          if (op == 1)
            epi_geglu(p.epi[1], trow, m, okr, n0, hf, stage, lane);
          else if (op == 3)
            epi_qkv(p.epi[3], trow, m, okr, n0, hf, cs4, stage, lane);
          else
            epi_partial(p.epi[op], trow, m, okr, n0, t.split, hf, stage, lane);
          tc_fence_before();
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&acc_empty[buf]);
        ++acc;
      } else {
        if (ok && t.wait_ctr != kNoCounter) {
          bool w = true;
          if (lane == 0) w = wait_counter(p.ctr + t.wait_ctr, t.wait_target, p.err);
          ok = __shfl_sync(0xffffffffu, w ? 1 : 0, 0) != 0;
        }
        __syncwarp();
        const int slot = ew & (kNormRows - 1);
        norm_task(p.norm[t.kind == BK_NORM_MID ? 0 : 1], p, t.m + slot, ok && slot < t.n, hf,
                  slot, red, lane);
      }
      if (t.done_ctr != kNoCounter) {
        fence_proxy_async_global();
        epi_bar_sync();
        if (ew == 0 && lane == 0) {
          __threadfence();
          red_release_add(p.ctr + t.done_ctr, 1u);
        }
      }
    }
  }
  // the producer and MMA lanes rejoin their warps first: a CTA barrier reached
  // by a split warp does not wait for the rest of the CTA
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace

bool block_supported(const BlockShape& s) {
  if (s.W % 256 != 0 || s.W > 1024) return false;  // norm: W / 256 float4 per lane and warp
  if (s.split_o < 1 || s.split_o > kBlockMaxSplits || s.split_d < 1 || s.split_d > kBlockMaxSplits)
    return false;
  if ((s.Dq / kBK) % s.split_o != 0 || (s.F / kBK) % s.split_d != 0) return false;
  if (s.F % (s.split_d * (kBnGU / 2)) != 0 || (2 * s.F) % kBnGU != 0 || s.N_qkv % kBnQ != 0 ||
      s.W % kBnO != 0 || s.W % kBnD != 0)
    return false;
  const int mt = (s.M + kBM - 1) / kBM;
  if (s.M <= 0 || s.M > 65535 || mt * kBlockCtrPerTile > 65535) return false;
  return true;
}

int block_max_tasks(const BlockShape& s) {
  const int mt = (s.M + kBM - 1) / kBM;
  return mt * ((s.W / kBnO) * s.split_o + kBM / kNormRows + (2 * s.F) / kBnGU +
               (s.W / kBnD) * s.split_d + kBM / kNormRows + (s.next_qkv ? s.N_qkv / kBnQ : 0));
}

void build_block_tasks(const BlockShape& s, BlockTask* out, int* n_tasks, int max_tasks) {
  const int mt = (s.M + kBM - 1) / kBM;
  const int gps = (s.F / s.split_d) / (kBnGU / 2);  // gate/up tiles per down K-slice
  enum { C_O = 0, C_N2 = 1, C_D = 2, C_N1 = 3, C_GU = 4 };
  auto ctr = [&](int m, int k) { return (uint16_t)(m * kBlockCtrPerTile + k); };
  auto groups = [&](int m) { return (std::min(kBM, s.M - m * kBM) + kNormRows - 1) / kNormRows; };
  int n = 0;
  auto put = [&](int kind, int m, int nn, int split, uint16_t wc, int wt, uint16_t dc) {
    if (n >= max_tasks) return;
    BlockTask& t = out[n++];
    t.kind = (uint16_t)kind;
    t.m = (uint16_t)m;
    t.n = (uint16_t)nn;
    t.split = (uint16_t)split;
    t.wait_ctr = wc;
    t.wait_target = (uint16_t)wt;
    t.done_ctr = dc;
    t.pad = 0;
  };
  auto norms = [&](int kind, int wait_k, int wait_target, int done_k) {
    for (int m = 0; m < mt; ++m) {
      const int rows = std::min(kBM, s.M - m * kBM);
      for (int r = 0; r < rows; r += kNormRows)
        put(kind, m * kBM + r, std::min(kNormRows, rows - r), 0, ctr(m, wait_k), wait_target,
            ctr(m, done_k));
    }
  };
  for (int m = 0; m < mt; ++m)
    for (int j = 0; j < s.W / kBnO; ++j)
      for (int z = 0; z < s.split_o; ++z) put(BK_OUT_PROJ, m, j, z, kNoCounter, 0, ctr(m, C_O));
  norms(BK_NORM_MID, C_O, (s.W / kBnO) * s.split_o, C_N2);
  for (int m = 0; m < mt; ++m)
    for (int j = 0; j < (2 * s.F) / kBnGU; ++j)
      put(BK_GATE_UP, m, j, 0, ctr(m, C_N2), groups(m), ctr(m, C_GU + j / gps));
  for (int m = 0; m < mt; ++m)
    for (int j = 0; j < s.W / kBnD; ++j)
      for (int z = 0; z < s.split_d; ++z)
        put(BK_DOWN, m, j, z, ctr(m, C_GU + z), gps, ctr(m, C_D));
  norms(BK_NORM_NEXT, C_D, (s.W / kBnD) * s.split_d, C_N1);
  if (s.next_qkv)
    for (int m = 0; m < mt; ++m)
      for (int j = 0; j < s.N_qkv / kBnQ; ++j)
        put(BK_QKV, m, j, 0, ctr(m, C_N1), groups(m), kNoCounter);
  *n_tasks = n;
}

cudaError_t block_kernel_init() {
  return cudaFuncSetAttribute(block_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              kSmemBytes);
}

cudaError_t launch_block_kernel(const BlockShape& s, const BlockLaunch& l, int grid,
                                cudaStream_t st) {
  if (!block_supported(s) || l.n_tasks <= 0) return cudaErrorInvalidValue;
  BlockParams p;
  memset(&p, 0, sizeof(p));
  const int bn[4] = {kBnO, kBnGU, kBnD, kBnQ};
  const int kbps[4] = {s.Dq / kBK / s.split_o, s.W / kBK, s.F / kBK / s.split_d, s.W / kBK};
  for (int i = 0; i < 4; ++i) {
    p.a[i] = *l.a[i];
    p.b[i] = *l.b[i];
    p.b_box[i] = l.b_box[i];
    p.bn[i] = bn[i];
    p.kb_per_split[i] = kbps[i];
    p.epi[i] = l.epi[i];
    if (bn[i] % l.b_box[i] != 0) return cudaErrorInvalidValue;
  }
  p.norm[0] = l.norm[0];
  p.norm[1] = l.norm[1];
  p.M = s.M;
  p.T = l.d.T;
  p.K = l.d.K;
  p.H = l.d.H;
  p.W = s.W;
  p.N_mod = l.d.N_mod;
  p.eps = l.d.eps;
  p.tasks = l.tasks;
  p.n_tasks = l.n_tasks;
  p.ctr = l.ctr;
  p.err = l.err;
  return launch_pdl(block_kernel, dim3(grid), dim3(kThreads), kSmemBytes, st, p);
}

}  // namespace fva
