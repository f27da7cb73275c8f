// Chunk-wise causal multi-query attention on tcgen05 (head_dim 256, bf16), split-KV.
//
// The paper's mask (§3.1): action token t of chunk c(t) = floor(t / H) attends to
// every prefix key of its request and to the action keys of chunks <= c(t)
// (bidirectional inside its own chunk).  In the concatenated key sequence
// [prefix ; action tokens] that is the leading range [0, P + (c(t)+1) H).
//
// Work decomposition.  A query tile is 128 rows = 128/nq consecutive tokens x
// all nq heads of one request: MQA heads share the single KV head, so one K/V
// tile in shared memory serves every head.  The key range of a tile is cut into
// splits of up to 256 keys (1-4 blocks of 64: fewer when there are few query
// tiles, so that more SMs take part); key blocks past the tile's largest limit
// are never loaded.  One CTA handles one (split, tile):
//   warp 0      TMA: the Q tile (64 KB) and the split's K blocks, then, once
//               the S MMAs have read K, the V blocks into the same space;
//   warp 1      TMEM (512 columns: S in 0..255, O in 256..511); one lane issues
//               S = Q K^T as one MMA per 16 head dims with N = all the split's
//               keys (each Q and K byte is read from shared memory once), and,
//               per key block, once its P is written, O += P V (M=128, N=256,
//               A = P from TMEM, MN-major V from shared memory);
//   warps 2..17 softmax + epilogue, four threads per query row (16 keys of every
//               block / 64 head-dim columns): block max, row max through shared
//               memory, P = exp(S - row max) as bf16 pairs written back over S's
//               TMEM columns (S is dead once every thread holds its values), with
//               the row's sum; then O from TMEM.
// K and V live slab-major: head-dim slab j (64 values, 128 bytes) of key k is
// at j * 32 KB + k * 128 bytes, so the split's keys form one uniformly strided
// operand for the S MMA and V's head-dim slabs are 32 KB apart for the P V MMA.
//
// Two ways to combine the splits of a tile (each split holds O_s / l_s in bf16
// with its row max m_s and sum l_s):
//   cluster form: the splits of a tile are one thread-block cluster of n CTAs; the
//     tile's key blocks are dealt out evenly (CTA s takes blocks
//     [s nkb / n, (s+1) nkb / n)), at most 4 per CTA.
//     Each CTA leaves its rows in its own shared memory; after a cluster barrier
//     CTA q combines rows [q 128/n, (q+1) 128/n) of every split, reading them
//     through distributed shared memory, and writes the bf16 output rows.
//     Nothing goes through global scratch and no second kernel runs.
//   global form (tiles with more splits than a cluster holds, and
//     fva_chunk_attention_noalloc): each split writes its rows and (m, l) to
//     global scratch and attn_merge_kernel combines them.
// Both combine in split order with the same arithmetic, so they give identical
// bits when they cut the keys at the same places.  A tile with one split writes
// O / l directly.
#include "common.cuh"
#include "kernels.h"

namespace fva {

namespace {

constexpr int kDH = 256;
constexpr int kRows = 128;
constexpr int kKB = kAttnKeyBlock;                        // 64 keys per block
constexpr int kBlocksPerSplit = kAttnKeysPerSplit / kKB;  // 4 K/V slots
static_assert(kBlocksPerSplit == kAttnMaxBlocksPerCta, "key blocks per CTA");
constexpr int kGroups = 4;  // softmax threads per query row (16 keys of every block each)
constexpr int kQBytes = kRows * kDH * 2;                  // 64 KB (Q, later P)
constexpr int kKVBytes = kKB * kDH * 2;                   // 32 KB per K or V block
constexpr int kSoftmaxThreads = 512;
constexpr int kThreads = 64 + kSoftmaxThreads;
constexpr int kSmem = kQBytes + kBlocksPerSplit * kKVBytes + 1024 /*align*/ + 1024 /*bars*/ +
                      8 * kRows * 4 /*row exchange*/ + kRows * 8 /*row (max, sum)*/;
// Largest cluster of the cluster form (the portable limit).
constexpr int kMaxClusterSplits = kAttnMaxClusterSplits;
constexpr uint32_t kTmemCols = 512;

__device__ __forceinline__ void softmax_bar() {
  asm volatile("bar.sync 1, 512;" ::: "memory");
}

// Row rr's 16-byte piece c of a split's staged output (cluster form) sits at piece
// c ^ (rr & 7) of its 512-byte row, so that the 32 rows a warp stages at once
// fall into different shared-memory banks.
__device__ __forceinline__ uint32_t stage_piece(int rr, int c) {
  return (uint32_t)rr * (kDH * 2) + (uint32_t)((c ^ (rr & 7)) << 4);
}

// Grid (tiles, splits, B).  kCluster: clusters of `splits` CTAs along y, one per
// query tile (the cluster form); otherwise the global form.
// 576 threads: 18 warps, 5 of them on two of the SM's four register files (16K
// registers each), so at most 96 registers a thread.
template <bool kCluster>
__global__ void __launch_bounds__(kThreads, 1)
    tc_attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmV, const AttnArgs a) {
  const int tile = blockIdx.x, split = blockIdx.y, r = blockIdx.z;
  const int tok_per_tile = kRows / a.nq;
  const int t0 = tile * tok_per_tile;
  const int t_last = min(a.T, t0 + tok_per_tile) - 1;
  const int P = __ldg(a.prefix_len + r);
  const int limit_max = attn_key_limit(P, t_last, a.H);
  const int nkb_tile = (limit_max + kKB - 1) / kKB;
  // splits of this tile: fixed-size ones (global form), or as many CTAs of the
  // cluster as the tile has key blocks, sharing them evenly (cluster form)
  const int bps = a.blocks_per_split > 0 ? min(a.blocks_per_split, kBlocksPerSplit) : kBlocksPerSplit;
  const int nsplit = kCluster ? min((int)gridDim.y, nkb_tile) : (nkb_tile + bps - 1) / bps;
  // a prefix length the KV rows cannot hold (its keys would run into the next
  // request's rows), more splits than the scratch holds or more key blocks than
  // the cluster takes: the tile is left unwritten and the error word records it
  const bool bad = P < 0 || P + a.T > a.S_cap ||
                   (kCluster ? nkb_tile > kBlocksPerSplit * (int)gridDim.y
                             : nsplit > a.max_splits);
  if (bad) {  // uniform over the tile, hence over its cluster
    if (split == 0 && threadIdx.x == 0) report_error(a.err, KERR_BAD_SHAPE);
    pdl_trigger();
    return;
  }
  // a split past the tile's last key block: nothing to compute (in the cluster
  // form the CTA still combines its share of the rows)
  const bool active = split < nsplit;
  if (!kCluster && !active) {
    pdl_trigger();
    return;
  }
  const int kb0 = kCluster ? split * nkb_tile / nsplit : split * bps;
  const int nblk = kCluster ? (split + 1) * nkb_tile / nsplit - kb0 : min(bps, nkb_tile - kb0);

  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sQP = smem;                      // 4 slabs [128 rows x 128 B]: Q
  uint8_t* sKV = smem + kQBytes;            // 4 slabs [256 keys x 128 B]: K, then V
  uint64_t* bars = (uint64_t*)(sKV + kBlocksPerSplit * kKVBytes);
  uint64_t* qk_full = bars + 0;   // [4]: head-dim slab j of Q and of every K block
  uint64_t* v_full = bars + 4;    // [4]: V of key block b
  uint64_t* k_free = bars + 8;    // the S MMAs have read K
  uint64_t* s_full = bars + 9;    // S is in TMEM
  uint64_t* o_full = bars + 10;
  uint64_t* p_full = bars + 11;   // [4]: P of key block b is in TMEM
  uint32_t* tmem_slot = (uint32_t*)(bars + 15);
  float* xmax = (float*)(bars + 128);   // [4][128] row max of each key quarter
  float* xsum = xmax + kGroups * kRows; // [4][128] row sum of each key quarter
  float2* sml = (float2*)(xsum + kGroups * kRows);  // [128] row (max, sum) of this split (cluster form)

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qrow0 = (r * a.T + t0) * a.nq;
  if (active) {
  if (threadIdx.x == 0) {
    for (int j = 0; j < 4; ++j) mbar_init(&qk_full[j], nblk + 1);  // Q slab + each K block's slab
    for (int b = 0; b < kBlocksPerSplit; ++b) mbar_init(&v_full[b], 1);
    mbar_init(k_free, 1);
    mbar_init(s_full, 1);
    for (int b = 0; b < kBlocksPerSplit; ++b) mbar_init(&p_full[b], kSoftmaxThreads / 32);
    mbar_init(o_full, 1);
    fence_barrier_init();
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
  }
  // Only one CTA of any tcgen05 kernel of this library fits on an SM (each uses
  // more than half of the shared memory), so this allocation never waits.
  if (warp == 1) tmem_alloc(tmem_slot, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tS = tmem, tO = tmem + 256;
  pdl_trigger();

  const int krow0 = a.kv_row0 + r * a.S_cap + kb0 * kKB;
  // blocks wholly inside the prefix of a request that shares another's prefix come
  // from that request's rows (same keys; the block that straddles P comes from this
  // request's own rows, which hold its copy of the prefix tail)
  const int src = a.prefix_src ? __ldg(a.prefix_src + r) : r;
  const int krow0_src = a.kv_row0 + src * a.S_cap + kb0 * kKB;

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer
    // Key blocks that lie wholly inside the prefix come from fva_set_prefix_kv,
    // not from the predecessor grid, so they are requested before waiting for
    // it; q and the action keys/values (written by the QKV projection) after.
    // Loads go out head-dim slab by slab, so the S MMAs of slab 0 can start
    // while later slabs are in flight.  Every other thread only runs behind
    // these loads.
    constexpr uint32_t kSlab = kBlocksPerSplit * kKB * 128;
    auto row_of = [&](int b) {
      return ((kb0 + b + 1) * kKB <= P ? krow0_src : krow0) + b * kKB;
    };
    auto load_k = [&](int j, int b) {
      mbar_arrive_expect_tx(&qk_full[j], kKB * 128);
      tma_load_2d(sKV + j * kSlab + b * (kKB * 128), &tmK, j * 64, row_of(b), &qk_full[j]);
    };
    int npre = 0;
    while (npre < nblk && (kb0 + npre + 1) * kKB <= P) ++npre;
    for (int j = 0; j < 4; ++j)
      for (int b = 0; b < npre; ++b) load_k(j, b);
    pdl_wait();
    for (int j = 0; j < 4; ++j) {
      mbar_arrive_expect_tx(&qk_full[j], kRows * 128);
      tma_load_2d(sQP + j * (kRows * 128), &tmQ, j * 64, qrow0, &qk_full[j]);
      for (int b = npre; b < nblk; ++b) load_k(j, b);
    }
    if (mbar_wait(k_free, 0, a.err, KERR_WAIT_MMA))
      for (int b = 0; b < nblk; ++b) {
        mbar_arrive_expect_tx(&v_full[b], kKVBytes);
        for (int j = 0; j < 4; ++j)
          tma_load_2d(sKV + j * kSlab + b * (kKB * 128), &tmV, j * 64, row_of(b), &v_full[b]);
      }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer
    const uint32_t idesc_s = umma_idesc_bf16(kRows, nblk * kKB, false);
    constexpr uint32_t idesc_o = umma_idesc_bf16(kRows, kDH, true);
    constexpr uint32_t kSlabK = kBlocksPerSplit * kKB * 128;  // 32 KB between head-dim slabs
    const uint64_t qd0 = umma_desc_sw128(smem_u32(sQP), 16, 1024);
    const uint64_t kd0 = umma_desc_sw128(smem_u32(sKV), 16, 1024);
    bool good = true;
    for (int j = 0; good && j < 4; ++j) {  // head-dim slab j: 4 steps of 16
      if (!mbar_wait(&qk_full[j], 0, a.err, KERR_WAIT_TMA)) {
        good = false;
        break;
      }
      tc_fence_after();
      const uint64_t ad = desc_advance(qd0, j * (kRows * 128));
      const uint64_t bd = desc_advance(kd0, j * kSlabK);
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)  // 16 bf16 = 32 bytes along K inside the 128-byte row
        umma_bf16(tS, ad + 2 * kk, bd + 2 * kk, idesc_s, (j > 0 || kk > 0) ? 1u : 0u);
    }
    if (good) {
      umma_commit(k_free);
      umma_commit(s_full);
    }
    const uint64_t vd0 = umma_desc_sw128(smem_u32(sKV), kSlabK, 1024);
    for (int j = 0; good && j < nblk; ++j) {
      // block j's P (written while the softmax threads still work on later
      // blocks) and V
      if (!mbar_wait(&p_full[j], 0, a.err, KERR_WAIT_SYNC) ||
          !mbar_wait(&v_full[j], 0, a.err, KERR_WAIT_TMA)) {
        good = false;
        break;
      }
      tc_fence_after();
      // P keys j*64 + 16 ks .. +15 from TMEM (bf16 pairs, 8 columns); V the same
      // keys, all 256 head dims: MN-major B operand whose 64-wide head-dim slabs
      // are kSlabK apart (16 keys = 2 KB further on per step).
      const uint64_t bv = desc_advance(vd0, j * kKB * 128);
#pragma unroll
      for (int ks = 0; ks < kKB / 16; ++ks)
        umma_bf16_ts(tO, tS + j * (kKB / 2) + ks * 8, bv + 128 * ks, idesc_o,
                     (j > 0 || ks > 0) ? 1u : 0u);
    }
    if (good) umma_commit(o_full);
  } else if (warp >= 2) {
    // ---------------- softmax + epilogue: thread (key quarter g, row) takes
    // keys 16g .. 16g+15 of every key block, block after block, so that block
    // j's P is complete (and its P V MMAs can start) while later blocks are
    // still being exponentiated; in the epilogue it takes O columns 64g .. +63.
    const int g = (warp - 2) >> 2;
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    const int t = t0 + row / a.nq;
    const bool valid = t < a.T;
    const int limit = valid ? attn_key_limit(P, t, a.H) : 0;
    // action keys in [P, P + lo) are padding (cold start) or, under the
    // block-diagonal mask, earlier chunks
    const int pad = a.pad_tokens ? __ldg(a.pad_tokens + r) : 0;
    const int lo = a.block_diag && valid ? max(pad, (t / a.H) * a.H) : pad;
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    bool good = __all_sync(0xffffffffu, mbar_wait(s_full, 0, a.err, KERR_WAIT_MMA));
    tc_fence_after();
    // visible keys of block j for this thread: i < nv[j] and not p_rel <= i < lo_rel
    auto key_vis = [&](int j, int i) {
      const int key = (kb0 + j) * kKB + g * 16 + i;
      return key < limit && (key < P || key >= P + lo);
    };
    auto block_all_vis = [&](int j) {
      const int k0 = (kb0 + j) * kKB + g * 16;
      return k0 + 16 <= limit && (k0 + 16 <= P || k0 >= P + lo);
    };
    float mx = -INFINITY;
    uint32_t sv[kBlocksPerSplit][16];
    if (good) {
#pragma unroll
      for (int j = 0; j < kBlocksPerSplit; ++j)
        if (j < nblk) tmem_ld16_nowait(tS + lane_off + j * kKB + g * 16, sv[j]);
      tmem_ld_wait();
#pragma unroll
      for (int j = 0; j < kBlocksPerSplit; ++j) {
        if (j >= nblk) break;
        if (block_all_vis(j)) {
#pragma unroll
          for (int i = 0; i < 16; ++i) mx = fmaxf(mx, __uint_as_float(sv[j][i]));
        } else {
#pragma unroll
          for (int i = 0; i < 16; ++i)
            if (key_vis(j, i)) mx = fmaxf(mx, __uint_as_float(sv[j][i]));
        }
      }
    }
    xmax[g * kRows + row] = mx;
    // every thread holds its S values past this barrier, so P may go over S's
    // TMEM columns
    softmax_bar();
    float mrow = xmax[row];
#pragma unroll
    for (int j = 1; j < kGroups; ++j) mrow = fmaxf(mrow, xmax[j * kRows + row]);
    const float mscaled = mrow > -INFINITY ? mrow * a.scale_log2 : 0.f;
    float l2[2] = {0.f, 0.f};
#pragma unroll
    for (int j = 0; j < kBlocksPerSplit; ++j) {
      if (j >= nblk) break;
      if (good) {
        // P = exp(S - row max) over visible keys, rounded to bf16 (the row sum
        // adds the rounded values the P V MMA uses)
        const bool all_vis = block_all_vis(j);
        uint32_t w[8];
#pragma unroll
        for (int i = 0; i < 16; i += 2) {
          float e0 = ex2_approx(fmaf(__uint_as_float(sv[j][i]), a.scale_log2, -mscaled));
          float e1 = ex2_approx(fmaf(__uint_as_float(sv[j][i + 1]), a.scale_log2, -mscaled));
          if (!all_vis) {
            if (!key_vis(j, i)) e0 = 0.f;
            if (!key_vis(j, i + 1)) e1 = 0.f;
          }
          const __nv_bfloat162 b2 = __floats2bfloat162_rn(e0, e1);
          w[i / 2] = *reinterpret_cast<const uint32_t*>(&b2);
          l2[0] += __uint_as_float(w[i / 2] << 16);
          l2[1] += __uint_as_float(w[i / 2] & 0xFFFF0000u);
        }
        // P of keys j*64 + 16g .. +15 over S's (already read) TMEM columns, as
        // the A operand of the P V MMAs
        tmem_st8(tS + lane_off + j * (kKB / 2) + g * 8, w);
        tmem_st_wait();
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[j]);
    }
    float l = l2[0] + l2[1];
    xsum[g * kRows + row] = l;
    mx = mrow;
    if (good) good = __all_sync(0xffffffffu, mbar_wait(o_full, 0, a.err, KERR_WAIT_MMA));
    tc_fence_after();
    softmax_bar();  // every quarter's sum is in xsum
    l = 0.f;
#pragma unroll
    for (int j = 0; j < kGroups; ++j) l += xsum[j * kRows + row];
    const int gtile = r * a.tiles_per_req + tile;
    const int grow = qrow0 + row;  // global q row = (r*T + t) * nq + head
    const int c0 = g * 64;         // O columns of this thread
    if (good) {
      uint32_t ov[64];
      uint32_t (&o0)[32] = *reinterpret_cast<uint32_t(*)[32]>(&ov[0]);
      uint32_t (&o1)[32] = *reinterpret_cast<uint32_t(*)[32]>(&ov[32]);
      tmem_ld32_nowait(tO + lane_off + c0, o0);
      tmem_ld32_nowait(tO + lane_off + c0 + 32, o1);
      tmem_ld_wait();
      // Q and K/V are dead once O is complete: each warp stages its 32 rows
      // there for coalesced stores
      uint8_t* stage = smem + (warp - 2) * (32 * 144);
      // one split: the output row; several: this split's partial (O / l, with
      // max and sum) for attn_merge_kernel
      const float inv = l > 0.f ? 1.f / l : 0.f;
      uint4 pk[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        float v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) v[u] = __uint_as_float(ov[8 * i + u]) * inv;
        pk[i] = pack_bf16x8(v);
      }
      if (kCluster && nsplit > 1) {
        // cluster form: the rows stay in this CTA's shared memory (Q is dead)
        // for the combination after the cluster barrier
#pragma unroll
        for (int i = 0; i < 8; ++i)
          *reinterpret_cast<uint4*>(sQP + stage_piece(row, g * 8 + i)) = pk[i];
        if (g == 0) sml[row] = make_float2(mx, l);
      } else {
        const size_t prow_idx = ((size_t)gtile * a.max_splits + split) * kRows + row;
        bf16* dst = nsplit == 1 ? (bf16*)a.out + (size_t)grow * kDH + c0
                                : (bf16*)a.part_o + prow_idx * kDH + c0;
        warp_store_rows<128>(stage, pk, valid ? dst : nullptr, lane);
        if (nsplit > 1 && valid && g == 0) __stcg(a.part_ml + prow_idx, make_float2(mx, l));
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
  } else {
    // inactive split of the cluster form: its output rows come after the QKV
    // projection's reads of them are over
    pdl_trigger();
    pdl_wait();
  }
  if constexpr (kCluster) {
    if (nsplit > 1) {
      // every split's rows and (max, sum) are staged (release / acquire across the
      // cluster); CTA `split` then combines rows [split 128/n, (split+1) 128/n)
      // with attn_merge_kernel's arithmetic, reading the splits through
      // distributed shared memory, one warp per row and 8 head dims per lane
      cluster_sync();
      const int ncl = gridDim.y;  // the cluster: this tile's CTAs, ranks 0..ncl-1 = split
      const int r_lo = split * kRows / ncl, r_hi = (split + 1) * kRows / ncl;
      for (int rr = r_lo + warp; rr < r_hi; rr += kThreads / 32) {
        if (t0 + rr / a.nq >= a.T) break;  // rows past the last token
        float2 ml = make_float2(-INFINITY, 0.f);
        if (lane < nsplit) ml = ld_shared_cluster_f2(mapa_shared(smem_u32(&sml[rr]), (uint32_t)lane));
        const uint32_t piece = smem_u32(sQP + stage_piece(rr, lane));
        uint4 x[kMaxClusterSplits];
#pragma unroll
        for (int u = 0; u < kMaxClusterSplits; ++u)
          if (u < nsplit) x[u] = ld_shared_cluster_v4(mapa_shared(piece, (uint32_t)u));
        const float m_all = warp_max(ml.y > 0.f ? ml.x : -INFINITY);
        // each split holds O_s / l_s; its weight is 2^((m_s - m) c) l_s
        const float w = ml.y > 0.f ? exp2f((ml.x - m_all) * a.scale_log2) * ml.y : 0.f;
        const float tot = warp_sum(w);
        const float inv = tot > 0.f ? 1.f / tot : 0.f;  // no visible key in any split: zeros
        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int u = 0; u < kMaxClusterSplits; ++u) {
          const float wu = __shfl_sync(0xffffffffu, w, u);
          if (u < nsplit) {
            const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&x[u]);
#pragma unroll
            for (int q2 = 0; q2 < 4; ++q2) {
              const float2 f = __bfloat1622float2(h2[q2]);
              acc[2 * q2] = fmaf(wu, f.x, acc[2 * q2]);
              acc[2 * q2 + 1] = fmaf(wu, f.y, acc[2 * q2 + 1]);
            }
          }
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] *= inv;
        *reinterpret_cast<uint4*>((bf16*)a.out + (size_t)(qrow0 + rr) * kDH + lane * 8) =
            pack_bf16x8(acc);
      }
      // no CTA leaves (releasing its shared memory) while another still reads it
      cluster_sync();
    }
  }
}

// Combine the key splits of every query row of tiles that have more than one.
// Split s stored o_s = O_s / l_s with its (m_s, l_s); with w_s = 2^((m_s - m) c) l_s,
// m = max over splits with keys, c = log2(e)/sqrt(dh):  o = sum_s w_s o_s / sum_s w_s,
// splits in order.  One warp per row, 8 dh
// values per lane.
__global__ void __launch_bounds__(256) attn_merge_kernel(const AttnArgs a) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gtile = blockIdx.x, r = blockIdx.y;
  const int row = blockIdx.z * 8 + warp;
  const int tok_per_tile = kRows / a.nq;
  const int t0 = gtile * tok_per_tile;
  pdl_trigger();
  const int t_last = min(a.T, t0 + tok_per_tile) - 1;
  const int t = t0 + row / a.nq;
  if (t >= a.T) return;
  pdl_wait();
  const int P = __ldg(a.prefix_len + r);
  const int nkb_tile = (attn_key_limit(P, t_last, a.H) + kKB - 1) / kKB;
  const int bps = a.blocks_per_split > 0 ? min(a.blocks_per_split, kBlocksPerSplit) : kBlocksPerSplit;
  const int nsplit = (nkb_tile + bps - 1) / bps;
  // written by the attention kernel, or a bad size it left unwritten
  if (nsplit <= 1 || nsplit > a.max_splits || P < 0 || P + a.T > a.S_cap) return;
  const size_t tbase = (size_t)(r * a.tiles_per_req + gtile) * a.max_splits;
  // the first 8 splits' partial rows are requested together with the (max, sum)
  // pairs, so both round trips overlap
  uint4 x[8];
#pragma unroll
  for (int u = 0; u < 8; ++u)
    if (u < nsplit)
      x[u] = __ldcg(reinterpret_cast<const uint4*>(
          (const bf16*)a.part_o + ((tbase + u) * kRows + row) * kDH + lane * 8));
  float2 ml = make_float2(-INFINITY, 0.f);
  if (lane < nsplit) ml = __ldcg(a.part_ml + (tbase + lane) * kRows + row);
  float m_all = warp_max(ml.y > 0.f ? ml.x : -INFINITY);
  // each split stored O_s / l_s; its weight is 2^((m_s - m) c) l_s
  const float w = ml.y > 0.f ? exp2f((ml.x - m_all) * a.scale_log2) * ml.y : 0.f;
  const float tot = warp_sum(w);
  const float inv = tot > 0.f ? 1.f / tot : 0.f;  // no visible key in any split: zeros
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  for (int s0 = 0; s0 < nsplit; s0 += 8) {  // up to 8 splits' loads in flight
    float ws[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      ws[u] = __shfl_sync(0xffffffffu, w, (s0 + u) & 31);
      if (s0 > 0 && s0 + u < nsplit)
        x[u] = __ldcg(reinterpret_cast<const uint4*>(
            (const bf16*)a.part_o + ((tbase + s0 + u) * kRows + row) * kDH + lane * 8));
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      if (s0 + u < nsplit) {
        const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&x[u]);
#pragma unroll
        for (int q2 = 0; q2 < 4; ++q2) {
          const float2 f = __bfloat1622float2(h2[q2]);
          acc[2 * q2] = fmaf(ws[u], f.x, acc[2 * q2]);
          acc[2 * q2 + 1] = fmaf(ws[u], f.y, acc[2 * q2 + 1]);
        }
      }
    }
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) acc[i] *= inv;
  const size_t grow = (size_t)(r * a.T + t0) * a.nq + row;
  *reinterpret_cast<uint4*>((bf16*)a.out + grow * kDH + lane * 8) = pack_bf16x8(acc);
}

}  // namespace

cudaError_t tc_attention_init() {
  cudaError_t e = cudaFuncSetAttribute(tc_attn_kernel<false>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(tc_attn_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kSmem);
  return e;
}

int attn_cluster_capacity(int splits) {
  if (splits < 1 || splits > kMaxClusterSplits) return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(1, splits, 1);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = splits;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, tc_attn_kernel<true>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

cudaError_t launch_tc_attention(const CUtensorMap* q, const CUtensorMap* k,
                                const CUtensorMap* v, const AttnArgs& a, int B,
                                cudaStream_t s, bool cluster) {
  if (cluster) {
    if (a.max_splits < 1 || a.max_splits > kMaxClusterSplits) return cudaErrorInvalidValue;
    return launch_pdl_cluster(tc_attn_kernel<true>, dim3(a.tiles_per_req, a.max_splits, B),
                              dim3(kThreads), kSmem, s, dim3(1, a.max_splits, 1), *q, *k, *v, a);
  }
  if (a.max_splits > 32) return cudaErrorInvalidValue;  // the merge holds one split per lane
  return launch_pdl(tc_attn_kernel<false>, dim3(a.tiles_per_req, a.max_splits, B),
                    dim3(kThreads), kSmem, s, *q, *k, *v, a);
}

cudaError_t launch_attn_merge(const AttnArgs& a, int B, cudaStream_t s) {
  if (a.max_splits == 1) return cudaSuccess;
  return launch_pdl(attn_merge_kernel, dim3(a.tiles_per_req, B, kRows / 8), dim3(256), 0, s, a);
}

}  // namespace fva
