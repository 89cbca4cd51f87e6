// LM head of the multi-kernel step, on CTA pairs (tcgen05 cta_group::2): the
// same quantities as lm_head_softmax_kernel (Box 1 of arXiv 2608.22646:
// c_i = max_v p_theta(x_i = v) and argmax_v p_theta, logits never leaving
// tensor memory), for any number M >= 1 of masked rows, in one of two
// orientations chosen per step from M (pair_swapped).
//
// Unswapped, for wide steps: with hundreds to thousands of rows the
// contraction is tensor-bound (2 V H M flops against 2 V H bytes of W), so
// the masked rows fill the MMA M dimension and the vocabulary the N
// dimension.  One tcgen05.mma of the pair computes a 256 x 256 tile: each CTA
// holds 128 of the rows (its A half) and 128 of the vocabulary rows (its B
// half) per K block, and keeps its 128 x 256 half of the accumulator in
// tensor memory.  Per K block a CTA loads 32 KiB (16 KiB of hidden rows,
// 16 KiB of W) for 2 * 128 * 256 * 64 flops, half the shared-memory traffic
// per flop of a single-CTA 128 x 256 tile.  A tensor-memory lane holds one
// row's logits, so the epilogue is a serial online softmax per thread over
// the 256 columns of a tile, no shuffles.
//
// Swapped, for narrow steps: the vocabulary fills the MMA M dimension (256
// rows per pair, 128 per CTA: the W half is the A operand) and the masked
// rows the N dimension.  The M rows are split into n_rt = ceil(M / 256) row
// tiles of equal width N (a multiple of 32, at most 256), so a step pads at
// most 31 rows per tile instead of up to 255: M = 305 runs as two 160-column
// tiles, M = 159 as one of 160, M = 5 as one of 32.  A tensor-memory lane
// then holds one vocabulary row of every column; the epilogue reduces across
// lanes (transpose_logits32) and across the four epilogue warps (a
// shared-memory exchange), and each CTA writes the triples of its 128
// vocabulary rows: two partials per pair.  Each CTA loads N / 2 of a tile's
// rows per K block as one box of exactly that many rows.  The cross-lane
// reduction costs more than the serial one, so wide tiles stay unswapped: a
// step runs swapped when N is at most swap_max_n (192 by default; measured
// per step on the Dream shape: N = 64..192 3 to 11 % faster than the padded
// unswapped tile, N = 224, 256 1 to 7 % slower).
//
// Partials: when the number of pairs is a multiple of the number of row
// tiles n_rt, every tile of a pair has the same row tile, and the epilogue
// folds its tiles into one partial (max * log2 e, sum of 2^(z log2 e - max),
// argmax) per row and pair (and CTA, swapped), which the commit reads
// directly (pair_partials_per_row); otherwise it writes one partial per row
// and vocabulary tile (and CTA), merged per row by reduce_partials_kernel.
//
// Work: tiles (v, j) of 256 vocabulary rows x one row tile, numbered
// t = v * n_rt + j and dealt round-robin to the pairs of a persistent grid.
// The pairs working at one time share few W tiles, each read from HBM once
// and by the n_rt pairs of its row tiles from L2; the gathered hidden rows
// (at most 2 x 65536 x 16384 bytes, in practice tens of MB) stay in L2.
//
// Roles per CTA (192 threads): warp 0 producer (hidden half and W half by
// TMA; W from a tile-major packed copy in which every box is one contiguous
// 16 KiB block); warp 1 allocates tensor memory and, in the even CTA, issues
// the MMAs; warps 2..5 epilogue.  Both CTAs' copies of a stage complete on
// the even CTA's barrier (cta_group::2 loads), which the even CTA's producer
// arms with the bytes of both.  Two accumulator buffers let the epilogue of
// one tile overlap the next tile's MMAs.
//
// What bounds a step: reading W from HBM with one row tile; with two or more,
// the MMAs.  The tensor core runs the MMAs of the one issuing thread one after
// another, about 63 + 0.085 N ns each (M = 256, K = 16, measured on GB300),
// so a 160-column tile costs nearly as much per K block as a 256-column one
// and two row tiles take twice one; each orientation issues the fewest MMAs
// its M allows (ceil(M / 256) per vocabulary tile and K slice).  A second
// issuing thread would run MMAs side by side, but two threads accumulating
// into one accumulator do so in no fixed order, and the fp32 logits (and the
// commit decisions at a threshold) would then change from run to run.
#pragma once

#include <climits>
#include "head_kernel.cuh"
#include "ptx.cuh"
#include "softmax.cuh"

namespace cai {

constexpr int kPairThreads = 192;
constexpr int kPairTileRows = 256;    // masked rows per pair tile (MMA M)
constexpr int kPairTileVocab = 256;   // vocabulary rows per pair tile (MMA N)
constexpr int kPairHalf = 128;        // rows of each per CTA
constexpr int kPairBlockK = 64;       // K per stage (one 128-byte swizzled row)
constexpr int kPairHalfBytes = kPairHalf * kPairBlockK * 2;  // 16 KiB
constexpr int kPairStageBytes = 2 * kPairHalfBytes;          // A half + B half
constexpr int kPairTmemCols = 2 * kPairTileVocab;            // two accumulators
constexpr int kSwapColStep = 32;    // swapped orientation: granularity of N
constexpr int kSwapXchBytes = 2 * 4 * kPairTileVocab * 16;  // cross-warp exchange, two buffers
constexpr int kPairMaxRing = 12;    // swapped stages are cut to size: up to this many

// Tensor maps of the gathered rows with boxes of 16, 32, ..., 128 rows
// (swapped orientation: a CTA's N / 2 rows of a tile, a multiple of 16, load
// as one exact box: each TMA copy has a fixed cost, and every byte written
// to shared memory competes with the MMAs' operand reads).
struct PairRowMaps {
  CUtensorMap box[8];  // box[q]: 16 (q + 1) rows
};

struct PairParams {
  const int* d_M;      // masked rows of this step (device)
  int* m_hist_slot;    // where this step's M is recorded, or null
  float4* part;        // [rows, n_vt] partial per row and vocabulary tile
  uint32_t* err;
  int V, H;
  int n_vt;            // ceil(V / 256)
  int min_M;           // smaller steps are left to lm_head_softmax_kernel (<= 1: this
                       // kernel decodes every step and records M = 0 too)
  int swap_max_n;      // steps whose swapped tile width is at most this run swapped
  int n_stages;
  const float* inv_r;  // final-norm row scales [rows] (kNorm only)
  int ring_max;        // most stages in flight (<= kPairMaxRing)
};

// Row tiles of a pair step with M rows (both orientations).
__host__ __device__ inline int pair_row_tiles(int M) {
  return (M + kPairTileRows - 1) / kPairTileRows;
}

// Swapped orientation: width N of each of the n_rt row tiles; tile j covers
// rows [j N, j N + N), the last one possibly past M (padding, never written).
__host__ __device__ inline int swap_tile_cols(int M, int n_rt) {
  const int per = (M + n_rt - 1) / n_rt;
  return (per + kSwapColStep - 1) / kSwapColStep * kSwapColStep;
}

// Orientation of a pair step with M rows: swapped when the tile width of the
// swapped orientation is at most swap_max_n (0: never).
__host__ __device__ inline bool pair_swapped(int M, int swap_max_n) {
  return M > 0 && swap_tile_cols(M, pair_row_tiles(M)) <= swap_max_n;
}

// Partials per row written by a pair step with M rows on n_pairs pairs: one
// per pair of the row's tile (two in the swapped orientation, one per CTA)
// when n_pairs is a multiple of the row-tile count, else 0 (one per
// vocabulary tile, two when swapped, merged by the reduce kernel).
__host__ __device__ inline int pair_partials_per_row(int M, int n_pairs, bool swap) {
  const int n_rt = pair_row_tiles(M);
  if (n_rt <= 0 || n_pairs % n_rt != 0) return 0;
  return (swap ? 2 : 1) * (n_pairs / n_rt);
}

__host__ __device__ inline size_t pair_smem_bytes(int n_stages, bool swap) {
  return 1024 + static_cast<size_t>(n_stages) * kPairStageBytes + (swap ? kSwapXchBytes : 0) +
         static_cast<size_t>(2 * kPairMaxRing + 7) * 8 + 16;
}

// Pack W [V, H] (row-major bf16) tile-major for the pair kernel: 128-row
// tile t, K block kb is the 16 KiB block at (t * (H / 64) + kb) * 16 KiB, in
// the 128-byte-swizzled K-major layout (row r's 16-byte chunk c at
// r * 128 + (c ^ (r & 7)) * 16).  Rows >= V are zero; n_tiles = 2 n_vt.  The
// kernel reads it through a tensor map of [2 n_vt (H / 64) 128, 64] bf16 with
// 64 x 128 boxes and no swizzle: box (t (H / 64) + kb) is that block.
__global__ void pack_w_tiles_kernel(const uint4* __restrict__ W, uint4* __restrict__ out, int V,
                                    int H, long long n_chunks, const __nv_bfloat16* __restrict__ gw) {
  const int KB = H / kPairBlockK;
  const long long tile_chunks = static_cast<long long>(KB) * (kPairHalfBytes / 16);
  for (long long d = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; d < n_chunks;
       d += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long t = d / tile_chunks;
    const int rem = static_cast<int>(d - t * tile_chunks);
    const int kb = rem / (kPairHalfBytes / 16);
    const int inblk = rem % (kPairHalfBytes / 16);  // 16-byte chunk in the block
    const int r = inblk >> 3;
    const int cl = (inblk & 7) ^ (r & 7);
    const long long v = t * kPairHalf + r;
    uint4 val = make_uint4(0u, 0u, 0u, 0u);
    if (v < V) val = W[(v * H + static_cast<long long>(kb) * kPairBlockK) / 8 + cl];
    if (gw) val = scale_chunk(val, gw + kb * kPairBlockK + cl * 8);
    out[d] = val;
  }
}

struct PairSmem {
  uint8_t* stage;      // n_stages x kPairStageBytes: the ring (A half, B half per stage)
  float4* xch;         // swapped orientation: 2 x [4 warps][256 columns] triples
  uint64_t* full;      // kPairMaxRing (even CTA): both CTAs' halves of the stage landed
  uint64_t* empty;     // kPairMaxRing: the pair's MMAs are done with the stage
  uint64_t* accf;      // 2: accumulator ready
  uint64_t* acce;      // 2 (even CTA): accumulator drained by both epilogues
  uint64_t* drain;     // 1 (even CTA): abort path, issued MMAs complete
  uint64_t* xchb;      // 2 (swapped): the four epilogue warps wrote xch[buffer]
  uint32_t* tmem_slot;
  volatile int* abort;
};

__device__ __forceinline__ PairSmem pair_carve(uint8_t* raw, int n_stages, bool swap) {
  PairSmem s;
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  s.stage = base;
  uint8_t* after = base + static_cast<size_t>(n_stages) * kPairStageBytes;
  s.xch = reinterpret_cast<float4*>(after);
  if (swap) after += kSwapXchBytes;
  s.full = reinterpret_cast<uint64_t*>(after);
  s.empty = s.full + kPairMaxRing;
  s.accf = s.empty + kPairMaxRing;
  s.acce = s.accf + 2;
  s.drain = s.acce + 2;
  s.xchb = s.drain + 1;
  s.tmem_slot = reinterpret_cast<uint32_t*>(s.xchb + 2);
  s.abort = reinterpret_cast<volatile int*>(s.tmem_slot + 1);
  return s;
}

struct PairRing {
  int slot = 0;
  uint32_t phase = 0;
  __device__ void next(int n) {
    if (++slot == n) {
      slot = 0;
      phase ^= 1u;
    }
  }
};

__device__ __forceinline__ void pair_drain(uint64_t* bar, uint32_t parity, uint32_t* err) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > kWaitLimitNs) {
      atomicOr(err, kErrDrain);
      return;
    }
  }
}

// kNorm: as in lm_head_softmax_kernel, row n's logits are scaled by inv_r[n]
// (written by the gather).  Swapped steps (pair_swapped) load a tile's rows
// through hm instead of tm_a.
template <bool kNorm>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kPairThreads, 1)
    lm_head_pair_kernel(const __grid_constant__ CUtensorMap tm_a,
                        const __grid_constant__ CUtensorMap tm_w,
                        const __grid_constant__ PairRowMaps hm, const PairParams p) {
  extern __shared__ uint8_t smem_raw[];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();  // 0: even CTA (issues the MMAs), 1: odd
  const int pair = blockIdx.x >> 1;
  const int n_pairs = gridDim.x >> 1;

  grid_dependency_wait();    // d_M and the gathered rows of this step
  // Every thread (the CTA counts once all of them have), after the wait: the
  // commit kernel, which may start from here, reads the previous step's state
  // before waiting for this kernel.
  grid_launch_dependents();
  const int M = *p.d_M;
  if (p.m_hist_slot && blockIdx.x == 0 && threadIdx.x == 0 && (M >= p.min_M || p.min_M <= 1))
    *p.m_hist_slot = M;
  if (M < p.min_M || M < 1) return;  // both CTAs of every pair take the same branch
  const bool swap = pair_swapped(M, p.swap_max_n);  // the same in every CTA

  PairSmem sm = pair_carve(smem_raw, p.n_stages, p.swap_max_n > 0);
  const int KB = p.H / kPairBlockK;
  const int n_rt = pair_row_tiles(M);
  // Rows per row tile: 256 (the MMA M of the pair), or N when swapped.
  const int rt_rows = swap ? swap_tile_cols(M, n_rt) : kPairTileRows;
  const int n_tiles = p.n_vt * n_rt;
  const int my_tiles = pair < n_tiles ? (n_tiles - pair + n_pairs - 1) / n_pairs : 0;
  // Swapped stages hold the W half and one box of rows_tile / 2 rows, so the
  // ring (n_stages slots of kPairStageBytes) is re-cut to that size: more
  // stages in flight for narrower tiles.  Unswapped steps do not use the
  // swapped epilogue's exchange buffer, which follows the ring: one more stage.
  const int stage_stride =
      swap ? kPairHalfBytes + (rt_rows / 2) * kPairBlockK * 2 : kPairStageBytes;
  const int ring_bytes =
      p.n_stages * kPairStageBytes + (!swap && p.swap_max_n > 0 ? kSwapXchBytes : 0);
  const int n_ring = min(p.ring_max, ring_bytes / stage_stride);

  if (threadIdx.x == 0) {
    for (int s = 0; s < n_ring; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&sm.accf[a], 1);
      mbar_init(&sm.acce[a], 8);  // four epilogue warps in each CTA
    }
    mbar_init(sm.drain, 1);
    if (swap) {
      mbar_init(&sm.xchb[0], 4);  // the four epilogue warps of this CTA
      mbar_init(&sm.xchb[1], 4);
    }
    *sm.abort = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&tm_w);
    if (swap) {
      prefetch_tmap(&hm.box[swap_tile_cols(M, n_rt) / 32 - 1]);
    } else {
      prefetch_tmap(&tm_a);
    }
  }
  if (warp == 1) {
    tmem_alloc_pair(sm.tmem_slot, kPairTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();  // barriers of both CTAs initialised, tensor memory allocated
  tc_fence_after();
  const uint32_t tmem_base = *sm.tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------ producer --
      const uint64_t pol_a = policy_evict_last();
      const uint32_t full0 = mapa_shared(sm.full, 0);  // the even CTA's barriers
      PairRing r;
      long long issued = 0;
      bool ok = true;
      // Swapped: a CTA's rt_rows / 2 rows (a multiple of 16) load as one box.
      const int q1 = rt_rows / 32 - 1;
      const int box_rows = rt_rows / 2;
      // Bytes of one stage, both CTAs (the even CTA arms its barrier for them).
      const uint32_t stage_tx =
          swap ? 2u * static_cast<uint32_t>(kPairHalfBytes + box_rows * kPairBlockK * 2)
                : 2u * kPairStageBytes;
      for (int i = 0; i < my_tiles && ok; ++i) {
        const int t = pair + i * n_pairs;
        const int v = t / n_rt, j = t - v * n_rt;
        // First row of this CTA's half of the tile's rows.
        const int a_row = j * rt_rows + static_cast<int>(rank) * (swap ? rt_rows / 2 : kPairHalf);
        const int w_box = (2 * v + static_cast<int>(rank)) * KB;
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(&sm.empty[r.slot], r.phase ^ 1u, sm.abort, p.err, kErrWaitEmpty)) {
            ok = false;
            break;
          }
          uint8_t* dst = sm.stage + static_cast<size_t>(r.slot) * stage_stride;
          const uint32_t bar = full0 + static_cast<uint32_t>(r.slot * 8);
          // The even CTA arms the stage for the bytes of both CTAs; a copy of
          // the odd CTA that completes first leaves the phase open until then.
          if (rank == 0) mbar_arrive_expect_tx(&sm.full[r.slot], stage_tx);
          if (swap) {
            // A: the W half; B: the CTA's rows, one box of box_rows.
            tma_load_2d_pair_nohint(dst, &tm_w, bar, 0, (w_box + kb) * kPairHalf);
            tma_load_2d_pair(dst + kPairHalfBytes, &hm.box[q1], bar, kb * kPairBlockK, a_row, pol_a);
          } else {
            tma_load_2d_pair(dst, &tm_a, bar, kb * kPairBlockK, a_row, pol_a);
            tma_load_2d_pair_nohint(dst + kPairHalfBytes, &tm_w, bar, 0, (w_box + kb) * kPairHalf);
          }
          ++issued;
          r.next(n_ring);
        }
      }
      if (!ok && rank == 0) {
        const long long f0 = issued > n_ring ? issued - n_ring : 0;
        for (long long q = f0; q < issued; ++q)
          pair_drain(&sm.full[q % n_ring], static_cast<uint32_t>((q / n_ring) & 1), p.err);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      // -------------------------------------------- MMA issuer (even CTA) --
      // Swapped: M = 256 vocabulary rows, N = the tile's rows; else M = 256
      // rows, N = 256 vocabulary rows.
      const uint32_t idesc =
          idesc_bf16_f32(256, swap ? static_cast<uint32_t>(rt_rows) : kPairTileVocab);
      PairRing r;
      bool ok = true;
      for (int i = 0; i < my_tiles && ok; ++i) {
        const int acc = i & 1;
        if (!mbar_wait_cluster(&sm.acce[acc], ((i >> 1) & 1) ^ 1u, sm.abort, p.err,
                               kErrWaitAccEmpty)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * kPairTileVocab);
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait_cluster(&sm.full[r.slot], r.phase, sm.abort, p.err, kErrWaitFull)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_addr = smem_addr(sm.stage + static_cast<size_t>(r.slot) * stage_stride);
          const uint32_t b_addr = a_addr + kPairHalfBytes;
#pragma unroll
          for (int kk = 0; kk < kPairBlockK / 16; ++kk)
            mma_bf16_pair(d_tmem, sdesc_k_sw128(a_addr + kk * 32), sdesc_k_sw128(b_addr + kk * 32),
                          idesc, (kb | kk) != 0 ? 1u : 0u);
          mma_commit_pair(&sm.empty[r.slot], 0x3);
          r.next(n_ring);
        }
        if (!ok) break;
        mma_commit_pair(&sm.accf[acc], 0x3);
      }
      if (!ok) {
        // Abort: wait for the MMAs already issued (they read both CTAs'
        // shared memory) before anything is released.
        mma_commit_pair(sm.drain, 0x1);
        pair_drain(sm.drain, 0, p.err);
      }
    }
    __syncwarp();
  } else if (swap) {
    // ----------------------------------------------- epilogue (swapped) --
    // Lane l of warp `quarter` holds vocabulary row 256 v + 128 rank + 32
    // quarter + l of all rt_rows columns (the tile's rows).  Per 32 columns the
    // warp's 32 rows are merged across lanes (lane l then holds column l), the
    // four warps' slices through xch, and thread et of the four warps keeps
    // columns et and et + 128.
    const int quarter = warp & 3;  // tensor-memory lanes 32 quarter .. 32 quarter + 31
    const int ew = warp - 2;       // 0..3: slot in the cross-warp exchange
    const int et = ew * 32 + lane;
    const uint32_t lane_base = static_cast<uint32_t>(quarter * 32) << 16;
    const uint32_t acce_remote = mapa_shared(sm.acce, 0);
    const int per_row = pair_partials_per_row(M, n_pairs, true);  // > 0: two partials per pair
    const int nch = rt_rows / 32;
    float am[2] = {kNegBig, kNegBig}, as[2] = {0.0f, 0.0f};
    int aix[2] = {INT_MAX, INT_MAX};
    for (int i = 0; i < my_tiles; ++i) {
      const int t = pair + i * n_pairs;
      const int v = t / n_rt, j = t - v * n_rt;
      const int acc = i & 1;
      if (!mbar_wait(&sm.accf[acc], (i >> 1) & 1, sm.abort, p.err, kErrWaitAccFull)) break;
      tc_fence_after();
      const uint32_t tbase = tmem_base + lane_base + static_cast<uint32_t>(acc * kPairTileVocab);
      const int vrow = v * kPairTileVocab + static_cast<int>(rank) * kPairHalf + quarter * 32 + lane;
      const bool valid = vrow < p.V;  // vocabulary rows past V are zero padding
      const bool pvalid = (vrow ^ 16) < p.V;
      const int row0 = j * rt_rows;
      // Buffer i & 1 is written again at tile i + 2, after every warp has
      // arrived for tile i + 1, which each does after reading tile i.  One
      // chunk of 32 columns at a time (the reduction is not unrolled over
      // chunks: its code stays small enough for the instruction cache).
      float4* xb = sm.xch + (i & 1) * 4 * kPairTileVocab;
#pragma unroll 1
      for (int c = 0; c < nch; ++c) {
        uint32_t x[32];
        tmem_ld_32cols(tbase + static_cast<uint32_t>(32 * c), x);
        tmem_ld_wait();
        float z[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          float sc = kLog2e;
          if constexpr (kNorm) {
            const int row = row0 + 32 * c + k;
            if (row < M) sc = kLog2e * __ldg(p.inv_r + row);
          }
          z[k] = valid ? __uint_as_float(x[k]) * sc : kNegBig;
        }
        float m, s;
        int ix;
        transpose_logits32(z, valid, pvalid, vrow, lane, m, s, ix);
        xb[ew * kPairTileVocab + 32 * c + lane] = make_float4(m, s, __int_as_float(ix), 0.0f);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (rank == 0)
          mbar_arrive(&sm.acce[acc]);
        else
          mbar_arrive_cluster(acce_remote + static_cast<uint32_t>(acc * 8));
      }
      if (lane == 0) mbar_arrive(&sm.xchb[i & 1]);
      if (!mbar_wait(&sm.xchb[i & 1], (i >> 1) & 1, sm.abort, p.err, kErrWaitEpi)) break;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int col = et + 128 * h;
        if (col < rt_rows) {
          float m = kNegBig, s = 0.0f;
          int ix = INT_MAX;
#pragma unroll
          for (int w = 0; w < 4; ++w) {
            const float4 a = xb[w * kPairTileVocab + col];
            merge_tri(m, s, ix, a.x, a.y, __float_as_int(a.z));
          }
          const int row = row0 + col;
          if (per_row > 0)
            merge_tri(am[h], as[h], aix[h], m, s, ix);
          else if (row < M && CAI_IN_RANGE(v < p.n_vt, p.err))
            p.part[static_cast<size_t>(row) * (2 * p.n_vt) + 2 * v + static_cast<int>(rank)] =
                make_float4(m, s, __int_as_float(ix), 0.0f);
        }
      }
    }
    if (per_row > 0) {
      // The pair's row tile is fixed (pair mod n_rt); a pair without tiles
      // writes the empty triple.
      const int row0 = (pair % n_rt) * rt_rows;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int col = et + 128 * h;
        if (col < rt_rows && row0 + col < M)
          p.part[static_cast<size_t>(row0 + col) * per_row + 2 * (pair / n_rt) +
                 static_cast<int>(rank)] = make_float4(am[h], as[h], __int_as_float(aix[h]), 0.0f);
      }
    }
  } else {
    // --------------------------------------------------------- epilogue --
    const int quarter = warp & 3;  // tensor-memory lanes 32 quarter .. 32 quarter + 31
    const uint32_t lane_base = static_cast<uint32_t>(quarter * 32) << 16;
    const uint32_t acce_remote = mapa_shared(sm.acce, 0);
    const int per_row = pair_partials_per_row(M, n_pairs, false);  // > 0: one partial per pair
    float am = kNegBig, as = 0.0f;
    int aix = INT_MAX;
    for (int i = 0; i < my_tiles; ++i) {
      const int t = pair + i * n_pairs;
      const int v = t / n_rt, j = t - v * n_rt;
      const int acc = i & 1;
      if (!mbar_wait(&sm.accf[acc], (i >> 1) & 1, sm.abort, p.err, kErrWaitAccFull)) break;
      tc_fence_after();
      const uint32_t tbase = tmem_base + lane_base + static_cast<uint32_t>(acc * kPairTileVocab);
      const int row = j * kPairTileRows + static_cast<int>(rank) * kPairHalf + quarter * 32 + lane;
      float rs = kLog2e;
      if constexpr (kNorm) {
        if (row < M) rs = kLog2e * __ldg(p.inv_r + row);
      }
      const int vbase = v * kPairTileVocab;
      float m = kNegBig, s = 0.0f;
      int ix = INT_MAX;
#pragma unroll 1
      for (int c = 0; c < kPairTileVocab / 32; ++c) {
        uint32_t x[32];
        tmem_ld_32cols(tbase + static_cast<uint32_t>(32 * c), x);
        tmem_ld_wait();
        const int v0 = vbase + 32 * c;
        const int nvalid = min(32, p.V - v0);  // vocabulary rows past V are zero padding
        float cm = kNegBig;
        int ci = 0;
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          const float z = __uint_as_float(x[k]) * rs;
          if (k < nvalid && z > cm) {
            cm = z;
            ci = k;
          }
        }
        if (cm > m) {  // strictly: an equal maximum keeps the lower index
          s *= fast_exp2(m - cm);
          m = cm;
          ix = v0 + ci;
        }
        float cs = 0.0f;
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          const float z = __uint_as_float(x[k]) * rs;
          cs += k < nvalid ? fast_exp2(z - m) : 0.0f;
        }
        s += cs;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (rank == 0)
          mbar_arrive(&sm.acce[acc]);
        else
          mbar_arrive_cluster(acce_remote + static_cast<uint32_t>(acc * 8));
      }
      if (per_row > 0)
        merge_tri(am, as, aix, m, s, ix);  // tiles in increasing v: ties keep the lower index
      else if (row < M && CAI_IN_RANGE(v < p.n_vt, p.err))
        p.part[static_cast<size_t>(row) * p.n_vt + v] = make_float4(m, s, __int_as_float(ix), 0.0f);
    }
    if (per_row > 0) {
      // The pair's row tile is fixed (pair mod n_rt); a pair without tiles
      // writes the empty triple.
      const int row = (pair % n_rt) * kPairTileRows + static_cast<int>(rank) * kPairHalf +
                      quarter * 32 + lane;
      if (row < M)
        p.part[static_cast<size_t>(row) * per_row + pair / n_rt] =
            make_float4(am, as, __int_as_float(aix), 0.0f);
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no CTA leaves while the pair's MMAs or arrivals may touch it
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kPairTmemCols);
  }
}

// Second stage of a pair step: one warp per masked row merges the row's
// n_vt tile partials (merge_tri: max, rescaled sum, lowest index among equal
// maxima) into one triple, rowres[row], so that the commit reads one value per
// row.  Returns at once when the step ran on the swapped-operand kernel.
struct ReduceParams {
  const float4* part;  // [rows, n_vt] partials (unswapped step), [rows, 2 n_vt] (swapped)
  float4* rowres;      // [rows]
  const int* d_M;
  int n_vt;
  int min_M;
  int n_pairs;         // the pair kernel's grid / 2 (its partials need no merge when
                       // pair_partials_per_row > 0)
  int swap_max_n;      // the pair kernel's orientation rule (pair_swapped)
};

constexpr int kReduceThreads = 256;

__global__ void __launch_bounds__(kReduceThreads) reduce_partials_kernel(const ReduceParams p) {
  grid_launch_dependents();  // every thread: the CTA counts once all of them have
  grid_dependency_wait();    // the pair kernel's partials
  const int M = *p.d_M;
  const bool swap = pair_swapped(M, p.swap_max_n);
  if (M < p.min_M || M < 1 || pair_partials_per_row(M, p.n_pairs, swap) > 0) return;
  const int n_part = (swap ? 2 : 1) * p.n_vt;
  const int lane = threadIdx.x & 31;
  const int nw = (gridDim.x * blockDim.x) >> 5;
  for (int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; row < M; row += nw) {
    const float4* pr = p.part + static_cast<size_t>(row) * n_part;
    float m = kNegBig, s = 0.0f;
    int ix = INT_MAX;
    int k = lane;
    for (; k + 96 < n_part; k += 128) {  // four loads in flight per lane
      const float4 a = __ldcg(pr + k), b = __ldcg(pr + k + 32), c = __ldcg(pr + k + 64),
                   d = __ldcg(pr + k + 96);
      merge_tri(m, s, ix, a.x, a.y, __float_as_int(a.z));
      merge_tri(m, s, ix, b.x, b.y, __float_as_int(b.z));
      merge_tri(m, s, ix, c.x, c.y, __float_as_int(c.z));
      merge_tri(m, s, ix, d.x, d.y, __float_as_int(d.z));
    }
    for (; k < n_part; k += 32) {
      const float4 a = __ldcg(pr + k);
      merge_tri(m, s, ix, a.x, a.y, __float_as_int(a.z));
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) {
      const float mo = __shfl_xor_sync(0xffffffffu, m, off);
      const float so = __shfl_xor_sync(0xffffffffu, s, off);
      const int io = __shfl_xor_sync(0xffffffffu, ix, off);
      merge_tri(m, s, ix, mo, so, io);
    }
    if (lane == 0) p.rowres[row] = make_float4(m, s, __int_as_float(ix), 0.0f);
  }
}

}  // namespace cai
