// LM-head projection fused with the full-vocabulary softmax reduction
// (Box 1 of arXiv 2608.22646: c_i = max_v p_theta(x_i = v), argmax_v p_theta).
//
// The masked positions of a step are few (M_t <= B P), so the contraction is
// run with A and B swapped: the vocabulary fills the MMA M dimension (128 rows
// of W per accumulator tile) and the positions form the N dimension
// (16..256 columns, rounded up to 16).  Each CTA owns a contiguous range of W
// rows (whole 8-row swizzle atoms, at least 64 rows, balanced over the grid
// to within 8 rows) and reads it once from HBM; the logits stay in
// tensor memory and are never written anywhere.  The epilogue reduces every
// accumulator tile to a running (max, sum of exponentials, argmax) per
// position in the log2 domain; the four epilogue warps merge their slices
// through shared memory and each CTA writes one partial triple per position,
// [M, gridDim.x].
//
// Tiles are processed in groups (up to `gmax` tiles of 128 rows): for each
// K block the hidden-state stage (B) is loaded once and used by every tile of
// the group, each tile accumulating into its own tensor-memory slot.  The B
// operand is thus read from L2 once per group instead of once per tile, and
// the group's tiles form independent accumulation chains whose MMAs overlap:
// at small N one chain alone is bound by MMA latency, not by HBM.  Two group
// buffers let the epilogue of one group overlap the MMAs of the next.
//
// W is read from a packed copy made once per context (pack_weight_kernel) in
// exactly the order the CTAs consume it: CTA c owns rows [8 u0, 8 u1) and
// the bytes [16 H u0, 16 H u1) of the packed copy, laid out group by group,
// K block by K block, tile by tile, each stage already in the
// 128-byte-swizzled K-major layout the MMA descriptors expect.  Every CTA thus
// streams one contiguous region front to back with one bulk copy per stage;
// contiguous copies keep DRAM pages open, the strided 128-byte rows of a 2-D
// tensor box do not.
//
// Single-kernel step (fused = 1, B P <= 64 and CAI_ROWS_HEAD=0, or more than
// 128 rows): the kernel decodes all
// B P rows straight from the caller's hidden states (no gather; at N <= 256 a
// step reads W once whatever N is), and the last CTA to finish (atomic
// ticket, no waiting) merges the partials and applies the commit rule for
// every sequence (commit.cuh).  A step is then one launch.  Nothing but the
// commit depends on the previous step: W and the caller's hidden rows are
// inputs, so under programmatic dependent launch the next step's CTAs start
// streaming as soon as this step's CTAs leave their SMs, and wait for this
// step (grid_dependency_wait) only to write their partials (which this
// step's commit reads) and to commit.  If this step leaves nothing masked,
// the next one learns it from the published step word (CommitParams::pub)
// while streaming and stops at the next K block.
//
// Multi-kernel steps (fused = 0) run on lm_head_pair_kernel; this kernel
// takes their steps of fewer than pair_min_M rows only when the pair kernel
// never runs swapped (CAI_PAIR_SWAP=0) or is off (CAI_PAIR=0).
//
// Warp roles (192 threads, one CTA per SM):
//   warp 0      producer (one lane): W stages (bulk copies), hidden stages (TMA)
//   warp 1      TMEM allocator; one lane issues tcgen05.mma
//   warps 2..5  epilogue: tcgen05.ld, transposing warp reduction, partials
#pragma once

#include <climits>
#include <cuda_bf16.h>
#include "commit.cuh"
#include "ptx.cuh"
#include "softmax.cuh"

namespace cai {

constexpr int kRowsPerTile = 128;  // MMA M: vocabulary rows per accumulator
constexpr int kUnitRows = 8;       // granularity of the per-CTA split of V (one swizzle atom)
constexpr int kMinCtaRows = 64;    // fewest vocabulary rows the launch gives one CTA
constexpr int kBlockK = 64;        // K per stage: one 128-byte swizzled row of bf16
constexpr int kChunkN = 256;       // largest MMA N (positions per pass over W)
constexpr int kBoxRowsB = 16;      // rows per TMA box of the hidden tile
constexpr int kHeadThreads = 192;
constexpr int kATileBytes = kRowsPerTile * kBlockK * 2;  // 16 KiB

struct HeadParams {
  const uint8_t* wpk;  // packed W (see pack_weight_kernel)
  const int* d_M;      // masked rows of this step (device; multi-kernel step)
  int* m_hist_slot;    // where this step's M is recorded (multi-kernel step)
  int fused;           // 1: single-kernel step (see below), 0: gather / head / merge kernels
  int M_fixed;         // rows decoded by the single-kernel step (all B P positions)
  int max_M;           // multi-kernel step: larger steps are left to lm_head_pair_kernel
  const unsigned long long* stage_word;  // single-kernel step on staged host rows: the rows
  unsigned long long stage_seq;          // are read once *stage_word >= stage_seq (or null)
  int prefetch;        // stream the first W stages before the dependency wait
  int first;           // the step is a block's step zero (every position masked)
  float4* part;        // [rows_cap, G] partial (m2, S, idx bits, 0) per CTA
  uint32_t* err;       // error word
  int V, H;
  int units;           // ceil(V / kUnitRows)
  int n_stages;        // depth of the W ring (16 KiB slots)
  int n_bslots;        // depth of the hidden-state ring
  int b_slot_bytes;    // n_max * 128
  int slot_cols;       // tensor-memory columns per tile accumulator (round32(n_max))
  int gmax;            // largest tile group
  int tmem_cols;       // allocated tensor-memory columns (>= 2 gmax slot_cols)
  const float* inv_r;  // final-norm row scales 1 / sqrt(mean h^2 + eps) [rows] (kNorm only)
  const __nv_bfloat16* hid;  // single-kernel step, kNorm: the step's rows [M_fixed, H], from
  float norm_eps;            // which the kernel computes the row scales itself (and epsilon)
  CommitParams cp;     // commit rule, run by the last CTA of a single-kernel step
};

// ------------------------------------------------------------ CTA plan --

// First unit (kUnitRows rows) of CTA c when `units` units are split over G CTAs.
__host__ __device__ inline int unit_begin(int c, int units, int G) {
  return static_cast<int>((static_cast<long long>(c) * units) / G);
}

// The work of one CTA: units [u0, u1), i.e. vocabulary rows [row0, row0 +
// rows), as tiles of 128 rows (the last may be shorter, by a multiple of
// kUnitRows), grouped gsz = min(gmax, tiles) tiles at a time.
struct CtaPlan {
  int u0, u1, n_tiles, gsz, n_groups;
  __host__ __device__ int row0() const { return u0 * kUnitRows; }
  __host__ __device__ int rows() const { return (u1 - u0) * kUnitRows; }
  __host__ __device__ int tile_rows(int t) const {
    const int r = rows() - t * kRowsPerTile;
    return r < kRowsPerTile ? r : kRowsPerTile;
  }
  __host__ __device__ int group_first(int g) const { return g * gsz; }
  __host__ __device__ int group_count(int g) const {
    const int n = n_tiles - g * gsz;
    return n < gsz ? n : gsz;
  }
  __host__ __device__ int group_rows(int g) const {
    const int t0 = group_first(g), n = group_count(g);
    return kRowsPerTile * (n - 1) + tile_rows(t0 + n - 1);
  }
  // Byte offset in the packed weight of W stage (group g, K block kb, tile t).
  __host__ __device__ size_t stage_offset(int g, int kb, int t, int H) const {
    return static_cast<size_t>(row0()) * 2 * H + static_cast<size_t>(g) * gsz * kRowsPerTile * 2 * H +
           static_cast<size_t>(kb) * group_rows(g) * 128 +
           static_cast<size_t>(t - group_first(g)) * kATileBytes;
  }
};

// Rows this launch decodes.  Multi-kernel step: the masked rows the gather
// kernel compacted, read after grid_dependency_wait(), unless there are more
// than max_M (lm_head_pair_kernel decodes those steps).  Single-kernel step:
// all B P rows, known at launch (a step that turns out to have nothing to
// decode stops early instead, see `skip`).
__device__ __forceinline__ int rows_to_decode(const int* d_M, int fused, int M_fixed, int max_M) {
  if (fused) return M_fixed;
  const int m = *d_M;
  return m > max_M ? 0 : m;
}

// Single-kernel step after step zero: whether the published step word `w`
// says the previous step left nothing masked.  `decided` is set once the
// word is the previous step's at all.  Step s publishes s + 1 (never 0,
// which is the word after a reset or a state upload), so step s + 1 looks
// for its own id.
__device__ __forceinline__ unsigned long long load_pub(const unsigned long long* pub) {
  return *reinterpret_cast<const volatile unsigned long long*>(pub);
}
__device__ __forceinline__ bool previous_left_nothing(unsigned long long w, int step_id,
                                                      bool& decided) {
  const uint32_t id = static_cast<uint32_t>(w >> 32);
  if (id == 0u || id != static_cast<uint32_t>(step_id)) return false;
  decided = true;
  return static_cast<uint32_t>(w) == 0u;
}

__host__ __device__ inline CtaPlan cta_plan(int c, int units, int G, int gmax) {
  CtaPlan p;
  p.u0 = unit_begin(c, units, G);
  p.u1 = unit_begin(c + 1, units, G);
  p.n_tiles = (p.rows() + kRowsPerTile - 1) / kRowsPerTile;
  const int g = gmax < p.n_tiles ? gmax : p.n_tiles;
  p.gsz = g < 1 ? 1 : g;
  p.n_groups = (p.n_tiles + p.gsz - 1) / p.gsz;
  return p;
}

// Eight bf16 values times eight bf16 weights, rounded to bf16 (final-norm
// weight folded into W: W[v,k] g[k]).
__device__ __forceinline__ uint4 scale_chunk(uint4 w, const __nv_bfloat16* g) {
  __nv_bfloat16* e = reinterpret_cast<__nv_bfloat16*>(&w);
#pragma unroll
  for (int i = 0; i < 8; ++i) e[i] = __float2bfloat16_rn(__bfloat162float(e[i]) * __bfloat162float(g[i]));
  return w;
}

// Pack W [V, H] (row-major bf16) for a grid of G CTAs over `units` units of
// kUnitRows rows and groups of up to gmax tiles.  Inside a stage block, row r's
// 16-byte chunk c (k = 8c..8c+7 of the block's 64) sits at
// r * 128 + ((c ^ (r & 7)) * 16): the 128-byte swizzle of 8-row, 1024-byte
// atoms.  Rows >= V are zero.  One thread per destination 16-byte chunk;
// n_chunks = units * kUnitRows * H / 8.
__global__ void pack_weight_kernel(const uint4* __restrict__ W, uint4* __restrict__ out, int V,
                                   int H, int units, int G, int gmax, long long n_chunks,
                                   const __nv_bfloat16* __restrict__ gw) {
  const long long unit_bytes = 2ll * kUnitRows * H;
  for (long long d = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; d < n_chunks;
       d += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long byte = d * 16;
    const int u = static_cast<int>(byte / unit_bytes);
    // CTA owning unit u: the largest c with unit_begin(c) <= u.
    int c = static_cast<int>((static_cast<long long>(u) * G) / units);
    while (c + 1 < G && unit_begin(c + 1, units, G) <= u) ++c;
    while (c > 0 && unit_begin(c, units, G) > u) --c;
    const CtaPlan pl = cta_plan(c, units, G, gmax);
    const long long off = byte - static_cast<long long>(pl.u0) * unit_bytes;
    const long long group_bytes = static_cast<long long>(pl.gsz) * kRowsPerTile * 2 * H;
    const int g = static_cast<int>(off / group_bytes);
    const long long rem = off - static_cast<long long>(g) * group_bytes;
    const int grow = pl.group_rows(g);
    const int kb = static_cast<int>(rem / (grow * 128));
    const int rem2 = static_cast<int>(rem - static_cast<long long>(kb) * grow * 128);
    const int t = pl.group_first(g) + rem2 / kATileBytes;
    const int inblk = rem2 % kATileBytes;
    const int r = inblk >> 7;
    const int cl = ((inblk >> 4) & 7) ^ (r & 7);
    const long long v = static_cast<long long>(pl.row0()) + t * kRowsPerTile + r;
    uint4 val = make_uint4(0u, 0u, 0u, 0u);
    if (v < V) val = W[(v * H + static_cast<long long>(kb) * kBlockK) / 8 + cl];
    if (gw) val = scale_chunk(val, gw + kb * kBlockK + cl * 8);
    out[d] = val;
  }
}

// Wait used only on the abort path, for copies this CTA already issued.
__device__ __forceinline__ void mbar_drain(uint64_t* bar, uint32_t parity, uint32_t* err) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > kWaitLimitNs) {
      atomicOr(err, kErrDrain);
      return;
    }
  }
}

// ------------------------------------------------------------- smem map --

struct HeadSmem {
  uint8_t* a;        // n_stages x 16 KiB (W)
  uint8_t* b;        // n_bslots x b_slot_bytes (hidden rows)
  float4* epi;       // [2][4][slot_cols] cross-warp merge, double-buffered by chunk
  uint64_t* full_a;  // n_stages
  uint64_t* empty_a; // n_stages
  uint64_t* full_b;  // n_bslots
  uint64_t* empty_b; // n_bslots
  uint64_t* accf;    // 2: group accumulators ready
  uint64_t* acce;    // 2: group accumulators drained by the epilogue
  uint64_t* drain;   // 1
  uint64_t* epib;    // 2: the four epilogue warps have written epi[buffer]
  uint32_t* tmem_slot;
  volatile int* abort;
  volatile int* skip;  // the step stops early: nothing was left to decode
};

__host__ __device__ inline size_t head_smem_bytes(int n_stages, int n_bslots, int b_slot_bytes,
                                                  int slot_cols) {
  return 1024 + static_cast<size_t>(n_stages) * kATileBytes +
         static_cast<size_t>(n_bslots) * b_slot_bytes + static_cast<size_t>(8) * slot_cols * 16 +
         static_cast<size_t>(2 * n_stages + 2 * n_bslots + 7) * 8 + 16;
}

__device__ __forceinline__ HeadSmem carve(uint8_t* raw, const HeadParams& p) {
  HeadSmem s;
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  s.a = base;
  s.b = s.a + static_cast<size_t>(p.n_stages) * kATileBytes;
  s.epi = reinterpret_cast<float4*>(s.b + static_cast<size_t>(p.n_bslots) * p.b_slot_bytes);
  s.full_a = reinterpret_cast<uint64_t*>(s.epi + 8 * p.slot_cols);
  s.empty_a = s.full_a + p.n_stages;
  s.full_b = s.empty_a + p.n_stages;
  s.empty_b = s.full_b + p.n_bslots;
  s.accf = s.empty_b + p.n_bslots;
  s.acce = s.accf + 2;
  s.drain = s.acce + 2;
  s.epib = s.drain + 1;
  s.tmem_slot = reinterpret_cast<uint32_t*>(s.epib + 2);
  s.abort = reinterpret_cast<volatile int*>(s.tmem_slot + 1);
  s.skip = s.abort + 1;
  return s;
}

// Ring position: slot index and the parity of its current phase.
struct Ring {
  int slot = 0;
  uint32_t phase = 0;
  __device__ void next(int n) {
    if (++slot == n) {
      slot = 0;
      phase ^= 1u;
    }
  }
};

// Single-kernel step, end of every CTA: the last CTA to finish (atomic
// ticket, no waiting) merges the partials and commits the step for every
// sequence, after the previous step's commit (state, ticket) is complete.
// `free_smem` is at least sizeof(CommitSmem) bytes of shared memory that no
// copy or MMA touches any more (the drained W ring).
__device__ __forceinline__ void fused_step_commit(const CommitParams& cp, uint8_t* free_smem) {
  grid_dependency_wait();
  __shared__ int s_last;
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(cp.ticket, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  int decoded = 0, remaining = 0;
  for (int b = 0; b < cp.B; ++b) {
    int left = 0;
    decoded += merge_commit_sequence(cp, b, *reinterpret_cast<CommitSmem*>(free_smem), cp.part,
                                     cp.n_part, &left);
    remaining += left;
  }
  if (threadIdx.x == 0) *cp.m_hist_slot = decoded;
  finish_step(cp, remaining);
}

// ---------------------------------------------------------------- kernel --

// kNorm: the model's final RMSNorm is part of the head.  Its weight is
// already folded into W; row n's logits are scaled by 1 / sqrt(mean h^2 +
// eps) of the row: computed by the epilogue warps from the caller's rows in a
// single-kernel step, inv_r[n] (written by the gather) in a multi-kernel one.
template <bool kNorm>
__global__ void __launch_bounds__(kHeadThreads, 1)
    lm_head_softmax_kernel(const __grid_constant__ CUtensorMap tm_h, const HeadParams p) {
  extern __shared__ uint8_t smem_raw[];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  HeadSmem sm = carve(smem_raw, p);

  const int G = gridDim.x;
  const int cta = blockIdx.x;
  const CtaPlan pl = cta_plan(cta, p.units, G, p.gmax);
  const int KB = p.H / kBlockK;

  // Multi-kernel step with the pair kernel on: most steps belong to the pair
  // kernel, so read M first and leave before any setup when it is one of them.
  if (!p.fused && p.max_M != INT_MAX) {
    grid_launch_dependents();
    grid_dependency_wait();
    if (*p.d_M > p.max_M) return;
  }

  // Prologue (overlaps the previous kernel under programmatic dependent launch).
  if (threadIdx.x == 0) {
    for (int s = 0; s < p.n_stages; ++s) {
      mbar_init(&sm.full_a[s], 1);
      mbar_init(&sm.empty_a[s], 1);
    }
    for (int s = 0; s < p.n_bslots; ++s) {
      mbar_init(&sm.full_b[s], 1);
      mbar_init(&sm.empty_b[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&sm.accf[a], 1);
      mbar_init(&sm.acce[a], 4);
      mbar_init(&sm.epib[a], 4);
    }
    mbar_init(sm.drain, 1);
    *sm.abort = 0;
    *sm.skip = 0;
    fence_mbar_init();
  }
  grid_launch_dependents();  // every thread: the CTA counts once all of them have
  if (warp == 0 && lane == 0) prefetch_tmap(&tm_h);
  if (warp == 1) {
    tmem_alloc(sm.tmem_slot, static_cast<uint32_t>(p.tmem_cols));
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *sm.tmem_slot;
  const int group_cols = p.gmax * p.slot_cols;  // tensor-memory columns per group buffer

  // The weight does not depend on the previous kernels: the producer starts
  // streaming the first ring of W stages before waiting for them.  Everything
  // that does (the masked-row count, the gathered rows, the partial buffer,
  // the commit state) is touched only after grid_dependency_wait().  A
  // single-kernel step reads nothing the previous step writes before its
  // partials, so only its epilogue and its commit wait.
  // When most steps go to the pair kernel, copies started before M is known
  // would mostly be wasted, so the launch asks for none.
  const int n_pre = p.prefetch ? min(p.n_stages, pl.n_tiles * KB) : 0;
  const bool spec = p.fused && !p.first;  // may find out that nothing is masked

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------ producer --
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_h = policy_evict_last();
      {
        int i = 0;
        for (int g = 0; g < pl.n_groups && i < n_pre; ++g)
          for (int kb = 0; kb < KB && i < n_pre; ++kb)
            for (int t = pl.group_first(g); t < pl.group_first(g) + pl.group_count(g) && i < n_pre;
                 ++t, ++i) {
              const uint32_t bytes = static_cast<uint32_t>(pl.tile_rows(t) * 128);
              mbar_expect_tx(&sm.full_a[i], bytes);
              bulk_load(sm.a + static_cast<size_t>(i) * kATileBytes,
                        p.wpk + pl.stage_offset(g, kb, t, p.H), bytes, &sm.full_a[i], pol_w);
            }
      }
      if (!p.fused) grid_dependency_wait();
      const int M = rows_to_decode(p.d_M, p.fused, p.M_fixed, p.max_M);
      const int n_chunks = (M + kChunkN - 1) / kChunkN;
      Ring ra, rb;
      long long a_issued = 0, b_issued = 0;
      bool ok = true, decided = !spec, skipped = false;
      // Rows copied from the host on the context's side stream: wait (bounded)
      // for that copy's sequence word before the first row load.
      if (p.stage_word && !wait_word_ge(p.stage_word, p.stage_seq, sm.abort, p.err, kErrWaitRows))
        ok = false;
      // The word is loaded one K block ahead of its use, so its latency never
      // holds up the stream of copies.
      unsigned long long pub_w = spec ? load_pub(p.cp.pub) : 0ull;
      for (int q = 0; q < n_chunks && ok && !skipped; ++q) {
        const int n0 = q * kChunkN;
        const int nq = (min(kChunkN, M - n0) + 15) & ~15;
        for (int g = 0; g < pl.n_groups && ok && !skipped; ++g) {
          for (int kb = 0; kb < KB && ok; ++kb) {
            if (!mbar_wait(&sm.empty_b[rb.slot], rb.phase ^ 1u, sm.abort, p.err, kErrWaitEmpty)) {
              ok = false;
              break;
            }
            if (!decided && previous_left_nothing(pub_w, p.cp.step_id, decided)) {
              // Stop at this K block: the hidden stage is completed empty and
              // carries the stop mark to the MMA warp, which has consumed
              // every W stage issued so far by the time it sees it.
              *sm.skip = 1;
              mbar_arrive(&sm.full_b[rb.slot]);
              skipped = true;
              break;
            }
            if (!decided) pub_w = load_pub(p.cp.pub);
            mbar_arrive_expect_tx(&sm.full_b[rb.slot], static_cast<uint32_t>(nq * 128));
            uint8_t* bdst = sm.b + static_cast<size_t>(rb.slot) * p.b_slot_bytes;
            for (int i = 0; i < nq / kBoxRowsB; ++i)
              tma_load_2d(bdst + i * kBoxRowsB * 128, &tm_h, &sm.full_b[rb.slot], kb * kBlockK,
                          n0 + i * kBoxRowsB, pol_h);
            ++b_issued;
            rb.next(p.n_bslots);
            for (int t = pl.group_first(g); t < pl.group_first(g) + pl.group_count(g); ++t) {
              if (a_issued < n_pre) {
                mbar_arrive(&sm.full_a[ra.slot]);  // copy already in flight
              } else {
                if (!mbar_wait(&sm.empty_a[ra.slot], ra.phase ^ 1u, sm.abort, p.err,
                               kErrWaitEmpty)) {
                  ok = false;
                  break;
                }
                const uint32_t bytes = static_cast<uint32_t>(pl.tile_rows(t) * 128);
                mbar_arrive_expect_tx(&sm.full_a[ra.slot], bytes);
                bulk_load(sm.a + static_cast<size_t>(ra.slot) * kATileBytes,
                          p.wpk + pl.stage_offset(g, kb, t, p.H), bytes, &sm.full_a[ra.slot],
                          pol_w);
              }
              ++a_issued;
              ra.next(p.n_stages);
            }
          }
        }
      }
      if (a_issued < n_pre) {
        // Nothing to decode (M = 0, or a stop) or an abort before the prefetched
        // stages were claimed: complete their phases so the copies can drain.
        for (long long i = a_issued; i < n_pre; ++i) mbar_arrive(&sm.full_a[i]);
        for (long long i = a_issued; i < n_pre; ++i) mbar_drain(&sm.full_a[i], 0, p.err);
      }
      if (!ok) {
        // Abort path: let the copies already in flight land before exit.
        const long long fa = a_issued > p.n_stages ? a_issued - p.n_stages : 0;
        for (long long i = fa; i < a_issued; ++i)
          mbar_drain(&sm.full_a[i % p.n_stages], static_cast<uint32_t>((i / p.n_stages) & 1),
                     p.err);
        const long long fb = b_issued > p.n_bslots ? b_issued - p.n_bslots : 0;
        for (long long i = fb; i < b_issued; ++i)
          mbar_drain(&sm.full_b[i % p.n_bslots], static_cast<uint32_t>((i / p.n_bslots) & 1),
                     p.err);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------------------------------------------- MMA issuer --
      if (!p.fused) grid_dependency_wait();
      const int M = rows_to_decode(p.d_M, p.fused, p.M_fixed, p.max_M);
      const int n_chunks = (M + kChunkN - 1) / kChunkN;
      Ring ra, rb, racc;
      bool ok = true, skipped = false;
      for (int q = 0; q < n_chunks && ok && !skipped; ++q) {
        const int n0 = q * kChunkN;
        const int nq = (min(kChunkN, M - n0) + 15) & ~15;
        const uint32_t idesc = idesc_bf16_f32(kRowsPerTile, static_cast<uint32_t>(nq));
        for (int g = 0; g < pl.n_groups && ok; ++g) {
          if (!mbar_wait(&sm.acce[racc.slot], racc.phase ^ 1u, sm.abort, p.err,
                         kErrWaitAccEmpty)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_group = tmem_base + static_cast<uint32_t>(racc.slot * group_cols);
          for (int kb = 0; kb < KB && ok; ++kb) {
            if (!mbar_wait(&sm.full_b[rb.slot], rb.phase, sm.abort, p.err, kErrWaitFull)) {
              ok = false;
              break;
            }
            if (spec && *sm.skip) {
              skipped = true;
              break;
            }
            const uint32_t b_addr =
                smem_addr(sm.b + static_cast<size_t>(rb.slot) * p.b_slot_bytes);
            for (int t = pl.group_first(g); t < pl.group_first(g) + pl.group_count(g); ++t) {
              if (!mbar_wait(&sm.full_a[ra.slot], ra.phase, sm.abort, p.err, kErrWaitFull)) {
                ok = false;
                break;
              }
              tc_fence_after();
              const uint32_t a_addr =
                  smem_addr(sm.a + static_cast<size_t>(ra.slot) * kATileBytes);
              const uint32_t d_tmem =
                  d_group + static_cast<uint32_t>((t - pl.group_first(g)) * p.slot_cols);
#pragma unroll
              for (int kk = 0; kk < kBlockK / 16; ++kk) {
                mma_bf16(d_tmem, sdesc_k_sw128(a_addr + kk * 32), sdesc_k_sw128(b_addr + kk * 32),
                         idesc, (kb | kk) != 0 ? 1u : 0u);
              }
              mma_commit(&sm.empty_a[ra.slot]);
              ra.next(p.n_stages);
            }
            if (!ok) break;
            mma_commit(&sm.empty_b[rb.slot]);
            rb.next(p.n_bslots);
          }
          if (!ok || skipped) break;
          mma_commit(&sm.accf[racc.slot]);
          racc.next(2);
        }
      }
      if (!ok || skipped) {
        // Abort or stop: wait for every MMA already issued before TMEM is freed.
        mma_commit(sm.drain);
        mbar_drain(sm.drain, 0, p.err);
      }
      // Stop: release the epilogue, which waits for this group's accumulators.
      if (skipped) mbar_arrive(&sm.accf[racc.slot]);
    }
    __syncwarp();
  } else {
    // --------------------------------------------------------- epilogue --
    if (!p.fused) grid_dependency_wait();
    const int M = rows_to_decode(p.d_M, p.fused, p.M_fixed, p.max_M);
    const int n_chunks = (M + kChunkN - 1) / kChunkN;
    if (!p.fused && threadIdx.x == 64 && cta == 0 && *p.d_M <= p.max_M) *p.m_hist_slot = M;
    const int ew = warp - 2;       // 0..3: slot in the cross-warp merge
    const int quarter = warp & 3;  // tensor-memory lanes this warp may read
    const uint32_t lane_base = static_cast<uint32_t>(quarter * 32) << 16;
    // Final-norm row scales: a single-kernel step computes them from the
    // caller's rows (nothing then waits on an earlier kernel); a multi-kernel
    // step reads the gather's.
    const float* scale = p.inv_r;
    if constexpr (kNorm) {
      __shared__ float s_scale[kChunkN];
      if (p.fused) {
        epilogue_row_scales(p.hid, M, p.H, p.norm_eps, s_scale, ew, lane);
        scale = s_scale;
      }
    }
    Ring racc;
    bool ok = true;
    for (int q = 0; q < n_chunks && ok; ++q) {
      const int n0 = q * kChunkN;
      const int nq = (min(kChunkN, M - n0) + 15) & ~15;
      const int ngroups = (nq + 31) >> 5;
      float rm[8], rs[8];
      int ri[8];
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        rm[c] = kNegBig;
        rs[c] = 0.0f;
        ri[c] = INT_MAX;
      }
      if (ngroups == 1) {
        // Up to 32 positions: each lane folds its own row of every tile into a
        // running triple per column (one exponential per logit, no shuffles);
        // the 32 lanes are merged once, after the last tile.
        float lm[32], ls[32];
        int li[32];
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          lm[c] = kNegBig;
          ls[c] = 0.0f;
          li[c] = INT_MAX;
        }
        for (int g = 0; g < pl.n_groups; ++g) {
          if (!mbar_wait(&sm.accf[racc.slot], racc.phase, sm.abort, p.err, kErrWaitAccFull)) {
            ok = false;
            break;
          }
          if (spec && *sm.skip) {
            ok = false;  // stop: nothing of this step is written
            break;
          }
          tc_fence_after();
          float sc[32];
#pragma unroll
          for (int c = 0; c < 32; ++c) sc[c] = kLog2e;
          if constexpr (kNorm) {
#pragma unroll
            for (int c = 0; c < 32; ++c)
              if (n0 + c < M) sc[c] = kLog2e * scale[n0 + c];
          }
          const uint32_t tgroup =
              tmem_base + lane_base + static_cast<uint32_t>(racc.slot * group_cols);
          for (int t = pl.group_first(g); t < pl.group_first(g) + pl.group_count(g); ++t) {
            const int row_local = quarter * 32 + lane;
            const int vrow = pl.row0() + t * kRowsPerTile + row_local;
            const bool valid = row_local < pl.tile_rows(t) && vrow < p.V;
            uint32_t v[32];
            tmem_ld_32cols(tgroup + static_cast<uint32_t>((t - pl.group_first(g)) * p.slot_cols),
                           v);
            tmem_ld_wait();
            if (valid) {
#pragma unroll
              for (int c = 0; c < 32; ++c)
                online_update(lm[c], ls[c], li[c], __uint_as_float(v[c]) * sc[c], vrow);
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&sm.acce[racc.slot]);
          racc.next(2);
        }
        if (!ok) break;
        transpose_merge32(lm, ls, li, lane);
        rm[0] = lm[0];
        rs[0] = ls[0];
        ri[0] = li[0];
      } else {
        for (int g = 0; g < pl.n_groups; ++g) {
          if (!mbar_wait(&sm.accf[racc.slot], racc.phase, sm.abort, p.err, kErrWaitAccFull)) {
            ok = false;
            break;
          }
          if (spec && *sm.skip) {
            ok = false;  // stop: nothing of this step is written
            break;
          }
          tc_fence_after();
          const uint32_t tgroup =
              tmem_base + lane_base + static_cast<uint32_t>(racc.slot * group_cols);
          for (int t = pl.group_first(g); t < pl.group_first(g) + pl.group_count(g); ++t) {
            const int row_local = quarter * 32 + lane;
            const int vrow = pl.row0() + t * kRowsPerTile + row_local;
            const bool valid = row_local < pl.tile_rows(t) && vrow < p.V;
            const uint32_t tcol =
                tgroup + static_cast<uint32_t>((t - pl.group_first(g)) * p.slot_cols);
#pragma unroll
            for (int c = 0; c < 8; ++c) {
              if (c < ngroups) {
                uint32_t v[32];
                tmem_ld_32cols(tcol + 32 * c, v);
                tmem_ld_wait();
                float m, s;
                int i;
                if constexpr (kNorm) {
                  transpose_reduce32(v, valid, vrow, lane, m, s, i, scale + n0 + 32 * c);
                } else {
                  transpose_reduce32(v, valid, vrow, lane, m, s, i);
                }
                merge_tri(rm[c], rs[c], ri[c], m, s, i);
              }
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&sm.acce[racc.slot]);
          racc.next(2);
        }
      }
      if (!ok) break;
      // Cross-warp merge of the four 32-row slices of every column, then one
      // partial per (position, CTA).  The buffer alternates by chunk: a warp
      // writes buffer q & 1 again only after every warp arrived for chunk q + 1,
      // which each does after reading chunk q.
      const int buf = q & 1;
      float4* epi = sm.epi + buf * 4 * p.slot_cols;
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        if (c < ngroups)
          epi[ew * p.slot_cols + 32 * c + lane] =
              make_float4(rm[c], rs[c], __int_as_float(ri[c]), 0.0f);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.epib[buf]);
      if (!mbar_wait(&sm.epib[buf], static_cast<uint32_t>((q >> 1) & 1), sm.abort, p.err,
                     kErrWaitEpi)) {
        ok = false;
        break;
      }
      // The previous step's commit reads the same partial buffer.
      if (p.fused) grid_dependency_wait();
      const int ncols = min(nq, M - n0);
      for (int col = ew * 32 + lane; col < ncols; col += 128) {
        const float4 a = epi[col];
        float m = a.x, s = a.y;
        int i = __float_as_int(a.z);
#pragma unroll
        for (int w = 1; w < 4; ++w) {
          const float4 b = epi[w * p.slot_cols + col];
          merge_tri(m, s, i, b.x, b.y, __float_as_int(b.z));
        }
        p.part[static_cast<size_t>(n0 + col) * G + cta] = make_float4(m, s, __int_as_float(i), 0.0f);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, static_cast<uint32_t>(p.tmem_cols));
  }

  if (p.fused) fused_step_commit(p.cp, sm.a);
}

}  // namespace cai
