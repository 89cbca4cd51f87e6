// LM head of the single-kernel step with the masked rows as the MMA's A
// operand: the same quantities as lm_head_softmax_kernel (Box 1 of
// arXiv 2608.22646: c_i = max_v p_theta(x_i = v) and argmax_v p_theta,
// logits never leaving tensor memory), for the M <= 128 rows of a step whose
// block holds at most 128 positions.
//
// Why this orientation.  In the swapped kernel (lm_head_softmax_kernel, W as
// the A operand, the rows as N = 32) every 16 KiB W stage took ~0.345 us of
// the MMA thread (four K = 16 MMAs, their waits and commits), whatever the
// stage held: ~48 GB/s of W per SM, the HBM share of 151 SMs, so the stream
// was paced by the MMA side and a CTA's short last tile cost as much as a
// full one (the same stream without MMAs, or with one MMA per stage, ran at
// 7.7-7.8 TB/s).  With the rows as A and up to 256 vocabulary rows as B, a
// 32 KiB stage of W takes four MMAs, half as many per byte, and the stream is
// HBM-bound.  The rows pad to M = 128, which the tensor cores absorb (an
// M = 128, N = 256, K = 16 MMA takes ~65 ns on resident operands).
//
// Rows stages.  The MMA reads 128 rows of A, but only the first mq =
// round16(M) are the step's; the accumulator rows past M are never read.  So
// a rows stage owns only mq rows (the stride between stages is mq * 128 bytes
// rounded up to 1 KiB, 4 KiB for M <= 32) and the MMA's read of the other
// rows runs on into the following stages (and, for the last ones, the W ring
// placed after them): whatever it finds there only reaches accumulator rows
// that no thread loads.  Small stages let the rows ring be as deep as the W
// ring, so the producer, which issues both, never holds back a W copy for
// want of a rows stage.
//
// Work split: as lm_head_softmax_kernel, V in units of 8 rows over the CTAs;
// a CTA's rows form equal groups of at most 256 vocabulary rows (RowsPlan),
// and the packed W (pack_weight_rows_kernel) stores each group's K block as
// one contiguous block of at most 32 KiB in the 128-byte-swizzled K-major
// layout, so one bulk copy loads one B stage.  The
// CTA runs its groups one after the other, each over all K blocks into one of
// two tensor-memory accumulators (128 lanes x 256 columns); the rows' K block
// is reloaded (from L2) for every group.
//
// Roles (192 threads): warp 0 producer (one lane: W stages by bulk copy, row
// stages by TMA); warp 1 allocates tensor memory and one lane issues the
// MMAs; warps 2..5 epilogue: tensor-memory lane r holds row r's logits, so
// the thread of lane r runs a serial online softmax over the group's columns
// (only warps whose 32 lanes hold rows < M have work).  Each thread writes
// one partial per (row, CTA); the last CTA merges them and commits the step
// (fused_step_commit), as in the single-kernel step of
// lm_head_softmax_kernel, with the same cross-step behaviour under
// programmatic dependent launch.
#pragma once

#include <climits>
#include "head_kernel.cuh"
#include "ptx.cuh"
#include "softmax.cuh"

namespace cai {

constexpr int kRowsM = 128;                          // MMA M: rows of the step, padded
constexpr int kRowsGroupRows = 256;                  // MMA N: vocabulary rows per group
constexpr int kRowsWStage = kRowsGroupRows * 128;    // 32 KiB: one K block of a group
constexpr int kRowsHStageMax = kRowsM * 128;         // 16 KiB: all 128 rows of a K block
constexpr int kRowsTmemCols = 2 * kRowsGroupRows;    // two accumulators

// Bytes between two rows stages for a step of M rows (see above).
__host__ __device__ inline int rows_h_stride(int M) {
  return (((M + 15) & ~15) * 128 + 1023) & ~1023;
}

// The rows ring comes first, then the W ring, whose first 12 KiB or more
// cover the last rows stage's read past its own bytes.
__host__ __device__ inline size_t rows_smem_bytes(int n_stages, int n_bslots, int h_stride) {
  return 1024 + static_cast<size_t>(n_bslots) * h_stride +
         static_cast<size_t>(n_stages) * kRowsWStage +
         static_cast<size_t>(2 * n_stages + 2 * n_bslots + 5) * 8 + 16;
}

struct RowsSmem {
  uint8_t* h;         // n_bslots x h_stride
  uint8_t* w;         // n_stages x 32 KiB
  uint64_t* full_w;   // n_stages
  uint64_t* empty_w;  // n_stages
  uint64_t* full_h;   // n_bslots
  uint64_t* empty_h;  // n_bslots
  uint64_t* accf;     // 2: accumulator ready
  uint64_t* acce;     // 2: accumulator drained by the four epilogue warps
  uint64_t* drain;    // 1
  uint32_t* tmem_slot;
  volatile int* abort;
  volatile int* skip;
};

__device__ __forceinline__ RowsSmem rows_carve(uint8_t* raw, int n_stages, int n_bslots,
                                               int h_stride) {
  RowsSmem s;
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  s.h = base;
  s.w = s.h + static_cast<size_t>(n_bslots) * h_stride;
  s.full_w = reinterpret_cast<uint64_t*>(s.w + static_cast<size_t>(n_stages) * kRowsWStage);
  s.empty_w = s.full_w + n_stages;
  s.full_h = s.empty_w + n_stages;
  s.empty_h = s.full_h + n_bslots;
  s.accf = s.empty_h + n_bslots;
  s.acce = s.accf + 2;
  s.drain = s.acce + 2;
  s.tmem_slot = reinterpret_cast<uint32_t*>(s.drain + 1);
  s.abort = reinterpret_cast<volatile int*>(s.tmem_slot + 1);
  s.skip = s.abort + 1;
  return s;
}

// The work of one CTA: units [u0, u1) of kUnitRows rows (the same split of V
// as lm_head_softmax_kernel), cut into n_groups = ceil(rows / 256) groups of
// equal size to within one unit.  Equal groups keep every group's MMAs (whose
// time hardly depends on N) under its share of the W stream; a short last
// group would be paced by its MMAs instead.
struct RowsPlan {
  int u0, u1, n_groups;
  __host__ __device__ int row0() const { return u0 * kUnitRows; }
  __host__ __device__ int rows() const { return (u1 - u0) * kUnitRows; }
  // First unit of group g, relative to u0.
  __host__ __device__ int group_unit(int g) const {
    return static_cast<int>((static_cast<long long>(g) * (u1 - u0)) / n_groups);
  }
  __host__ __device__ int group_row0(int g) const { return row0() + group_unit(g) * kUnitRows; }
  __host__ __device__ int group_rows(int g) const {
    return (group_unit(g + 1) - group_unit(g)) * kUnitRows;
  }
  // Byte offset in the packed weight of group g's K block kb: a group's K
  // blocks follow one another, each group_rows(g) x 128 bytes.
  __host__ __device__ size_t stage_offset(int g, int kb, int H) const {
    return static_cast<size_t>(group_row0(g)) * 2 * H +
           static_cast<size_t>(kb) * group_rows(g) * 128;
  }
};

__host__ __device__ inline RowsPlan rows_plan(int c, int units, int G) {
  RowsPlan p;
  p.u0 = unit_begin(c, units, G);
  p.u1 = unit_begin(c + 1, units, G);
  p.n_groups = (p.rows() + kRowsGroupRows - 1) / kRowsGroupRows;
  return p;
}

// Pack W [V, H] (row-major bf16) for lm_head_rows_kernel on G CTAs: CTA c's
// groups in order, each group's K blocks in order, each K block the group's
// rows in the 128-byte-swizzled K-major layout (row r's 16-byte chunk c at
// r * 128 + (c ^ (r & 7)) * 16, 8-row atoms of 1 KiB).  Rows >= V are zero;
// gw (bf16 [H], or null) is the final-norm weight folded in.  One thread per
// destination 16-byte chunk; n_chunks = units * kUnitRows * H / 8.
__global__ void pack_weight_rows_kernel(const uint4* __restrict__ W, uint4* __restrict__ out, int V,
                                        int H, int units, int G, long long n_chunks,
                                        const __nv_bfloat16* __restrict__ gw) {
  const long long unit_bytes = 2ll * kUnitRows * H;
  for (long long d = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; d < n_chunks;
       d += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long byte = d * 16;
    const int u = static_cast<int>(byte / unit_bytes);
    int c = static_cast<int>((static_cast<long long>(u) * G) / units);
    while (c + 1 < G && unit_begin(c + 1, units, G) <= u) ++c;
    while (c > 0 && unit_begin(c, units, G) > u) --c;
    const RowsPlan pl = rows_plan(c, units, G);
    // Group holding unit u (groups are whole units).
    int g = static_cast<int>((static_cast<long long>(u - pl.u0) * pl.n_groups) / (pl.u1 - pl.u0));
    while (g + 1 < pl.n_groups && pl.group_unit(g + 1) <= u - pl.u0) ++g;
    while (g > 0 && pl.group_unit(g) > u - pl.u0) --g;
    const long long rem = byte - static_cast<long long>(pl.group_row0(g)) * 2 * H;
    const int grow = pl.group_rows(g);
    const int kb = static_cast<int>(rem / (grow * 128));
    const int rem2 = static_cast<int>(rem - static_cast<long long>(kb) * grow * 128);
    const int r = rem2 >> 7;
    const int cl = ((rem2 >> 4) & 7) ^ (r & 7);
    const long long v = static_cast<long long>(pl.group_row0(g)) + r;
    uint4 val = make_uint4(0u, 0u, 0u, 0u);
    if (v < V) val = W[(v * H + static_cast<long long>(kb) * kBlockK) / 8 + cl];
    if (gw) val = scale_chunk(val, gw + kb * kBlockK + cl * 8);
    out[d] = val;
  }
}

// Single-kernel step only (p.fused = 1, p.M_fixed <= 128), W packed by
// pack_weight_rows_kernel.  p.n_stages is the W ring depth (32 KiB stages),
// p.n_bslots the rows ring depth (stages rows_h_stride(M) apart).  kNorm: row
// r's logits are scaled by 1 / sqrt(mean h^2 + eps) of the row, which the
// epilogue warps compute from the step's rows (p.hid).
template <bool kNorm>
__global__ void __launch_bounds__(kHeadThreads, 1)
    lm_head_rows_kernel(const __grid_constant__ CUtensorMap tm_h, const HeadParams p) {
  extern __shared__ uint8_t smem_raw[];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int h_stride = rows_h_stride(p.M_fixed);
  RowsSmem sm = rows_carve(smem_raw, p.n_stages, p.n_bslots, h_stride);
  const int cta = blockIdx.x;
  const RowsPlan pl = rows_plan(cta, p.units, gridDim.x);
  const int KB = p.H / kBlockK;
  const int M = p.M_fixed;
  const int mq = (M + 15) & ~15;  // rows loaded per K block (TMA fills rows past B P with zeros)
  const bool spec = !p.first;     // may find out that nothing is masked
  const int n_pre = p.prefetch ? min(p.n_stages, pl.n_groups * KB) : 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < p.n_stages; ++s) {
      mbar_init(&sm.full_w[s], 1);
      mbar_init(&sm.empty_w[s], 1);
    }
    for (int s = 0; s < p.n_bslots; ++s) {
      mbar_init(&sm.full_h[s], 1);
      mbar_init(&sm.empty_h[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&sm.accf[a], 1);
      mbar_init(&sm.acce[a], 4);
    }
    mbar_init(sm.drain, 1);
    *sm.abort = 0;
    *sm.skip = 0;
    fence_mbar_init();
    // The weight does not depend on earlier kernels: the first ring of W
    // stages is issued now, before the tensor-memory allocation.
    const uint64_t pol_w = policy_evict_first();
    int i = 0;
    for (int g = 0; g < pl.n_groups && i < n_pre; ++g)
      for (int kb = 0; kb < KB && i < n_pre; ++kb, ++i) {
        const uint32_t bytes = static_cast<uint32_t>(pl.group_rows(g) * 128);
        mbar_expect_tx(&sm.full_w[i], bytes);
        bulk_load(sm.w + static_cast<size_t>(i) * kRowsWStage,
                  p.wpk + pl.stage_offset(g, kb, p.H), bytes, &sm.full_w[i], pol_w);
      }
  }
  grid_launch_dependents();  // every thread: the CTA counts once all of them have
  if (warp == 0 && lane == 0) prefetch_tmap(&tm_h);
  if (warp == 1) {
    tmem_alloc(sm.tmem_slot, kRowsTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *sm.tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------ producer --
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_h = policy_evict_last();
      Ring rw, rh;
      long long w_issued = 0, h_issued = 0;
      bool ok = true, decided = !spec;
      // Rows copied from the host on the context's side stream: wait (bounded)
      // for that copy's sequence word before the first row load.
      if (p.stage_word && !wait_word_ge(p.stage_word, p.stage_seq, sm.abort, p.err, kErrWaitRows))
        ok = false;
      // The previous step's published word, loaded one K block ahead of its use.
      unsigned long long pub_w = spec ? load_pub(p.cp.pub) : 0ull;
      for (int g = 0; g < pl.n_groups && ok; ++g) {
        const uint32_t wbytes = static_cast<uint32_t>(pl.group_rows(g) * 128);
        for (int kb = 0; kb < KB && ok; ++kb) {
          if (!mbar_wait(&sm.empty_h[rh.slot], rh.phase ^ 1u, sm.abort, p.err, kErrWaitEmpty)) {
            ok = false;
            break;
          }
          if (!decided && previous_left_nothing(pub_w, p.cp.step_id, decided)) {
            // Stop: the rows stage completes empty and carries the stop mark
            // to the MMA thread, which has consumed every W stage issued so
            // far by the time it sees it.
            *sm.skip = 1;
            mbar_arrive(&sm.full_h[rh.slot]);
            g = pl.n_groups;
            break;
          }
          if (!decided) pub_w = load_pub(p.cp.pub);
          mbar_arrive_expect_tx(&sm.full_h[rh.slot], static_cast<uint32_t>(mq * 128));
          uint8_t* hdst = sm.h + static_cast<size_t>(rh.slot) * h_stride;
          for (int i = 0; i < mq / kBoxRowsB; ++i)
            tma_load_2d(hdst + i * kBoxRowsB * 128, &tm_h, &sm.full_h[rh.slot], kb * kBlockK,
                        i * kBoxRowsB, pol_h);
          ++h_issued;
          rh.next(p.n_bslots);
          if (w_issued < n_pre) {
            mbar_arrive(&sm.full_w[rw.slot]);  // copy already in flight
          } else {
            if (!mbar_wait(&sm.empty_w[rw.slot], rw.phase ^ 1u, sm.abort, p.err, kErrWaitEmpty)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&sm.full_w[rw.slot], wbytes);
            bulk_load(sm.w + static_cast<size_t>(rw.slot) * kRowsWStage,
                      p.wpk + pl.stage_offset(g, kb, p.H), wbytes, &sm.full_w[rw.slot],
                      pol_w);
          }
          ++w_issued;
          rw.next(p.n_stages);
        }
      }
      if (w_issued < n_pre) {
        // A stop or an abort before the prefetched stages were claimed:
        // complete their phases so the copies can drain.
        for (long long i = w_issued; i < n_pre; ++i) mbar_arrive(&sm.full_w[i]);
        for (long long i = w_issued; i < n_pre; ++i) mbar_drain(&sm.full_w[i], 0, p.err);
      }
      if (!ok) {
        // Abort path: let the copies already in flight land before exit.
        const long long fw = w_issued > p.n_stages ? w_issued - p.n_stages : 0;
        for (long long i = fw; i < w_issued; ++i)
          mbar_drain(&sm.full_w[i % p.n_stages], static_cast<uint32_t>((i / p.n_stages) & 1),
                     p.err);
        const long long fh = h_issued > p.n_bslots ? h_issued - p.n_bslots : 0;
        for (long long i = fh; i < h_issued; ++i)
          mbar_drain(&sm.full_h[i % p.n_bslots], static_cast<uint32_t>((i / p.n_bslots) & 1),
                     p.err);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------------------------------------------- MMA issuer --
      Ring rw, rh, racc;
      bool ok = true, skipped = false;
      for (int g = 0; g < pl.n_groups && ok && !skipped; ++g) {
        const uint32_t n = static_cast<uint32_t>((pl.group_rows(g) + 15) & ~15);
        const uint32_t idesc = idesc_bf16_f32(kRowsM, n);
        if (!mbar_wait(&sm.acce[racc.slot], racc.phase ^ 1u, sm.abort, p.err, kErrWaitAccEmpty)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(racc.slot * kRowsGroupRows);
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(&sm.full_h[rh.slot], rh.phase, sm.abort, p.err, kErrWaitFull)) {
            ok = false;
            break;
          }
          if (spec && *sm.skip) {
            skipped = true;
            break;
          }
          if (!mbar_wait(&sm.full_w[rw.slot], rw.phase, sm.abort, p.err, kErrWaitFull)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_addr = smem_addr(sm.h + static_cast<size_t>(rh.slot) * h_stride);
          const uint32_t b_addr = smem_addr(sm.w + static_cast<size_t>(rw.slot) * kRowsWStage);
#pragma unroll
          for (int kk = 0; kk < kBlockK / 16; ++kk)
            mma_bf16(d_tmem, sdesc_k_sw128(a_addr + kk * 32), sdesc_k_sw128(b_addr + kk * 32),
                     idesc, (kb | kk) != 0 ? 1u : 0u);
          mma_commit(&sm.empty_w[rw.slot]);
          mma_commit(&sm.empty_h[rh.slot]);
          rw.next(p.n_stages);
          rh.next(p.n_bslots);
        }
        if (!ok || skipped) break;
        mma_commit(&sm.accf[racc.slot]);
        racc.next(2);
      }
      if (!ok || skipped) {
        // Abort or stop: wait for every MMA already issued before tensor
        // memory is freed, then release the epilogue.
        mma_commit(sm.drain);
        mbar_drain(sm.drain, 0, p.err);
      }
      if (skipped) mbar_arrive(&sm.accf[racc.slot]);
    }
    __syncwarp();
  } else {
    // --------------------------------------------------------- epilogue --
    const int quarter = warp & 3;  // tensor-memory lanes 32 quarter .. 32 quarter + 31
    const uint32_t lane_base = static_cast<uint32_t>(quarter * 32) << 16;
    const int row = quarter * 32 + lane;
    const bool active = quarter * 32 < M;  // warp-uniform: some lane holds a row
    float m = kNegBig, s = 0.0f;
    int ix = INT_MAX;
    float rs = kLog2e;
    if constexpr (kNorm) {
      // The final RMSNorm's row scales, from the step's rows while the first
      // group accumulates.  Nothing here depends on an earlier kernel, so the
      // accumulators are drained as in a step without the norm.
      __shared__ float s_scale[kRowsM];
      epilogue_row_scales(p.hid, M, p.H, p.norm_eps, s_scale, warp - 2, lane);
      if (row < M) rs = kLog2e * s_scale[row];
    }
    Ring racc;
    bool ok = true;
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
      if (active) {
        const uint32_t tbase =
            tmem_base + lane_base + static_cast<uint32_t>(racc.slot * kRowsGroupRows);
        const int vbase = pl.group_row0(g);
        const int gr = pl.group_rows(g);
        const int nch = (gr + 31) >> 5;
#pragma unroll 1
        for (int c = 0; c < nch; ++c) {
          uint32_t x[32];
          tmem_ld_32cols(tbase + static_cast<uint32_t>(32 * c), x);
          tmem_ld_wait();
          const int v0 = vbase + 32 * c;
          // vocabulary rows past the group's (stale stage bytes) or past V
          const int nvalid = min(min(32, gr - 32 * c), p.V - v0);
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
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.acce[racc.slot]);
      racc.next(2);
    }
    if (ok && row < M) {
      // The previous step's commit reads the same partial buffer.
      grid_dependency_wait();
      p.part[static_cast<size_t>(row) * gridDim.x + cta] = make_float4(m, s, __int_as_float(ix), 0.0f);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kRowsTmemCols);
  }
  fused_step_commit(p.cp, sm.w);
}

}  // namespace cai
