// LM-head projection fused with the full-vocabulary softmax reduction
// (Box 1 of arXiv 2608.22646: c_i = max_v p_theta(x_i = v), argmax_v p_theta).
//
// The masked positions of a step are few (M_t <= B P), so the contraction is
// run with A and B swapped: the vocabulary fills the MMA M dimension (128 rows
// of W per accumulator tile) and the positions form the N dimension
// (16..256 columns, rounded up to 16).  Each CTA owns a contiguous range of W
// rows in units of 64 rows and streams it once from HBM through a ring of
// K = 64 stages, and keeps the logits in tensor memory: they are never
// written anywhere.
//
// W is read from a packed copy made once per context (pack_weight_kernel) in
// exactly the order the CTAs consume it: CTA c owns rows [64 u0, 64 u1) and
// the bytes [128 H u0, 128 H u1) of the packed copy, laid out tile by tile and
// k block by k block, each stage already in the 128-byte-swizzled K-major
// layout the MMA descriptors expect.  Every CTA therefore streams one
// contiguous region front to back with one bulk copy per stage; contiguous
// copies keep DRAM pages open, the strided 128-byte rows of a 2-D tensor box
// do not.
#pragma once

#include <climits>
#include "ptx.cuh"

namespace cai {

constexpr int kRowsPerTile = 128;  // MMA M: vocabulary rows per accumulator
constexpr int kUnitRows = 64;      // granularity of the per-CTA split of V
constexpr int kBlockK = 64;        // K per stage: one 128-byte swizzled row of bf16
constexpr int kChunkN = 256;       // largest MMA N (positions per pass over W)
constexpr int kBoxRowsB = 16;      // rows per TMA box of the hidden tile
constexpr int kHeadThreads = 192;
constexpr int kATileBytes = kRowsPerTile * kBlockK * 2;  // 16 KiB
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kNegBig = -3.0e38f;  // "no logit yet": exp2(x - m) underflows to 0

struct HeadParams {
  const uint8_t* wpk; // packed W (see pack_weight_kernel)
  const int* d_M;     // masked rows of this step (device)
  int* m_hist_slot;   // where this step's M is recorded
  float4* part;       // [rows_cap, G] partial (m2, S, idx bits, 0) per CTA
  uint32_t* err;      // error word
  int V, H;
  int units;          // ceil(V / 64)
  int n_stages;
  int b_stage_bytes;  // n_max * 128
  int acc_stride;     // tensor-memory columns per accumulator buffer
  int tmem_cols;      // allocated tensor-memory columns
};

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Merge two online-softmax triples (m in log2 units, S = sum 2^(z - m), idx).
// The larger maximum keeps weight 1; ties keep the lower vocabulary index.
__device__ __forceinline__ void merge_tri(float& m, float& s, int& i, float mo, float so,
                                          int io) {
  const float e = fast_exp2(-fabsf(m - mo));
  const bool mine = m >= mo;
  const float sn = mine ? fmaf(so, e, s) : fmaf(s, e, so);
  const int in = (m > mo) ? i : ((mo > m) ? io : min(i, io));
  m = fmaxf(m, mo);
  s = sn;
  i = in;
}

// 32 rows (one per lane) x 32 columns (one register each) -> lane l holds the
// (max, sum, argmax) of column l over the 32 rows.  Five halving steps: at
// width w each lane keeps half of its live columns and receives the partner's
// copy of the same columns (31 merges per lane, one exponential each).
__device__ __forceinline__ void transpose_reduce32(const uint32_t (&v)[32], bool valid, int vrow,
                                                   int lane, float& om, float& os, int& oi) {
  float m[32], s[32];
  int ix[32];
#pragma unroll
  for (int c = 0; c < 32; ++c) {
    m[c] = valid ? __uint_as_float(v[c]) * kLog2e : kNegBig;
    s[c] = valid ? 1.0f : 0.0f;
    ix[c] = valid ? vrow : INT_MAX;
  }
#pragma unroll
  for (int w = 16; w >= 1; w >>= 1) {
    const bool up = (lane & w) != 0;
#pragma unroll
    for (int c = 0; c < w; ++c) {
      float km = up ? m[c + w] : m[c];
      float ks = up ? s[c + w] : s[c];
      int ki = up ? ix[c + w] : ix[c];
      const float sm = up ? m[c] : m[c + w];
      const float ss = up ? s[c] : s[c + w];
      const int si = up ? ix[c] : ix[c + w];
      const float rm = __shfl_xor_sync(0xffffffffu, sm, w);
      const float rs = __shfl_xor_sync(0xffffffffu, ss, w);
      const int ri = __shfl_xor_sync(0xffffffffu, si, w);
      merge_tri(km, ks, ki, rm, rs, ri);
      m[c] = km;
      s[c] = ks;
      ix[c] = ki;
    }
  }
  om = m[0];
  os = s[0];
  oi = ix[0];
}

// First 64-row unit of CTA c when `units` units are split over G CTAs.
__host__ __device__ inline int unit_begin(int c, int units, int G) {
  return static_cast<int>((static_cast<long long>(c) * units) / G);
}

// Byte offset in the packed weight of the stage (tile j, k block kb) of a CTA
// whose range starts at unit u0; rows = 128, or 64 for a final half tile.
__host__ __device__ inline size_t packed_stage(int u0, int j, int kb, int rows, int H) {
  return static_cast<size_t>(u0) * 128 * H + static_cast<size_t>(j) * 256 * H +
         static_cast<size_t>(kb) * rows * 128;
}

// Pack W [V, H] (row-major bf16) for a grid of G CTAs over `units` 64-row
// units.  Inside a stage block, row r's 16-byte chunk c (k = 8c..8c+7 of the
// block's 64) sits at r * 128 + ((c ^ (r & 7)) * 16): the 128-byte swizzle of
// 8-row, 1024-byte atoms.  Rows >= V are zero.  One thread per destination
// 16-byte chunk; n_chunks = units * 64 * H / 8.
__global__ void pack_weight_kernel(const uint4* __restrict__ W, uint4* __restrict__ out, int V,
                                   int H, int units, int G, long long n_chunks) {
  const long long unit_bytes = 128ll * H;
  for (long long d = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; d < n_chunks;
       d += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long byte = d * 16;
    const int u = static_cast<int>(byte / unit_bytes);
    // CTA owning unit u: the largest c with unit_begin(c) <= u.
    int c = static_cast<int>((static_cast<long long>(u) * G) / units);
    while (c + 1 < G && unit_begin(c + 1, units, G) <= u) ++c;
    while (c > 0 && unit_begin(c, units, G) > u) --c;
    const int u0 = unit_begin(c, units, G), u1 = unit_begin(c + 1, units, G);
    const long long off = byte - static_cast<long long>(u0) * unit_bytes;
    const int j = static_cast<int>(off / (2 * unit_bytes));
    const long long rem = off - static_cast<long long>(j) * 2 * unit_bytes;
    const int ut = u0 + 2 * j;
    const int rows = (u1 - ut >= 2) ? 128 : 64;
    const int kb = static_cast<int>(rem / (rows * 128));
    const int inblk = static_cast<int>(rem - static_cast<long long>(kb) * rows * 128);
    const int r = inblk >> 7;
    const int cl = ((inblk >> 4) & 7) ^ (r & 7);
    const long long v = static_cast<long long>(ut) * 64 + r;
    uint4 val = make_uint4(0u, 0u, 0u, 0u);
    if (v < V) val = W[(v * H + static_cast<long long>(kb) * kBlockK) / 8 + cl];
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

struct HeadSmem {
  uint8_t* a;       // n_stages x 16 KiB
  uint8_t* b;       // n_stages x b_stage_bytes
  float4* epi;      // [2][4][acc_stride] cross-warp merge, double-buffered by chunk
  uint64_t* full;   // n_stages
  uint64_t* empty;  // n_stages
  uint64_t* accf;   // 2
  uint64_t* acce;   // 2
  uint64_t* drain;  // 1
  uint64_t* epib;   // 2: the four epilogue warps have written epi[buffer]
  uint32_t* tmem_slot;
  volatile int* abort;
};

__host__ __device__ inline size_t head_smem_bytes(int n_stages, int b_stage_bytes, int acc_stride) {
  return 1024 + (size_t)n_stages * (kATileBytes + b_stage_bytes) + (size_t)8 * acc_stride * 16 +
         (size_t)(2 * n_stages + 7) * 8 + 16;
}

__device__ __forceinline__ HeadSmem carve(uint8_t* raw, const HeadParams& p) {
  HeadSmem s;
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  s.a = base;
  s.b = s.a + (size_t)p.n_stages * kATileBytes;
  s.epi = reinterpret_cast<float4*>(s.b + (size_t)p.n_stages * p.b_stage_bytes);
  s.full = reinterpret_cast<uint64_t*>(s.epi + 8 * p.acc_stride);
  s.empty = s.full + p.n_stages;
  s.accf = s.empty + p.n_stages;
  s.acce = s.accf + 2;
  s.drain = s.acce + 2;
  s.epib = s.drain + 1;
  s.tmem_slot = reinterpret_cast<uint32_t*>(s.epib + 2);
  s.abort = reinterpret_cast<volatile int*>(s.tmem_slot + 1);
  return s;
}

// Stage (tile j, k block kb) of this CTA's packed range: one contiguous copy.
__device__ __forceinline__ void load_w_stage(uint8_t* dst, const uint8_t* wpk, int u0, int j,
                                             int rows, int kb, int H, uint64_t* bar, uint64_t pol) {
  bulk_load(dst, wpk + packed_stage(u0, j, kb, rows, H), static_cast<uint32_t>(rows * 128), bar,
            pol);
}

__global__ void __launch_bounds__(kHeadThreads, 1)
    lm_head_softmax_kernel(const __grid_constant__ CUtensorMap tm_h, const HeadParams p) {
  extern __shared__ uint8_t smem_raw[];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  HeadSmem sm = carve(smem_raw, p);

  const int G = gridDim.x;
  const int cta = blockIdx.x;
  const int u0 = unit_begin(cta, p.units, G);
  const int u1 = unit_begin(cta + 1, p.units, G);
  const int n_tiles = (u1 - u0 + 1) >> 1;
  const int KB = p.H / kBlockK;

  // Prologue (overlaps the previous kernel under programmatic dependent launch).
  if (threadIdx.x == 0) {
    for (int s = 0; s < p.n_stages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&sm.accf[a], 1);
      mbar_init(&sm.acce[a], 4);
    }
    mbar_init(sm.drain, 1);
    mbar_init(&sm.epib[0], 4);
    mbar_init(&sm.epib[1], 4);
    *sm.abort = 0;
    fence_mbar_init();
    grid_launch_dependents();
  }
  if (warp == 0 && lane == 0) prefetch_tmap(&tm_h);
  if (warp == 1) {
    tmem_alloc(sm.tmem_slot, static_cast<uint32_t>(p.tmem_cols));
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *sm.tmem_slot;

  // The weight does not depend on the previous kernels: the producer starts
  // streaming the first ring of W tiles before waiting for them.  Everything
  // that does (the masked-row count, the gathered rows, the partial buffer)
  // is touched only after grid_dependency_wait().
  const int n_pre = min(p.n_stages, n_tiles * KB);

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------ producer --
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_h = policy_evict_last();
      for (int i = 0; i < n_pre; ++i) {
        const int j = i / KB, kb = i - j * KB;
        const int ut = u0 + 2 * j;
        const int rows = (u1 - ut >= 2) ? 128 : 64;
        mbar_expect_tx(&sm.full[i], static_cast<uint32_t>(rows * 128));
        load_w_stage(sm.a + (size_t)i * kATileBytes, p.wpk, u0, j, rows, kb, p.H, &sm.full[i],
                     pol_w);
      }
      grid_dependency_wait();
      const int M = *p.d_M;
      const int n_chunks = (M + kChunkN - 1) / kChunkN;
      int stage = 0;
      uint32_t phase = 0;
      long long issued = 0;
      bool ok = true;
      for (int q = 0; q < n_chunks && ok; ++q) {
        const int n0 = q * kChunkN;
        const int nq = (min(kChunkN, M - n0) + 15) & ~15;
        for (int j = 0; j < n_tiles && ok; ++j) {
          const int ut = u0 + 2 * j;
          const int rows = (u1 - ut >= 2) ? 128 : 64;
          for (int kb = 0; kb < KB; ++kb) {
            const bool pre = issued < n_pre;  // A already in flight for this stage
            if (!pre &&
                !mbar_wait(&sm.empty[stage], phase ^ 1u, sm.abort, p.err, kErrWaitEmpty)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&sm.full[stage],
                                  static_cast<uint32_t>((pre ? 0 : rows * 128) + nq * 128));
            if (!pre)
              load_w_stage(sm.a + (size_t)stage * kATileBytes, p.wpk, u0, j, rows, kb, p.H,
                           &sm.full[stage], pol_w);
            uint8_t* bdst = sm.b + (size_t)stage * p.b_stage_bytes;
            for (int i = 0; i < nq / kBoxRowsB; ++i)
              tma_load_2d(bdst + i * kBoxRowsB * 128, &tm_h, &sm.full[stage], kb * kBlockK,
                          n0 + i * kBoxRowsB, pol_h);
            ++issued;
            if (++stage == p.n_stages) {
              stage = 0;
              phase ^= 1u;
            }
          }
        }
      }
      if (issued < n_pre) {
        // Nothing to decode (M = 0) or an abort before the prefetched stages
        // were claimed: complete their phases so the W copies can be drained.
        for (long long i = issued; i < n_pre; ++i) mbar_arrive(&sm.full[i]);
        for (long long i = issued; i < n_pre; ++i) mbar_drain(&sm.full[i], 0, p.err);
      }
      if (!ok) {
        // Abort path: let the copies already in flight land before exit.
        const long long first = issued > p.n_stages ? issued - p.n_stages : 0;
        for (long long i = first; i < issued; ++i)
          mbar_drain(&sm.full[i % p.n_stages], static_cast<uint32_t>((i / p.n_stages) & 1),
                     p.err);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------------------------------------------- MMA issuer --
      grid_dependency_wait();
      const int M = *p.d_M;
      const int n_chunks = (M + kChunkN - 1) / kChunkN;
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int q = 0; q < n_chunks && ok; ++q) {
        const int n0 = q * kChunkN;
        const int nq = (min(kChunkN, M - n0) + 15) & ~15;
        const uint32_t idesc = idesc_bf16_f32(kRowsPerTile, static_cast<uint32_t>(nq));
        for (int j = 0; j < n_tiles && ok; ++j) {
          if (!mbar_wait(&sm.acce[acc], acc_phase ^ 1u, sm.abort, p.err, kErrWaitAccEmpty)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * p.acc_stride);
          for (int kb = 0; kb < KB; ++kb) {
            if (!mbar_wait(&sm.full[stage], phase, sm.abort, p.err, kErrWaitFull)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t a_addr = smem_addr(sm.a + (size_t)stage * kATileBytes);
            const uint32_t b_addr = smem_addr(sm.b + (size_t)stage * p.b_stage_bytes);
#pragma unroll
            for (int kk = 0; kk < kBlockK / 16; ++kk) {
              mma_bf16(d_tmem, sdesc_k_sw128(a_addr + kk * 32), sdesc_k_sw128(b_addr + kk * 32),
                       idesc, (kb | kk) != 0 ? 1u : 0u);
            }
            mma_commit(&sm.empty[stage]);
            if (++stage == p.n_stages) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (!ok) break;
          mma_commit(&sm.accf[acc]);
          acc ^= 1;
          if (acc == 0) acc_phase ^= 1u;
        }
      }
      if (!ok) {
        // Abort path: wait for every MMA already issued before TMEM is freed.
        mma_commit(sm.drain);
        mbar_drain(sm.drain, 0, p.err);
      }
    }
    __syncwarp();
  } else {
    // --------------------------------------------------------- epilogue --
    grid_dependency_wait();
    const int M = *p.d_M;
    const int n_chunks = (M + kChunkN - 1) / kChunkN;
    if (threadIdx.x == 64 && cta == 0) *p.m_hist_slot = M;
    const int ew = warp - 2;       // 0..3: slot in the cross-warp merge
    const int quarter = warp & 3;  // tensor-memory lanes this warp may read
    const uint32_t lane_base = static_cast<uint32_t>(quarter * 32) << 16;
    int acc = 0;
    uint32_t acc_phase = 0;
    bool ok = true;
    for (int q = 0; q < n_chunks && ok; ++q) {
      const int n0 = q * kChunkN;
      const int nq = (min(kChunkN, M - n0) + 15) & ~15;
      const int ngroups = (nq + 31) >> 5;
      float rm[8], rs[8];
      int ri[8];
#pragma unroll
      for (int g = 0; g < 8; ++g) {
        rm[g] = kNegBig;
        rs[g] = 0.0f;
        ri[g] = INT_MAX;
      }
      for (int j = 0; j < n_tiles; ++j) {
        const int ut = u0 + 2 * j;
        const int rows = (u1 - ut >= 2) ? 128 : 64;
        const int row_local = quarter * 32 + lane;
        const int vrow = ut * kUnitRows + row_local;
        const bool valid = row_local < rows && vrow < p.V;
        if (!mbar_wait(&sm.accf[acc], acc_phase, sm.abort, p.err, kErrWaitAccFull)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t tcol = tmem_base + lane_base + static_cast<uint32_t>(acc * p.acc_stride);
#pragma unroll
        for (int g = 0; g < 8; ++g) {
          if (g < ngroups) {
            uint32_t v[32];
            tmem_ld_32cols(tcol + 32 * g, v);
            tmem_ld_wait();
            float m, s;
            int i;
            transpose_reduce32(v, valid, vrow, lane, m, s, i);
            merge_tri(rm[g], rs[g], ri[g], m, s, i);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.acce[acc]);
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
      }
      if (!ok) break;
      // Cross-warp merge of the four 32-row slices of every column, then one
      // partial per (position, CTA).  The buffer alternates by chunk: a warp
      // writes buffer q & 1 again only after every warp arrived for chunk q + 1,
      // which each does after reading chunk q.
      const int buf = q & 1;
      float4* epi = sm.epi + buf * 4 * p.acc_stride;
#pragma unroll
      for (int g = 0; g < 8; ++g) {
        if (g < ngroups)
          epi[ew * p.acc_stride + 32 * g + lane] =
              make_float4(rm[g], rs[g], __int_as_float(ri[g]), 0.0f);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.epib[buf]);
      if (!mbar_wait(&sm.epib[buf], static_cast<uint32_t>((q >> 1) & 1), sm.abort, p.err,
                     kErrWaitEpi)) {
        ok = false;
        break;
      }
      const int ncols = min(nq, M - n0);
      for (int col = ew * 32 + lane; col < ncols; col += 128) {
        const float4 a = epi[col];
        float m = a.x, s = a.y;
        int i = __float_as_int(a.z);
#pragma unroll
        for (int w = 1; w < 4; ++w) {
          const float4 b = epi[w * p.acc_stride + col];
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
}

}  // namespace cai
