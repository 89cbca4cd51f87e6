// The two light kernels around the LM head in one denoising step:
//   gather_rows_kernel    copies the hidden rows of the step's masked
//                         positions into the compact [rows_cap, H] operand;
//   merge_commit_kernel   merges the per-CTA softmax partials into c_i and the
//                         argmax, then runs the commit rule of Algorithm 1
//                         (arXiv 2608.22646) for one sequence per CTA; the last
//                         CTA to finish builds the next step's masked-row list.
#pragma once

#include <cuda_bf16.h>
#include "head_kernel.cuh"
#include "pair_kernel.cuh"

namespace cai {

constexpr int kGatherRowsPerCta = 4;
constexpr int kGatherVecs = 8;       // 16-byte loads in flight per gather thread (H <= 4096 in one round)
constexpr int kGatherThreads = 256;
constexpr int kListThreads = 256;    // rebuild_list_kernel
// Merge kernel: one CTA per sequence, 16 warps of 4 positions each, so that
// a 64-position block merges in one round of loads and the last CTA builds
// the next step's list 512 tokens at a time (measured against 256 threads of
// 6 positions: see the design notes).
constexpr int kCommitThreads = 512;
constexpr int kCommitPPW = 4;

// ------------------------------------------------------------ gather (K1) --

struct GatherParams {
  const __nv_bfloat16* hidden;  // [B P, H] hidden states of the current block
  __nv_bfloat16* hc;            // [rows_cap, H] compact operand of the LM head
  int* list;                    // [B P] token (b P + p) of each masked row
  int* row_of;                  // [B P] row of each token in this step's list, -1
  int* d_M;                     // masked rows of this step
  uint32_t* err;                // error word (CAI_DEBUG range checks)
  int B, BP, H;
  int first;                    // step zero: every position of every sequence
  float* inv_r;                 // final norm: 1 / sqrt(mean h^2 + eps) per row, or null
  float eps;
  const unsigned long long* stage_word;  // host rows staged by the side stream: read
  unsigned long long stage_seq;          // once *stage_word >= stage_seq (or null)
};

__global__ void __launch_bounds__(kGatherThreads)
    gather_rows_kernel(const GatherParams p) {
  grid_launch_dependents();  // every thread: the CTA counts once all of them have
  grid_dependency_wait();  // the previous step's merge wrote list, row_of and d_M
  if (p.stage_word) {
    // The side stream's copy of the rows: one thread waits (bounded) for its
    // word; on giving up the error word is set and the step's results are
    // not to be used (the host reads the error with them).
    __shared__ volatile int s_abort;
    if (threadIdx.x == 0) {
      s_abort = 0;
      wait_word_ge(p.stage_word, p.stage_seq, &s_abort, p.err, kErrWaitRows);
    }
    __syncthreads();
  }
  const int M = p.first ? p.BP : *p.d_M;
  if (p.first) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < p.BP; i += gridDim.x * blockDim.x) {
      p.list[i] = i;
      p.row_of[i] = i;
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) *p.d_M = p.BP;
  }
  const int rows_pad = (M + 15) & ~15;
  const int r = blockIdx.x * kGatherRowsPerCta + threadIdx.x / 64;
  const int t = threadIdx.x & 63;
  const int nvec = p.H / 8;  // 16-byte vectors per row
  float ss = 0.0f;
  if (r < rows_pad) {
    uint4* dst = reinterpret_cast<uint4*>(p.hc + static_cast<size_t>(r) * p.H);
    if (r < M) {
      int src_row = p.first ? r : p.list[r];
      if (!CAI_IN_RANGE(src_row >= 0 && src_row < p.BP, p.err)) src_row = 0;
      const uint4* src =
          reinterpret_cast<const uint4*>(p.hidden + static_cast<size_t>(src_row) * p.H);
      // All of a thread's loads are issued before its first store (the
      // compiler cannot reorder them: dst and src could alias as far as it
      // knows), so a row costs one memory round trip, not one per vector.
      for (int v0 = t; v0 < nvec; v0 += 64 * kGatherVecs) {
        uint4 x[kGatherVecs];
#pragma unroll
        for (int j = 0; j < kGatherVecs; ++j) {
          const int v = v0 + 64 * j;
          x[j] = v < nvec ? __ldg(src + v) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int j = 0; j < kGatherVecs; ++j) {
          const int v = v0 + 64 * j;
          if (v < nvec) {
            dst[v] = x[j];
            if (p.inv_r) ss += sumsq8(x[j]);
          }
        }
      }
    } else {
      for (int v = t; v < nvec; v += 64) dst[v] = make_uint4(0u, 0u, 0u, 0u);
    }
  }
  if (!p.inv_r) return;
  // A row's 64 threads are two whole warps: reduce in each, then across the two.
  __shared__ float s_half[kGatherThreads / 32];
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
  if ((threadIdx.x & 31) == 0) s_half[threadIdx.x >> 5] = ss;
  __syncthreads();
  if (t == 0 && r < rows_pad) {
    const float tot = s_half[threadIdx.x >> 5] + s_half[(threadIdx.x >> 5) + 1];
    p.inv_r[r] = r < M ? rsqrtf(tot / static_cast<float>(p.H) + p.eps) : 1.0f;
  }
}

// ----------------------------------------------------------- diagnostics --

struct DriftParams {
  const __nv_bfloat16* hidden;  // [B P, H] this step's rows (every position of the block)
  __nv_bfloat16* prev;          // [B P, H] the previous step's rows (kept by this kernel)
  float* drift;                 // [B, n_blocks, T]
  int P, H, n_blocks, T, blk, t;
};

// One CTA per sequence: D^(t) = mean over the block's positions of
// ||h^(t) - h^(t-1)|| / ||h^(t-1)|| (Eq. relative_drift; fp32 sums of the bf16
// rows), then this step's rows become the previous ones.  At t = 0 only the
// copy is made.
__global__ void __launch_bounds__(kGatherThreads) drift_kernel(const DriftParams p) {
  __shared__ float s_sum[kGatherThreads / 32];
  grid_launch_dependents();  // every thread: the CTA counts once all of them have
  grid_dependency_wait();    // the previous step's drift kernel wrote prev
  const int b = blockIdx.x, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nw = blockDim.x >> 5, nvec = p.H / 8;
  float acc = 0.0f;
  for (int pp = warp; pp < p.P; pp += nw) {
    const size_t row = static_cast<size_t>(b) * p.P + pp;
    const uint4* cur = reinterpret_cast<const uint4*>(p.hidden + row * p.H);
    uint4* prv = reinterpret_cast<uint4*>(p.prev + row * p.H);
    float num = 0.0f, den = 0.0f;
    for (int v = lane; v < nvec; v += 32) {
      const uint4 x = __ldg(cur + v);
      if (p.t > 0) {
        const uint4 y = prv[v];
        const __nv_bfloat16* xe = reinterpret_cast<const __nv_bfloat16*>(&x);
        const __nv_bfloat16* ye = reinterpret_cast<const __nv_bfloat16*>(&y);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const float a = __bfloat162float(ye[i]);
          const float d = __bfloat162float(xe[i]) - a;
          num = fmaf(d, d, num);
          den = fmaf(a, a, den);
        }
      }
      prv[v] = x;
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) {
      num += __shfl_xor_sync(0xffffffffu, num, off);
      den += __shfl_xor_sync(0xffffffffu, den, off);
    }
    acc += sqrtf(num) / sqrtf(den);
  }
  if (lane == 0) s_sum[warp] = acc;
  __syncthreads();
  if (threadIdx.x == 0 && p.t > 0) {
    float tot = 0.0f;
    for (int w = 0; w < nw; ++w) tot += s_sum[w];
    p.drift[(static_cast<size_t>(b) * p.n_blocks + p.blk) * p.T + p.t] = tot / static_cast<float>(p.P);
  }
}

// ------------------------------------------------- bounded-wait test hook --

// Waits, through the same bounded mbar_wait every step kernel uses, on a
// barrier nothing arrives at: after the wait limit it records `site` in the
// error word and returns (no trap, no fault; the context stays valid until
// the host reads the word).
__global__ void wait_timeout_probe_kernel(uint32_t* err, uint32_t site) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_wait(&bar, 0, &abort_flag, err, site);
}

// ------------------------------------------------------ list rebuild -----

struct ListParams {
  const int* tok;
  const int* exit_reason;
  int* list;
  int* row_of;
  int* d_M;
  int B, P, L, n_blocks, blk;
};

// Rebuild the masked-row list from the state (after a state upload).
__global__ void __launch_bounds__(kListThreads) rebuild_list_kernel(const ListParams p) {
  const int n = build_masked_list(p.tok, p.exit_reason, p.list, p.row_of, p.B, p.P, p.L,
                                  p.n_blocks, p.blk);
  if (threadIdx.x == 0) *p.d_M = n;
}

// ------------------------------------------ vocabulary-parallel head (shards) --

// A shard context holds the rows [v_off, v_off + V_shard) of W.  After its
// LM head, shard_rows_kernel reduces each masked row's partials into one
// triple (max * log2 e, sum of 2^(z log2 e - max), argmax as a global
// vocabulary index) in the exchange buffer; rows past M get the empty triple.
// Box 1's max, sum of exponentials and lowest-index argmax over the whole
// vocabulary are exact merges of these triples over the shards, which
// shard_merge_kernel does for every row before the commit.
constexpr int kShardThreads = 256;

struct ShardRowsParams {
  const float4* part;    // [rows, per_row] pair partials of this step (local indices)
  const float4* rowres;  // [rows] merged triple when the step wrote per-tile partials
  const int* d_M;
  float4* out;           // [rows_cap] exchange buffer
  int rows_cap;
  int n_pairs;           // the pair kernel's pairs
  int swap_max_n;        // its orientation rule
  int v_off;             // first vocabulary row of this shard
};

__global__ void __launch_bounds__(kShardThreads) shard_rows_kernel(const ShardRowsParams p) {
  grid_launch_dependents();  // every thread: the CTA counts once all of them have
  grid_dependency_wait();    // the pair kernel's partials (and the row merge's)
  const int M = *p.d_M;
  const int per_row = M > 0 ? pair_partials_per_row(M, p.n_pairs, pair_swapped(M, p.swap_max_n)) : 0;
  const int lane = threadIdx.x & 31;
  const int nw = (gridDim.x * blockDim.x) >> 5;
  for (int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; row < p.rows_cap; row += nw) {
    float m = kNegBig, s = 0.0f;
    int ix = INT_MAX;
    if (row < M) {
      if (per_row > 0) {
        for (int k = lane; k < per_row; k += 32) {
          const float4 a = __ldcg(p.part + static_cast<size_t>(row) * per_row + k);
          merge_tri(m, s, ix, a.x, a.y, __float_as_int(a.z));
        }
      } else if (lane == 0) {
        const float4 a = __ldcg(p.rowres + row);
        merge_tri(m, s, ix, a.x, a.y, __float_as_int(a.z));
      }
#pragma unroll
      for (int off = 16; off >= 1; off >>= 1) {
        const float mo = __shfl_xor_sync(0xffffffffu, m, off);
        const float so = __shfl_xor_sync(0xffffffffu, s, off);
        const int io = __shfl_xor_sync(0xffffffffu, ix, off);
        merge_tri(m, s, ix, mo, so, io);
      }
    }
    if (lane == 0)
      p.out[row] = make_float4(m, s, __int_as_float(ix == INT_MAX ? INT_MAX : ix + p.v_off), 0.0f);
  }
}

struct ShardMergeParams {
  const float4* gathered;  // [n_shards, rows_cap] every shard's exchange buffer, any order
  float4* rowres;          // [rows_cap] merged triple per row, read by the commit
  const int* d_M;
  int rows_cap, n_shards;
};

// One warp per masked row: the merge of the row's triples from every shard.
__global__ void __launch_bounds__(kShardThreads) shard_merge_kernel(const ShardMergeParams p) {
  grid_launch_dependents();  // every thread: the CTA counts once all of them have
  grid_dependency_wait();    // the previous commit's M and rowres readers
  const int M = *p.d_M;
  const int lane = threadIdx.x & 31;
  const int nw = (gridDim.x * blockDim.x) >> 5;
  for (int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; row < M; row += nw) {
    float m = kNegBig, s = 0.0f;
    int ix = INT_MAX;
    for (int k = lane; k < p.n_shards; k += 32) {
      const float4 a = __ldcg(p.gathered + static_cast<size_t>(k) * p.rows_cap + row);
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

// ------------------------------------------------------ merge + commit (K3) --

// One CTA per sequence: merge_commit_sequence for sequence blockIdx.x, then the
// last CTA to finish (atomic ticket; none needed for a single CTA) builds the
// next step's list and publishes the step.
__global__ void __launch_bounds__(kCommitThreads) merge_commit_kernel(const CommitParams p) {
  __shared__ int s_last;
  __shared__ CommitSmem cs;
  grid_launch_dependents();  // every thread: the CTA counts once all of them have
  // This step's M (d_M is rewritten only by the last CTA, after every CTA's
  // merge; at a block's first step every row is decoded) tells which LM-head
  // kernel decoded it: the pair kernel's tile partials were already merged
  // into one triple per row.  With prefetch_state, the kernel before this one
  // started only after the previous step had finished, so M and the
  // sequence's state are read before waiting for this step's partials.
  int M = 0;
  if (p.prefetch_state) {
    M = p.t == 0 ? p.B * p.P : __ldcg(p.d_M);
    commit_load(p, blockIdx.x, cs);
  }
  grid_dependency_wait();    // partials of this step (and state of the previous one)
  if (!p.prefetch_state) M = *p.d_M;
  const bool loaded = p.prefetch_state != 0;
  if (M >= p.pair_min_M) {
    const int per_row =
        pair_partials_per_row(M, p.pair_pairs, pair_swapped(M, p.pair_swap_max_n));
    if (per_row > 0)
      merge_commit_sequence<kCommitPPW>(p, blockIdx.x, cs, p.part, per_row, nullptr, loaded);
    else
      merge_commit_sequence<kCommitPPW>(p, blockIdx.x, cs, p.rowres, 1, nullptr, loaded);
  } else {
    merge_commit_sequence<kCommitPPW>(p, blockIdx.x, cs, p.part, p.n_part, nullptr, loaded);
  }
  if (gridDim.x > 1) {
    if (threadIdx.x == 0) {
      __threadfence();
      s_last = atomicAdd(p.ticket, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
  }
  finish_step(p);
}

}  // namespace cai
