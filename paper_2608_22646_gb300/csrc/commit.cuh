// The commit rule of CAI-dLLM (arXiv 2608.22646, Algorithm 1 with Boxes 2-7)
// for one sequence, run by one CTA, and the end-of-step bookkeeping (the next
// step's masked-row list and the host-visible record).  Shared by the merge
// kernel of the multi-kernel step and by the single-kernel step, whose last
// LM-head CTA runs it.
#pragma once

#include <cstdint>

#include "ptx.cuh"
#include "softmax.cuh"

namespace cai {

constexpr int kMask = -1;
enum : int { kRunning = 0, kExitDone = 1, kExitGrind = 2, kExitTmax = 3 };
enum : uint32_t {
  kFlagGating = 1u,
  kFlagPosFactor = 2u,
  kFlagFlush = 4u,
  kFlagQuarterPos = 8u,
  kFlagQuarterBlocks = 16u,
  kFlagDiag = 128u
};
constexpr int kMaxP = 256;
constexpr int kPosPerWarp = 6;   // positions whose partials a warp loads at once
constexpr int kPartPerLane = 5;  // partial slots a lane loads per position (G <= 160)

// Host-visible record of the last committed step, one 64-bit word in mapped
// pinned memory written by a single store (so the host never sees a torn
// record): bits 0-31 step id + 1, bit 32 every sequence has exited the block,
// bit 33 the device error word is non-zero, bits 34-48 the block index.
struct HostFlag {
  unsigned long long word;  // 0 = no step committed yet
  unsigned long long pad;
};
__host__ __device__ inline unsigned long long host_flag_word(int step_id, bool all_done, bool err,
                                                             int blk) {
  return static_cast<unsigned long long>(static_cast<uint32_t>(step_id) + 1u) |
         (static_cast<unsigned long long>(all_done ? 1u : 0u) << 32) |
         (static_cast<unsigned long long>(err ? 1u : 0u) << 33) |
         (static_cast<unsigned long long>(static_cast<uint32_t>(blk) & 0x7FFFu) << 34);
}

struct StateArrays {
  int* tok;
  float* conf;
  float* s0;
  uint8_t* budget;
  int16_t* cstep;
  int* cand;
  int* ell;
  int* eta;
  int* exit_reason;
  int* exit_step;
  int* unresolved;
  int* m_hist;
  uint8_t* run;     // diagnostics: consecutive decoded steps with the same argmax
  int16_t* stable;  // diagnostics: stability step t_i^*, -1
  float* drift;     // diagnostics: [B, n_blocks, T] relative drift D^(t)
};

struct CommitParams {
  const float4* part;     // [rows, n_part] softmax partials of this step
  int n_part;             // partial slots per row (one per LM-head CTA)
  const float4* rowres;   // [rows] merged triple per row when the pair kernel decoded the step
  int pair_min_M;         // steps with at least this many rows ran the pair kernel
  int pair_pairs;         // pairs of the pair kernel's grid
  int pair_swap_max_n;    // the pair kernel's orientation rule (pair_swapped)
  int identity_rows;      // 1: row of (b, p) is b P + p; 0: row_of[b P + p]
  int prefetch_state;     // merge kernel: read the sequence's state before waiting for the
                          // LM head (the kernel before it starts only after its own wait)
  StateArrays st;
  int* list;
  int* row_of;
  int* d_M;
  int* m_hist_slot;       // this step's M_t (written by the single-kernel step)
  unsigned* ticket;       // zero between launches
  unsigned long long* pub;  // (step id + 1) << 32 | masked rows left, written by finish_step
  HostFlag* hf;           // device alias of the mapped host record
  uint32_t* err;
  int B, P, L, n_blocks, T, blk, t, step_id;
  int K;
  int eta_mode;           // 0 count, 1 fraction of the generation length
  float eta_bar;
  float theta_fb;
  int budget_half;        // Box 5 "p < 32" tier boundary
  int budget_late;        // Box 5 "p >= 48" tier boundary
  uint32_t flags;
  float theta_tab[kMaxP]; // theta_i(t) per position (Box 6), from the host
};

__device__ __forceinline__ int budget_tier(float s, int p, int half, int late) {
  if (s > 0.50f && p < half) return 8;
  if (s < 0.25f || p >= late) return 64;
  return 32;
}

// Per-position working set of merge_commit_sequence, in shared memory the
// caller provides (the LM-head kernel lends its drained W ring).
struct CommitSmem {
  int tok[kMaxP];      // token after this step (kMask while masked)
  int cand[kMaxP];     // argmax of the previous decoded step, then of this step
  float conf[kMaxP];   // confidence of this step
  int row[kMaxP];      // partial row of the position in this step (masked positions)
  uint8_t bud[kMaxP];  // budget before this step
  uint8_t run[kMaxP];  // diagnostics: same-argmax run before this step
  int16_t stable[kMaxP];  // diagnostics: stability step before this step
  int running;         // the sequence has not left the block
  int ell;             // low-yield counter before this step
};

// Reads what one step of Algorithm 1 needs of sequence b's state into cs, in
// one round of loads by the whole calling CTA (visible to it after its next
// __syncthreads): the block's tokens and budgets, the exit state, ell, and
// the partial row of every position.  All of it was written by the previous
// step's commit (or by the reset) except, at a block's first step, the row
// list, which the gather then makes the identity; so a commit that follows an
// LM head which itself waited for the previous step may read it before
// waiting for the partials.
__device__ __forceinline__ void commit_load(const CommitParams& p, int b, CommitSmem& cs) {
  const int tid = threadIdx.x;
  const int eb = b * p.n_blocks + p.blk;
  const size_t g0 = static_cast<size_t>(b) * p.L + p.blk * p.P;
  if (tid == 0) {
    cs.running = __ldcg(&p.st.exit_reason[eb]) == kRunning;
    cs.ell = __ldcg(&p.st.ell[b]);
  }
  const bool diag = (p.flags & kFlagDiag) != 0;
  const bool ident = p.identity_rows || p.t == 0;
  for (int pp = tid; pp < p.P; pp += blockDim.x) {
    cs.tok[pp] = __ldcg(&p.st.tok[g0 + pp]);
    cs.bud[pp] = p.st.budget[g0 + pp];
    cs.row[pp] = ident ? b * p.P + pp : __ldcg(&p.row_of[b * p.P + pp]);
    if (diag) {
      cs.cand[pp] = __ldcg(&p.st.cand[g0 + pp]);
      cs.run[pp] = __ldcg(&p.st.run[g0 + pp]);
      cs.stable[pp] = __ldcg(&p.st.stable[g0 + pp]);
    }
  }
}

// One step of Algorithm 1 for sequence b, by the whole calling CTA (blockDim.x
// a multiple of 32; every thread must call it).  The sequence's state is in
// cs (commit_load, by this call unless `loaded`); warps merge the partials of
// the still-masked positions (kPPW at a time, all loads issued before any
// merge) and lane 0 applies the commit rule (Box 6, Eq. position_commit,
// with the step-zero init of Boxes 2 and 5); thread 0 updates the low-yield
// counter and the exit state (Box 7, Algorithm 1).  Global state is only
// written, never re-read.  Returns, in every thread, the positions decoded
// (M_t of the sequence) and, in *left_after, the positions still masked
// afterwards in a running sequence.
template <int kPPW = kPosPerWarp>
__device__ int merge_commit_sequence(const CommitParams& p, int b, CommitSmem& cs,
                                     const float4* part, int n_part, int* left_after = nullptr,
                                     bool loaded = false) {
  __shared__ int s_eta, s_left, s_reason, s_unres;
  int* s_tok = cs.tok;
  int* s_cand = cs.cand;
  float* s_conf = cs.conf;
  uint8_t* s_bud = cs.bud;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nwarps = blockDim.x >> 5;
  const int eb = b * p.n_blocks + p.blk;
  const size_t g0 = static_cast<size_t>(b) * p.L + p.blk * p.P;
  if (!loaded) commit_load(p, b, cs);
  if (tid == 0) {
    s_eta = 0;
    s_left = 0;
    s_reason = kRunning;
    s_unres = 0;
  }
  const bool diag = (p.flags & kFlagDiag) != 0;
  __syncthreads();
  const bool running = cs.running != 0;
  const bool gating = (p.flags & kFlagGating) != 0;

  if (running) {
    for (int base = warp; base < p.P; base += nwarps * kPPW) {
      int row[kPPW];
      float4 q[kPPW][kPartPerLane];
#pragma unroll
      for (int j = 0; j < kPPW; ++j) {
        const int pp = base + j * nwarps;
        row[j] = -1;
        if (pp < p.P && s_tok[pp] == kMask) {
          row[j] = cs.row[pp];
          if (!CAI_IN_RANGE(row[j] < p.B * p.P, p.err)) row[j] = -2;
          if (row[j] < 0) {
            if (lane == 0) atomicOr(p.err, kErrBadRow);
            row[j] = -2;
          }
        }
      }
#pragma unroll
      for (int j = 0; j < kPPW; ++j) {
        const float4* pr = part + static_cast<size_t>(row[j] < 0 ? 0 : row[j]) * n_part;
#pragma unroll
        for (int u = 0; u < kPartPerLane; ++u) {
          const int k = lane + 32 * u;
          q[j][u] = (row[j] >= 0 && k < n_part)
                        ? __ldcg(pr + k)
                        : make_float4(kNegBig, 0.0f, __int_as_float(INT_MAX), 0.0f);
        }
      }
#pragma unroll
      for (int j = 0; j < kPPW; ++j) {
        if (row[j] < 0) continue;  // warp-uniform
        const int pp = base + j * nwarps;
        float m = kNegBig, s = 0.0f;
        int ix = INT_MAX;
#pragma unroll
        for (int u = 0; u < kPartPerLane; ++u)
          merge_tri(m, s, ix, q[j][u].x, q[j][u].y, __float_as_int(q[j][u].z));
        for (int k = lane + 32 * kPartPerLane; k < n_part; k += 32) {
          const float4 r = __ldcg(part + static_cast<size_t>(row[j]) * n_part + k);
          merge_tri(m, s, ix, r.x, r.y, __float_as_int(r.z));
        }
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) {
          const float mo = __shfl_xor_sync(0xffffffffu, m, off);
          const float so = __shfl_xor_sync(0xffffffffu, s, off);
          const int io = __shfl_xor_sync(0xffffffffu, ix, off);
          merge_tri(m, s, ix, mo, so, io);
        }
        if (lane == 0) {
          const size_t g = g0 + pp;
          const float c = 1.0f / s;  // max_v p_v = exp(m - LSE) = 1 / sum_v exp(z_v - m)
          int bud = s_bud[pp];
          if (p.t == 0) {
            bud = budget_tier(c, pp, p.budget_half, p.budget_late);
            p.st.s0[g] = c;
            p.st.budget[g] = static_cast<uint8_t>(bud);
          }
          if (diag) {
            // Section 2.1: stable once the argmax has held for three decoded steps.
            const int run = (p.t > 0 && s_cand[pp] == ix) ? cs.run[pp] + 1 : 1;
            p.st.run[g] = static_cast<uint8_t>(run < 255 ? run : 255);
            if (run >= 3 && cs.stable[pp] < 0) p.st.stable[g] = static_cast<int16_t>(p.t);
          }
          p.st.conf[g] = c;
          p.st.cand[g] = ix;
          s_conf[pp] = c;
          s_cand[pp] = ix;
          const bool by_conf = c >= p.theta_tab[pp];
          const bool by_budget = gating && p.t >= bud;
          if (by_conf || by_budget) {
            s_tok[pp] = ix;
            p.st.tok[g] = ix;
            p.st.cstep[g] = static_cast<int16_t>(p.t);
            atomicAdd(&s_eta, 1);
          } else {
            atomicAdd(&s_left, 1);
          }
        }
      }
    }
  }
  __syncthreads();
  if (running && tid == 0) {
    const int eta = s_eta;
    p.st.eta[b] = eta;
    const bool low = p.eta_mode == 1
                         ? (static_cast<double>(eta) / (static_cast<double>(p.n_blocks) * p.P) <
                            static_cast<double>(p.eta_bar))
                         : (static_cast<float>(eta) < p.eta_bar);
    // Algorithm 1 sets ell <- 0 before the block's first step.
    const int ell = low ? (p.t == 0 ? 0 : cs.ell) + 1 : 0;
    p.st.ell[b] = ell;
    int reason = kRunning;
    if (gating && ell >= p.K)
      reason = kExitGrind;
    else if (s_left == 0)
      reason = kExitDone;
    else if (p.t == p.T - 1)
      reason = kExitTmax;
    s_reason = reason;
  }
  __syncthreads();
  const int reason = s_reason;
  const int decoded = s_eta + s_left;
  if (running && reason != kRunning) {
    for (int pp = tid; pp < p.P; pp += blockDim.x) {
      if (s_tok[pp] != kMask) continue;
      const size_t g = g0 + pp;
      if ((reason == kExitGrind && s_conf[pp] > p.theta_fb) || (p.flags & kFlagFlush)) {
        p.st.tok[g] = s_cand[pp];
        p.st.cstep[g] = static_cast<int16_t>(p.t);
      } else {
        atomicAdd(&s_unres, 1);
      }
    }
    __syncthreads();
    if (tid == 0) {
      p.st.exit_reason[eb] = reason;
      p.st.exit_step[eb] = p.t;
      p.st.unresolved[eb] = s_unres;
    }
  }
  if (left_after) *left_after = (running && reason == kRunning) ? s_left : 0;
  __syncthreads();
  return decoded;
}

// Compact, in (b, p) order, the still-masked tokens of running sequences of
// block blk into list / row_of; returns the count.  One CTA (blockDim.x a
// multiple of 32, at most 1024).  Reads bypass L1: other CTAs wrote this state.
__device__ int build_masked_list(const int* tok, const int* exit_reason, int* list, int* row_of,
                                 int B, int P, int L, int n_blocks, int blk) {
  __shared__ int s_wsum[32];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nwarps = blockDim.x >> 5;
  const int BP = B * P;
  int base = 0;
  for (int i0 = 0; i0 < BP; i0 += blockDim.x) {
    const int i = i0 + tid;
    bool mk = false;
    if (i < BP) {
      // Both loads issued before either is tested (one round trip, not two).
      const int b = i / P, pp = i - b * P;
      const int tk = __ldcg(&tok[static_cast<size_t>(b) * L + blk * P + pp]);
      const int ex = __ldcg(&exit_reason[b * n_blocks + blk]);
      mk = (tk == kMask) & (ex == kRunning);
    }
    const unsigned bal = __ballot_sync(0xffffffffu, mk);
    const int wpre = __popc(bal & ((1u << lane) - 1u));
    if (lane == 0) s_wsum[warp] = __popc(bal);
    __syncthreads();
    int woff = 0, tot = 0;
    for (int w = 0; w < nwarps; ++w) {
      const int c = s_wsum[w];
      woff += (w < warp) ? c : 0;
      tot += c;
    }
    if (i < BP) {
      if (mk) {
        list[base + woff + wpre] = i;
        row_of[i] = base + woff + wpre;
      } else {
        row_of[i] = -1;
      }
    }
    base += tot;
    __syncthreads();
  }
  return base;
}

// End of a step, by the last CTA: the next step's list (multi-kernel step
// only; the single-kernel step decodes every row and needs none), M_{t+1},
// the reset ticket and the host-visible record.  `remaining` is the masked
// count of running sequences when the caller already knows it (-1: count).
__device__ void finish_step(const CommitParams& p, int remaining = -1) {
  const int n = remaining >= 0 ? remaining
                               : build_masked_list(p.st.tok, p.st.exit_reason, p.list, p.row_of,
                                                   p.B, p.P, p.L, p.n_blocks, p.blk);
  if (threadIdx.x == 0) {
    *p.d_M = n;
    *p.ticket = 0u;
    const bool err = *reinterpret_cast<volatile uint32_t*>(p.err) != 0u;
    // The host uses this word only for control flow; it reads the state
    // itself through stream-ordered copies, so no system fence is needed.
    *reinterpret_cast<volatile unsigned long long*>(&p.hf->word) =
        host_flag_word(p.step_id, n == 0, err, p.blk);
    // Device copy for the next step, which may already be running (see the
    // LM-head kernel): it stops early when this step left nothing masked.
    *reinterpret_cast<volatile unsigned long long*>(p.pub) =
        (static_cast<unsigned long long>(static_cast<uint32_t>(p.step_id + 1)) << 32) |
        static_cast<uint32_t>(n);
  }
}

}  // namespace cai
