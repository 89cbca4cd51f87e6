// Online-softmax triples: (m, S, idx) with m the running maximum in log2 units,
// S = sum of 2^(z - m) over the values seen, idx the lowest index reaching m.
// Merging two triples or folding in one value is exact up to fp32 rounding, so
// any split of the vocabulary reduces to max_v z, sum_v exp(z_v - max) and the
// argmax (Box 1 of arXiv 2608.22646: c = exp(max - LSE) = 1 / S).
#pragma once

#include <climits>
#include <cstdint>
#include <cuda_bf16.h>

namespace cai {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kNegBig = -3.0e38f;  // "no logit yet": exp2(x - m) underflows to 0

// Sum of squares of eight bf16 values, in fp32 (the final RMSNorm's row
// statistic).
__device__ __forceinline__ float sumsq8(uint4 x) {
  const __nv_bfloat16* e = reinterpret_cast<const __nv_bfloat16*>(&x);
  float s = 0.0f;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float f = __bfloat162float(e[i]);
    s = fmaf(f, f, s);
  }
  return s;
}

// Final RMSNorm row scales 1 / sqrt(mean h^2 + eps) of rows [0, M) of the
// [M, H] bf16 rows `hid` into s_scale (shared memory), by the four epilogue
// warps of an LM-head kernel (ew = 0..3, each a whole warp; every one must
// call it), which then meet at named barrier 1: a row at a time per warp, 32
// lanes with eight 16-byte loads each in flight.
__device__ __forceinline__ void epilogue_row_scales(const __nv_bfloat16* hid, int M, int H,
                                                    float eps, float* s_scale, int ew,
                                                    int lane) {
  const int nvec = H / 8;
  for (int r = ew; r < M; r += 4) {
    const uint4* src = reinterpret_cast<const uint4*>(hid + static_cast<size_t>(r) * H);
    float ss = 0.0f;
    for (int v0 = lane; v0 < nvec; v0 += 32 * 8) {
      uint4 x[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int v = v0 + 32 * j;
        x[j] = v < nvec ? __ldg(src + v) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) ss += sumsq8(x[j]);
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
    if (lane == 0) s_scale[r] = rsqrtf(ss / static_cast<float>(H) + eps);
  }
  asm volatile("bar.sync 1, 128;" ::: "memory");  // the four epilogue warps
}

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

// 32 lanes x 32 columns of online-softmax triples -> lane l holds the merge of
// column l over the 32 lanes, in m[0], s[0], ix[0].  Five halving steps: at
// width w each lane keeps half of its live columns and receives the partner's
// copy of the same columns (31 merges per lane, one exponential each).
__device__ __forceinline__ void transpose_merge32(float (&m)[32], float (&s)[32], int (&ix)[32],
                                                  int lane) {
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
}

// 32 rows (one per lane) x 32 columns of logits z (log2 units) -> lane l
// holds the (max, sum, argmax) of column l over the 32 rows, as
// transpose_merge32 but with the first halving step specialised: a lane's
// partner at width 16 holds vocabulary row vrow ^ 16, so only the logits are
// exchanged (16 shuffles instead of 48).  vrow is this lane's vocabulary row
// (lane-aligned: vrow % 32 == lane), valid / pvalid whether this lane's and
// the partner's rows exist.  On return m[0], s[0], ix[0] hold the column's
// triple; z is clobbered.
__device__ __forceinline__ void transpose_logits32(float (&z)[32], bool valid, bool pvalid,
                                                   int vrow, int lane, float& om, float& os,
                                                   int& oi) {
  float m[16], s[16];
  int ix[16];
  const bool up = (lane & 16) != 0;
  const float ks = valid ? 1.0f : 0.0f, rs = pvalid ? 1.0f : 0.0f;
  const int ki = valid ? vrow : INT_MAX, ri = pvalid ? (vrow ^ 16) : INT_MAX;
#pragma unroll
  for (int c = 0; c < 16; ++c) {
    const float keep = up ? z[c + 16] : z[c];
    const float send = up ? z[c] : z[c + 16];
    const float rm = __shfl_xor_sync(0xffffffffu, send, 16);
    float km = keep, kss = ks;
    int kii = ki;
    merge_tri(km, kss, kii, rm, rs, ri);
    m[c] = km;
    s[c] = kss;
    ix[c] = kii;
  }
#pragma unroll
  for (int w = 8; w >= 1; w >>= 1) {
    const bool hi = (lane & w) != 0;
#pragma unroll
    for (int c = 0; c < w; ++c) {
      float km = hi ? m[c + w] : m[c];
      float kss = hi ? s[c + w] : s[c];
      int kii = hi ? ix[c + w] : ix[c];
      const float sm = hi ? m[c] : m[c + w];
      const float ss = hi ? s[c] : s[c + w];
      const int si = hi ? ix[c] : ix[c + w];
      const float rm = __shfl_xor_sync(0xffffffffu, sm, w);
      const float rss = __shfl_xor_sync(0xffffffffu, ss, w);
      const int rii = __shfl_xor_sync(0xffffffffu, si, w);
      merge_tri(km, kss, kii, rm, rss, rii);
      m[c] = km;
      s[c] = kss;
      ix[c] = kii;
    }
  }
  om = m[0];
  os = s[0];
  oi = ix[0];
}

// 32 rows (one per lane) x 32 columns of logits -> lane l holds the
// (max, sum, argmax) of column l over the 32 rows.  Column c's logits are
// scaled by log2 e, times col_scale[c] when given (a per-row normalisation
// of the decoded hidden states, see lm_head_softmax_kernel; global or shared
// memory).
__device__ __forceinline__ void transpose_reduce32(const uint32_t (&v)[32], bool valid, int vrow,
                                                   int lane, float& om, float& os, int& oi,
                                                   const float* col_scale = nullptr) {
  float m[32], s[32];
  int ix[32];
#pragma unroll
  for (int c = 0; c < 32; ++c) {
    const float sc = col_scale ? kLog2e * col_scale[c] : kLog2e;
    m[c] = valid ? __uint_as_float(v[c]) * sc : kNegBig;
    s[c] = valid ? 1.0f : 0.0f;
    ix[c] = valid ? vrow : INT_MAX;
  }
  transpose_merge32(m, s, ix, lane);
  om = m[0];
  os = s[0];
  oi = ix[0];
}

// Fold one logit z (log2 units) of vocabulary row `row` into a running
// triple.  Rows arrive in increasing order, so only a strictly larger value
// replaces the argmax (ties keep the lower index).
__device__ __forceinline__ void online_update(float& m, float& s, int& i, float z, int row) {
  const float d = z - m;
  const float e = fast_exp2(-fabsf(d));
  const bool up = d > 0.0f;
  s = up ? fmaf(s, e, 1.0f) : s + e;
  m = up ? z : m;
  i = up ? row : i;
}

}  // namespace cai
