// Host side of the C ABI declared in include/cai.h: context ownership, argument
// validation, TMA descriptor set-up, launch sequencing of one denoising step
// (gather -> LM head + softmax -> merge + commit), the host-side threshold
// schedule (Boxes 3, 4 and 6 of arXiv 2608.22646, in double), polling and
// state transfer.
#include <cuda.h>
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include <atomic>
#include <chrono>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <thread>
#include <utility>
#include <vector>

#include "cai.h"
#include "pair_kernel.cuh"
#include "rows_kernel.cuh"
#include "step_kernels.cuh"

using namespace cai;

namespace {

std::atomic<int> g_fail_alloc_after{0};
std::atomic<int> g_head_grid_limit{0};

// Programmatic dependent launch between the step's kernels; CAI_PDL=0 in the
// environment turns it off (read once per context at cai_init).
// Largest B P that runs single-kernel steps by default.
constexpr int kFusedMaxRows = 64;

bool pdl_enabled() {
  const char* e = std::getenv("CAI_PDL");
  return !(e && e[0] == '0');
}

// NVTX ranges around every step call (CAI_NVTX=1), for profilers that show
// them (ncu --nvtx); without a profiler attached the calls do nothing.
bool nvtx_enabled() {
  const char* e = std::getenv("CAI_NVTX");
  return e && e[0] == '1';
}

bool pair_enabled() {
  const char* e = std::getenv("CAI_PAIR");
  return !(e && e[0] == '0');
}

// Widest tile the pair kernel runs in the swapped orientation (masked rows in
// the MMA N dimension, 32-row granularity): CAI_PAIR_SWAP_MAX_N (32..256), or
// 0 with CAI_PAIR_SWAP=0; default 192.
int pair_swap_max_n() {
  const char* e = std::getenv("CAI_PAIR_SWAP");
  if (e && e[0] == '0') return 0;
  const char* n = std::getenv("CAI_PAIR_SWAP_MAX_N");
  const int v = n ? std::atoi(n) : 0;
  return v >= 32 && v <= 256 ? v : 192;
}

// Optional caps on the LM head's W ring depth (CAI_HEAD_STAGES) and tile
// group size (CAI_HEAD_GMAX), read once per context at cai_init; 0 or unset
// keeps the defaults.  Tuning knobs only: results do not depend on them.
int env_int(const char* name) {
  const char* e = std::getenv(name);
  return e ? std::atoi(e) : 0;
}

int dev_alloc(void** p, size_t bytes) {
  *p = nullptr;
  int n = g_fail_alloc_after.load();
  if (n > 0) {
    if (n == 1) {
      g_fail_alloc_after.store(0);
      return CAI_ERR_NOMEM;
    }
    g_fail_alloc_after.store(n - 1);
  }
  if (bytes == 0) bytes = 16;
  cudaError_t e = cudaMalloc(p, bytes);
  if (e == cudaErrorMemoryAllocation) {
    cudaGetLastError();
    return CAI_ERR_NOMEM;
  }
  if (e != cudaSuccess) return CAI_ERR_CUDA;
  return CAI_OK;
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// A driver API entry point, or null if the driver does not provide it.
void* driver_entry(const char* name) {
  void* ptr = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion(name, &ptr, 12000, cudaEnableDefault, &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return ptr;
}

// Each entry point is resolved once; a function-local static is initialised
// once even when contexts are created on several host threads at a time.
// cuStreamWriteValue64, for the staged-rows sequence words:
typedef CUresult (*WriteValue64Fn)(CUstream, CUdeviceptr, cuuint64_t, unsigned int);
WriteValue64Fn get_write_value64() {
  static const WriteValue64Fn fn =
      reinterpret_cast<WriteValue64Fn>(driver_entry("cuStreamWriteValue64"));
  return fn;
}

EncodeTiledFn get_encoder() {
  static const EncodeTiledFn fn =
      reinterpret_cast<EncodeTiledFn>(driver_entry("cuTensorMapEncodeTiled"));
  return fn;
}

// Row-major bf16 matrix [rows, cols] with a box of box_rows x 64 columns and
// the 128-byte swizzle that the MMA descriptors expect.
bool make_map(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows,
              CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B) {
  EncodeTiledFn enc = get_encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBlockK), box_rows};
  cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int round_up(int x, int m) { return (x + m - 1) / m * m; }

// Swapped pair tiles: one map of the gathered rows per box height 16..128.
template <typename Ctx>
bool make_row_maps(Ctx* c, int H) {
  for (int q = 0; q < 8; ++q)
    if (!make_map(&c->tm_rows.box[q], c->hc, c->rows_cap, H, 16 * (q + 1))) return false;
  return true;
}
int next_pow2(int x) {
  int p = 1;
  while (p < x) p <<= 1;
  return p;
}

// Launch with programmatic stream serialization: the kernel may be scheduled
// while the previous kernel in the stream is still running; every kernel of
// this library waits for its predecessor (griddepcontrol.wait) before it
// reads or writes anything that predecessor produces or consumes.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(bool pdl, void (*kernel)(KArgs...), int grid, int block, size_t smem,
                       cudaStream_t stream, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(static_cast<unsigned>(block));
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

bool is_device_ptr(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

// Device address of page-locked, device-mapped host memory, or null.
const void* host_mapped_ptr(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return a.type == cudaMemoryTypeHost ? a.devicePointer : nullptr;
}

}  // namespace

struct cai_ctx {
  cai_config cfg{};
  int L = 0, BP = 0, rows_cap = 0;
  StateArrays st{};
  int* list = nullptr;
  int* row_of = nullptr;
  int* d_M = nullptr;
  unsigned* ticket = nullptr;
  unsigned long long* pub = nullptr;  // last published step (CommitParams::pub)
  uint32_t* err = nullptr;
  __nv_bfloat16* hc = nullptr;
  float4* part = nullptr;
  float4* rowres = nullptr;  // [rows_cap] merged triple per row (pair steps)
  void* hidden_stage = nullptr;
  HostFlag* hf_host = nullptr;
  HostFlag* hf_dev = nullptr;
  void* wpk = nullptr;   // packed copy of W (pack_weight_kernel layout), if head_in_step
  void* wt = nullptr;    // tile-major packed copy of W (pack_w_tiles_kernel), pair kernel
  CUtensorMap tm_a{};    // compact gathered rows in 128-row boxes (pair kernel)
  PairRowMaps tm_rows{};  // ... in 16-, 32-, ..., 128-row boxes (swapped pair kernel)
  CUtensorMap tm_w{};    // wt as [2 n_vt (H / 64) 128, 64], 16 KiB unswizzled boxes
  bool use_pair = false; // steps with >= pair_min_M rows run lm_head_pair_kernel
  int swap_max_n = 0;       // ... swapped when its tile width is at most this (pair_swapped)
  bool head_in_step = true; // the swapped-operand kernel is launched in multi-kernel steps
  bool need_reduce = false; // some step size leaves per-tile partials to reduce_partials_kernel
  bool norm = false;     // the model's final RMSNorm is part of the head (cai_init_rmsnorm)
  float norm_eps = 0.0f;
  float* inv_r = nullptr;  // [rows_cap] 1 / sqrt(mean h^2 + eps) of this step's rows
  __nv_bfloat16* h_prev = nullptr;  // [B P, H] previous step's rows (CAI_DIAGNOSTICS)
  void (*head_kernel)(CUtensorMap, HeadParams) = nullptr;
  void (*pair_kernel)(CUtensorMap, CUtensorMap, PairRowMaps, PairParams) = nullptr;
  int pair_min_M = 0, pair_grid = 0, pair_stages = 0, n_vt = 0, reduce_grid = 0;
  // Most pair stages in flight: swapped stages cut to size would give up to
  // 10 for narrow tiles, but beyond 8 the narrowest steps slow down again
  // (measured at fixed M, long-Dream shape: M = 30 160.8 us at 8, 165 at 10).
  // CAI_PAIR_RING_MAX overrides (2..12; tuning knob).
  int pair_ring_max = 8;
  size_t pair_smem = 0;
  CUtensorMap tm_h{};    // compact gathered rows (multi-kernel step)
  CUtensorMap tm_hid{};  // the caller's rows (single-kernel step), for hid_mapped
  const void* hid_mapped = nullptr;
  // Steps on host rows: the rows are copied on copy_stream into stage2[step
  // id & 1] (hidden_stage and a second buffer), and the step's stream waits
  // only for that copy, so the copy of step t + 1 overlaps step t and no copy
  // sits between two step kernels in the step's stream.  A buffer is refilled
  // after the kernel that read it (ev_read: the single-kernel step's LM head,
  // the multi-kernel step's gather) has finished.
  void* stage2[2] = {nullptr, nullptr};
  CUtensorMap tm_stage[2]{};
  cudaStream_t copy_stream = nullptr;
  cudaEvent_t ev_copied[2] = {nullptr, nullptr};
  cudaEvent_t ev_read[2] = {nullptr, nullptr};
  bool read_pending[2] = {false, false};
  // After its copy the side stream writes the step's id + 1 into
  // stage_seq_dev[k]; the step's first kernel that reads the rows (the
  // single-kernel LM head, or the gather) waits for that word before reading
  // them, so the step's stream waits for nothing and consecutive steps keep
  // their programmatic overlap.  Used when nothing else of the step reads the
  // rows (not with the diagnostics' drift kernel, nor with the final norm in
  // single-kernel steps, whose row scales are computed from the rows outside
  // the TMA pipeline) and the driver provides stream memory writes;
  // otherwise the step's stream waits for ev_copied.
  unsigned long long* stage_seq_dev = nullptr;
  bool stage_by_word = false;
  bool fused = false;    // single-kernel step (B P <= 64)
  bool rows_head = false;  // the single-kernel step runs lm_head_rows_kernel
  // Vocabulary shard (cai_init_vocab_shard): the context's LM head covers the
  // rows [v_off, v_off + cfg.V) of a vocabulary of V_total rows; a step is
  // cai_shard_head, an exchange of every shard's triples, cai_shard_commit.
  bool shard = false;
  int v_off = 0, V_total = 0;
  bool shard_pending = false;  // a shard head ran; its commit has not
  bool shard_first = false;    // ... and it was the block's step zero
  int G = 0, n_stages = 0, n_bslots = 0, n_max = 0, slot_cols = 0, gmax = 1, tmem_cols = 0;
  int b_slot_bytes = 0;
  size_t head_smem = 0;
  int blk = 0, t_next = 0;
  int64_t last_step_id = -1;
  bool block_done_seen = false;
  int sticky = CAI_OK;
  cai_stats stats{};
  bool profiling = false;
  bool pdl = true;
  bool nvtx = false;
  std::vector<cudaEvent_t> ev_pool;  // per profiled step: step start, head start, head end, step end
  size_t ev_used = 0;                // events recorded since the last stats call
  std::vector<void*> allocs;
  std::vector<size_t> alloc_bytes;   // usable bytes of each allocation (guard bytes follow)
};

namespace {

int fail(cai_ctx* c, int code) {
  if (c && (code == CAI_ERR_CUDA || code == CAI_ERR_DEVICE) && c->sticky == CAI_OK) c->sticky = code;
  return code;
}

int check_launch(cai_ctx* c) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    fprintf(stderr, "cai: CUDA error %s\n", cudaGetErrorString(e));
    return fail(c, CAI_ERR_CUDA);
  }
  return CAI_OK;
}

int validate(const cai_config* c) {
  if (c->B < 1 || c->P < 1 || c->P > kMaxP || c->H < 64 || c->H > 16384 || (c->H % 64) != 0 ||
      c->V < 64 || c->T < 1 || c->T > 32767 || c->n_blocks < 1 ||
      static_cast<int64_t>(c->B) * c->P > 65536 ||
      c->n_blocks > 32767 || static_cast<int64_t>(c->n_blocks) * c->P > (1 << 24))
    return CAI_ERR_SHAPE;
  if (c->warmup_pct < 0 || c->warmup_pct > 100 || c->K < 1 || (c->eta_mode != 0 && c->eta_mode != 1) ||
      !(c->clip_lo <= c->clip_hi) || (c->flags & ~255u) != 0)
    return CAI_ERR_ARG;
  return CAI_OK;
}

// Every context buffer is followed by kGuardBytes of a fixed pattern; a write
// past the end of a buffer shows up in cai_test_check_guards.
constexpr size_t kGuardBytes = 256;
constexpr unsigned char kGuardByte = 0xC3;

int alloc_into(cai_ctx* c, void** dst, size_t bytes) {
  const size_t padded = (bytes + 255) / 256 * 256;
  int r = dev_alloc(dst, padded + kGuardBytes);
  if (r != CAI_OK) return r;
  c->allocs.push_back(*dst);
  c->alloc_bytes.push_back(padded);
  if (cudaMemset(static_cast<char*>(*dst) + padded, kGuardByte, kGuardBytes) != cudaSuccess)
    return CAI_ERR_CUDA;
  return CAI_OK;
}

void release(cai_ctx* c) {
  for (void* p : c->allocs) cudaFree(p);
  c->allocs.clear();
  c->alloc_bytes.clear();
  if (c->hf_host) cudaFreeHost(c->hf_host);
  c->hf_host = nullptr;
  for (cudaEvent_t e : c->ev_pool) cudaEventDestroy(e);
  c->ev_pool.clear();
  for (int k = 0; k < 2; ++k) {
    if (c->ev_copied[k]) cudaEventDestroy(c->ev_copied[k]);
    if (c->ev_read[k]) cudaEventDestroy(c->ev_read[k]);
    c->ev_copied[k] = c->ev_read[k] = nullptr;
  }
  if (c->copy_stream) cudaStreamDestroy(c->copy_stream);
  c->copy_stream = nullptr;
}

// ---- threshold schedule (Boxes 3, 4, 6), double precision on the host ----

double theta_e_of(const cai_config& c, int b1) {
  int be = b1;
  if (c.flags & CAI_QUARTER_BLOCKS) be = 1 + (4 * (b1 - 1)) / c.n_blocks;
  if (c.flags & CAI_NO_BLOCK_SCHEDULE) be = 1;
  double th = c.theta_e1 - c.theta_e_step * static_cast<double>(be - 1);
  return th < c.theta_e_min ? c.theta_e_min : th;
}

double theta_block_of(const cai_config& c, int b1, int t) {
  if (c.flags & CAI_FIXED_THRESHOLD) return c.theta_s;
  if (100 * t < c.warmup_pct * c.T) return c.theta_s;
  const double wT = static_cast<double>(c.warmup_pct) * c.T / 100.0;
  const double u = (t - wT) / (c.T - wT);
  const double te = theta_e_of(c, b1);
  return te + 0.5 * (c.theta_s - te) * (1.0 + std::cos(M_PI * u));
}

double pos_factor_of(const cai_config& c, int p) {
  if (!(c.flags & CAI_POS_FACTOR)) return 1.0;
  int q1 = 16, q2 = 32, q3 = 48;
  if (c.flags & CAI_QUARTER_POS) {
    q1 = c.P / 4;
    q2 = c.P / 2;
    q3 = 3 * c.P / 4;
  }
  return p < q1 ? 0.80 : p < q2 ? 0.90 : p < q3 ? 1.05 : 1.10;
}

// theta_i(t) of position p in block b1 (1-based), Eq. position_threshold:
// the block's threshold times the position factor, clipped, in double, then
// rounded once to the fp32 value the commit rule compares against.
float theta_token_of(const cai_config& c, int b1, int t, int p) {
  double th = theta_block_of(c, b1, t) * pos_factor_of(c, p);
  th = th < c.clip_lo ? c.clip_lo : th;
  th = th > c.clip_hi ? c.clip_hi : th;
  return static_cast<float>(th);
}

CommitParams commit_params(cai_ctx* c, int t, int64_t step_id) {
  const cai_config& cfg = c->cfg;
  CommitParams cp{};
  cp.part = c->part;
  cp.n_part = c->G;
  cp.rowres = c->rowres;
  cp.pair_pairs = c->pair_grid / 2;
  cp.pair_swap_max_n = c->swap_max_n;
  cp.pair_min_M = c->use_pair ? c->pair_min_M : INT_MAX;
  cp.identity_rows = c->fused ? 1 : 0;
  // The pair kernel, the last LM-head kernel of a multi-kernel step, starts
  // its dependents only after its own wait for the gather, hence for the
  // previous step's commit.
  cp.prefetch_state = !c->fused && c->use_pair ? 1 : 0;
  cp.st = c->st;
  cp.list = c->list;
  cp.row_of = c->row_of;
  cp.d_M = c->d_M;
  cp.m_hist_slot = c->st.m_hist + c->blk * cfg.T + t;
  cp.ticket = c->ticket;
  cp.pub = c->pub;
  cp.hf = c->hf_dev;
  cp.err = c->err;
  cp.B = cfg.B;
  cp.P = cfg.P;
  cp.L = c->L;
  cp.n_blocks = cfg.n_blocks;
  cp.T = cfg.T;
  cp.blk = c->blk;
  cp.t = t;
  cp.step_id = static_cast<int>(step_id);
  cp.K = cfg.K;
  cp.eta_mode = cfg.eta_mode;
  cp.eta_bar = static_cast<float>(cfg.eta_bar);
  cp.theta_fb = static_cast<float>(cfg.theta_fb);
  cp.budget_half = (cfg.flags & CAI_QUARTER_POS) ? cfg.P / 2 : 32;
  cp.budget_late = (cfg.flags & CAI_QUARTER_POS) ? 3 * cfg.P / 4 : 48;
  cp.flags = cfg.flags;
  for (int p = 0; p < cfg.P; ++p) cp.theta_tab[p] = theta_token_of(cfg, c->blk + 1, t, p);
  return cp;
}

// Multi-kernel step, kernel 1: the gather of this step's masked rows into
// the compact operand (all rows at step zero).
int launch_gather(cai_ctx* c, const void* hid, bool first, cudaStream_t stream,
                  const unsigned long long* stage_word = nullptr,
                  unsigned long long stage_seq = 0) {
  GatherParams gp{};
  gp.stage_word = stage_word;
  gp.stage_seq = stage_seq;
  gp.hidden = static_cast<const __nv_bfloat16*>(hid);
  gp.hc = c->hc;
  gp.list = c->list;
  gp.row_of = c->row_of;
  gp.d_M = c->d_M;
  gp.B = c->cfg.B;
  gp.BP = c->BP;
  gp.H = c->cfg.H;
  gp.first = first ? 1 : 0;
  gp.inv_r = c->norm ? c->inv_r : nullptr;
  gp.err = c->err;
  gp.eps = c->norm_eps;
  const int g_grid = c->rows_cap / kGatherRowsPerCta;
  if (launch_pdl(c->pdl, gather_rows_kernel, g_grid, kGatherThreads, 0, stream, gp) !=
      cudaSuccess)
    return check_launch(c);
  c->stats.launches++;
  return CAI_OK;
}

// Multi-kernel step: the CTA-pair LM head at local step t, and the row merge
// of its per-tile partials in contexts where some step size leaves them.
int launch_pair_head(cai_ctx* c, int t, cudaStream_t stream) {
  const cai_config& cfg = c->cfg;
  PairParams pp{};
  pp.d_M = c->d_M;
  pp.m_hist_slot = c->st.m_hist + c->blk * cfg.T + t;
  pp.part = c->part;
  pp.err = c->err;
  pp.V = cfg.V;
  pp.H = cfg.H;
  pp.n_vt = c->n_vt;
  pp.min_M = c->pair_min_M;
  pp.swap_max_n = c->swap_max_n;
  pp.n_stages = c->pair_stages;
  pp.inv_r = c->inv_r;
  pp.ring_max = c->pair_ring_max;
  if (launch_pdl(c->pdl, c->pair_kernel, c->pair_grid, kPairThreads, c->pair_smem, stream,
                 c->tm_a, c->tm_w, c->tm_rows, pp) != cudaSuccess)
    return check_launch(c);
  c->stats.launches++;
  if (c->need_reduce) {
    ReduceParams rp{};
    rp.part = c->part;
    rp.rowres = c->rowres;
    rp.d_M = c->d_M;
    rp.n_vt = c->n_vt;
    rp.min_M = c->pair_min_M;
    rp.n_pairs = c->pair_grid / 2;
    rp.swap_max_n = c->swap_max_n;
    if (launch_pdl(c->pdl, reduce_partials_kernel, c->reduce_grid, kReduceThreads, 0, stream,
                   rp) != cudaSuccess)
      return check_launch(c);
    c->stats.launches++;
  }
  return CAI_OK;
}

// The rows a multi-kernel step reads: device rows as they are, page-locked
// host rows in place over the host link (the gather reads only the masked
// ones), other host rows copied to the device on the stream first.
int multi_kernel_rows(cai_ctx* c, const void* hidden, cudaStream_t stream, const void** hid) {
  *hid = hidden;
  if (is_device_ptr(hidden)) return CAI_OK;
  if (const void* mapped = host_mapped_ptr(hidden)) {
    *hid = mapped;
    return CAI_OK;
  }
  const size_t bytes = static_cast<size_t>(c->BP) * c->cfg.H * 2;
  if (cudaMemcpyAsync(c->hidden_stage, hidden, bytes, cudaMemcpyHostToDevice, stream) !=
      cudaSuccess)
    return fail(c, CAI_ERR_CUDA);
  *hid = c->hidden_stage;
  return CAI_OK;
}

// One denoising step.  Single-kernel step (B P <= 64): the LM-head kernel
// reads the hidden states in place and its last CTA commits.  Otherwise:
// gather -> LM head -> merge + commit.
int step_impl(cai_ctx* c, const void* hidden, void* stream_v, bool first);

int step(cai_ctx* c, const void* hidden, void* stream_v, bool first) {
  if (!c->nvtx) return step_impl(c, hidden, stream_v, first);
  char name[48];
  std::snprintf(name, sizeof name, "cai step b%d t%d", c->blk, c->t_next);
  nvtxRangePushA(name);
  const int r = step_impl(c, hidden, stream_v, first);
  nvtxRangePop();
  return r;
}

int step_impl(cai_ctx* c, const void* hidden, void* stream_v, bool first) {
  cudaStream_t stream = static_cast<cudaStream_t>(stream_v);
  const cai_config& cfg = c->cfg;
  const void* hid = hidden;
  const int64_t step_id = c->last_step_id + 1;
  int stage_slot = -1;  // step on host rows: stage2 buffer used
  if (!is_device_ptr(hidden)) {
    // Host rows are copied to the device on the side stream (see stage2),
    // overlapping the previous step; the step's first reader waits for them.
    const size_t bytes = static_cast<size_t>(c->BP) * cfg.H * 2;
    {
      const int k = static_cast<int>(step_id & 1);
      if ((c->read_pending[k] &&
           cudaStreamWaitEvent(c->copy_stream, c->ev_read[k], 0) != cudaSuccess) ||
          cudaMemcpyAsync(c->stage2[k], hidden, bytes, cudaMemcpyHostToDevice, c->copy_stream) !=
              cudaSuccess)
        return fail(c, CAI_ERR_CUDA);
      if (c->stage_by_word) {
        // Default flags: the write follows the copy and makes its bytes visible.
        if (get_write_value64()(reinterpret_cast<CUstream>(c->copy_stream),
                                reinterpret_cast<CUdeviceptr>(c->stage_seq_dev + k),
                                static_cast<cuuint64_t>(step_id + 1), 0) != CUDA_SUCCESS)
          return fail(c, CAI_ERR_CUDA);
      } else if (cudaEventRecord(c->ev_copied[k], c->copy_stream) != cudaSuccess ||
                 cudaStreamWaitEvent(stream, c->ev_copied[k], 0) != cudaSuccess) {
        return fail(c, CAI_ERR_CUDA);
      }
      hid = c->stage2[k];
      stage_slot = k;
    }
  }
  const int t = c->t_next;
  cudaEvent_t ev[4] = {nullptr, nullptr, nullptr, nullptr};
  const bool diag = (cfg.flags & CAI_DIAGNOSTICS) != 0;
  if (c->profiling) {
    while (c->ev_used + 4 > c->ev_pool.size()) {
      cudaEvent_t e;
      if (cudaEventCreate(&e) != cudaSuccess) return fail(c, CAI_ERR_CUDA);
      c->ev_pool.push_back(e);
    }
    for (int k = 0; k < 4; ++k) ev[k] = c->ev_pool[c->ev_used + k];
    c->ev_used += 4;
    cudaEventRecord(ev[0], stream);
  }
  if (diag) {
    DriftParams dp{};
    dp.hidden = static_cast<const __nv_bfloat16*>(hid);
    dp.prev = c->h_prev;
    dp.drift = c->st.drift;
    dp.P = cfg.P;
    dp.H = cfg.H;
    dp.n_blocks = cfg.n_blocks;
    dp.T = cfg.T;
    dp.blk = c->blk;
    dp.t = t;
    if (launch_pdl(c->pdl, drift_kernel, cfg.B, kGatherThreads, 0, stream, dp) != cudaSuccess)
      return check_launch(c);
    c->stats.launches++;
  }

  if (!c->fused) {
    const unsigned long long* word =
        stage_slot >= 0 && c->stage_by_word ? c->stage_seq_dev + stage_slot : nullptr;
    const int r =
        launch_gather(c, hid, first, stream, word, static_cast<unsigned long long>(step_id + 1));
    if (r != CAI_OK) return r;
    if (stage_slot >= 0) {
      // stage2[stage_slot] may be refilled once the gather is done.
      if (cudaEventRecord(c->ev_read[stage_slot], stream) != cudaSuccess)
        return fail(c, CAI_ERR_CUDA);
      c->read_pending[stage_slot] = true;
    }
  } else {
    if (stage_slot < 0 && hid != c->hid_mapped) {
      // The single-kernel step reads the caller's [B P, H] rows through TMA.
      if (!make_map(&c->tm_hid, hid, c->BP, cfg.H, kBoxRowsB)) return CAI_ERR_ARG;
      c->hid_mapped = hid;
    }
    // With the final norm the LM-head kernel computes the row scales from
    // the rows itself.
  }

  HeadParams hp{};
  hp.wpk = static_cast<const uint8_t*>(c->wpk);
  hp.d_M = c->d_M;
  hp.m_hist_slot = c->st.m_hist + c->blk * cfg.T + t;
  hp.fused = c->fused ? 1 : 0;
  hp.M_fixed = c->BP;
  hp.max_M = c->use_pair ? c->pair_min_M - 1 : INT_MAX;
  if (c->fused && stage_slot >= 0 && c->stage_by_word) {
    hp.stage_word = c->stage_seq_dev + stage_slot;
    hp.stage_seq = static_cast<unsigned long long>(step_id + 1);
  }
  hp.prefetch = c->use_pair ? 0 : 1;
  hp.first = first ? 1 : 0;
  hp.part = c->part;
  hp.err = c->err;
  hp.V = cfg.V;
  hp.H = cfg.H;
  hp.units = (cfg.V + kUnitRows - 1) / kUnitRows;
  hp.n_stages = c->n_stages;
  hp.n_bslots = c->n_bslots;
  hp.b_slot_bytes = c->b_slot_bytes;
  hp.slot_cols = c->slot_cols;
  hp.gmax = c->gmax;
  hp.tmem_cols = c->tmem_cols;
  hp.inv_r = c->inv_r;
  hp.hid = static_cast<const __nv_bfloat16*>(hid);
  hp.norm_eps = c->norm_eps;
  const CommitParams cp = commit_params(c, t, step_id);
  if (c->fused) hp.cp = cp;
  if (c->profiling) cudaEventRecord(ev[1], stream);
  if (c->head_in_step) {
    const CUtensorMap& tm_rows =
        !c->fused ? c->tm_h : stage_slot >= 0 ? c->tm_stage[stage_slot] : c->tm_hid;
    if (launch_pdl(c->pdl, c->head_kernel, c->G, kHeadThreads, c->head_smem, stream, tm_rows,
                   hp) != cudaSuccess)
      return check_launch(c);
    c->stats.launches++;
    if (c->fused && stage_slot >= 0) {
      // stage2[stage_slot] may be refilled once this step's kernel is done.
      if (cudaEventRecord(c->ev_read[stage_slot], stream) != cudaSuccess)
        return fail(c, CAI_ERR_CUDA);
      c->read_pending[stage_slot] = true;
    }
  }
  if (c->use_pair) {
    // Only one of the two LM-head kernels decodes a step: the other reads
    // this step's M and returns at once (with pair_min_M = 1 the pair kernel
    // decodes every step and the other one is not launched).
    const int r = launch_pair_head(c, t, stream);
    if (r != CAI_OK) return r;
  }
  if (c->profiling) cudaEventRecord(ev[2], stream);
  c->stats.head_launches++;

  if (!c->fused) {
    const int commit_threads = cfg.P < kCommitThreads / 32 ? 32 * cfg.P : kCommitThreads;
    if (launch_pdl(c->pdl, merge_commit_kernel, cfg.B, commit_threads, 0, stream, cp) !=
        cudaSuccess)
      return check_launch(c);
    c->stats.launches++;
  }
  if (c->profiling) cudaEventRecord(ev[3], stream);
  c->stats.steps++;
  int r = check_launch(c);
  if (r != CAI_OK) return r;
  c->last_step_id = step_id;
  c->t_next = t + 1;
  return CAI_OK;
}

}  // namespace

extern "C" {

int cai_config_default(cai_config* cfg, int32_t preset, int32_t B, int32_t P, int32_t H, int32_t V,
                       int32_t T, int32_t n_blocks) {
  if (!cfg || (preset != CAI_PRESET_LLADA && preset != CAI_PRESET_DREAM)) return CAI_ERR_ARG;
  cai_config c{};
  c.B = B;
  c.P = P;
  c.H = H;
  c.V = V;
  c.T = T;
  c.n_blocks = n_blocks;
  c.theta_s = 0.90;
  c.theta_e1 = 0.70;
  c.theta_e_step = 0.10;
  c.theta_e_min = 0.40;
  c.warmup_pct = 15;
  c.K = 4;
  c.theta_fb = 0.40;
  c.clip_lo = 0.20;
  c.clip_hi = 0.98;
  c.eta_bar = 1.5;
  c.eta_mode = 0;
  c.flags = CAI_POS_FACTOR | (preset == CAI_PRESET_LLADA ? CAI_GATING : 0u);
  *cfg = c;
  return CAI_OK;
}

namespace {

// cai_init, cai_init_rmsnorm and cai_init_vocab_shard; g (bf16 [H], host or
// device) is null except for cai_init_rmsnorm; V_shard > 0 makes a shard
// context whose W holds the vocabulary rows [v0, v0 + V_shard).
int init_impl(const cai_config* cfg_in, const void* W, const void* g, double eps, int v0,
              int V_shard, void* stream, cai_ctx** out) {
  if (!cfg_in || !W || !out) return CAI_ERR_ARG;
  *out = nullptr;
  int r = validate(cfg_in);
  if (r != CAI_OK) return r;
  if (reinterpret_cast<uintptr_t>(W) % 16 != 0) return CAI_ERR_ARG;
  const bool shard = V_shard > 0;
  if (shard && (v0 < 0 || V_shard < 64 ||
                static_cast<int64_t>(v0) + V_shard > static_cast<int64_t>(cfg_in->V)))
    return CAI_ERR_SHAPE;
  // A shard context runs its LM head over its own V_shard rows.
  cai_config local_cfg = *cfg_in;
  if (shard) local_cfg.V = V_shard;
  const cai_config* cfg = &local_cfg;

  int dev = 0, major = 0, minor = 0, sms = 0, smem_optin = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
          cudaSuccess) {
    cudaGetLastError();
    return CAI_ERR_CUDA;
  }
  if (major != 10 || minor != 3) return CAI_ERR_UNSUPPORTED;

  cai_ctx* c = new (std::nothrow) cai_ctx();
  if (!c) return CAI_ERR_NOMEM;
  c->cfg = *cfg;
  c->L = cfg->n_blocks * cfg->P;
  c->BP = cfg->B * cfg->P;
  c->rows_cap = round_up(c->BP, 16);
  c->pdl = pdl_enabled();
  c->nvtx = nvtx_enabled();
  // Single-kernel steps decode every row of the block each step (the
  // rows-operand LM head pads the rows to 128 anyway) and save the gather and
  // commit launches; larger batches run multi-kernel steps, whose pair kernel
  // decodes only the masked rows.  Measured, LLaDA shape, positions/s,
  // single- against multi-kernel: B P = 64 197.8k against 169.5k, B P = 128
  // 329.3k against 331.5k.  CAI_FUSED_MAX_BP overrides the limit (up to 256;
  // above 128 rows the swapped-operand kernel runs).
  const int fmax = env_int("CAI_FUSED_MAX_BP");
  c->fused = !shard && c->BP <= (fmax > 0 && fmax <= kChunkN ? fmax : kFusedMaxRows);
  c->norm = g != nullptr;
  c->norm_eps = static_cast<float>(eps);
  c->head_kernel = c->norm ? lm_head_softmax_kernel<true> : lm_head_softmax_kernel<false>;
  // Shard contexts always run multi-kernel steps on the pair kernel with
  // swapped narrow steps, so that the pair kernel decodes every step.
  c->shard = shard;
  c->v_off = shard ? v0 : 0;
  c->V_total = cfg_in->V;
  c->use_pair = shard || (!c->fused && pair_enabled());
  c->swap_max_n = c->use_pair ? pair_swap_max_n() : 0;
  if (shard && c->swap_max_n < kSwapColStep) c->swap_max_n = 192;
  c->pair_kernel = c->norm ? lm_head_pair_kernel<true> : lm_head_pair_kernel<false>;

  // LM-head launch shape.  N chunk (positions per MMA), grid (one CTA per SM,
  // at least kMinCtaRows vocabulary rows per CTA), tile group size (tiles sharing one hidden
  // stage; two group buffers of gmax * slot_cols tensor-memory columns fit in
  // 512), ring depths within the opt-in shared memory.
  // Pair kernel (multi-kernel steps only): steps with at least pair_min_M
  // masked rows run on CTA pairs (CAI_PAIR=0 disables it, CAI_PAIR_MIN_M sets
  // the threshold); the swapped-operand kernel then needs N < pair_min_M only,
  // which keeps its tile groups large.  When narrow steps run swapped the pair
  // kernel decodes every step (pair_min_M = 1: a 32-column tile is as cheap as
  // the W stream it rides on), and the swapped-operand kernel is not launched.
  if (c->use_pair) {
    const int mset = env_int("CAI_PAIR_MIN_M");
    c->pair_min_M = mset > 0 ? mset : (c->swap_max_n >= kSwapColStep ? 1 : 32);
  }
  c->head_in_step = !c->use_pair || c->pair_min_M > 1;
  c->n_max = c->rows_cap < kChunkN ? c->rows_cap : kChunkN;
  if (c->use_pair) {
    const int cap = round_up(c->pair_min_M > 1 ? c->pair_min_M - 1 : 1, 16);
    if (c->n_max > cap) c->n_max = cap;
  }
  c->slot_cols = round_up(c->n_max, 32);
  const int units = (cfg->V + kUnitRows - 1) / kUnitRows;
  // Single-kernel step: one SM is left to the CTA that commits the step, so
  // the next step's CTAs all find a free SM instead of one of them waiting
  // for the commit to finish (and becoming the next step's straggler).
  const int usable_sms = c->fused && sms > 1 ? sms - 1 : sms;
  // V is split in units of one swizzle atom (kUnitRows rows), so any grid
  // size balances the rows to within kUnitRows per CTA.
  const int min_units = kMinCtaRows / kUnitRows;
  const int g_rows = (units + min_units - 1) / min_units;
  c->G = g_rows < usable_sms ? g_rows : usable_sms;
  const int glim = g_head_grid_limit.load();
  if (glim > 0 && c->G > glim) c->G = glim;
  const int max_units = (units + c->G - 1) / c->G;
  const int max_tiles = (max_units * kUnitRows + kRowsPerTile - 1) / kRowsPerTile;
  // Default: as many tiles per group as two group buffers of tensor memory
  // allow (all of a CTA's tiles for N <= 32).  Every tile of a group is an
  // independent accumulation chain, and at small N a single chain is bound by
  // MMA latency rather than HBM; interleaving the chains of the group hides
  // it.  CAI_HEAD_GMAX overrides (bounded by the tensor memory).
  c->gmax = max_tiles;
  const int gset = env_int("CAI_HEAD_GMAX");
  if (gset > 0) c->gmax = gset;
  if (c->gmax > 256 / c->slot_cols) c->gmax = 256 / c->slot_cols;
  if (c->gmax < 1) c->gmax = 1;
  c->tmem_cols = next_pow2(2 * c->gmax * c->slot_cols < 32 ? 32 : 2 * c->gmax * c->slot_cols);
  c->b_slot_bytes = c->n_max * 128;
  // CAI_HEAD_BSLOTS_TIGHT=1: size the hidden ring for full groups only (a
  // shorter last group then throttles the producer a little; tuning knob).
  const bool tight = env_int("CAI_HEAD_BSLOTS_TIGHT") == 1;
  auto bslots_for = [&](int stages) {
    // One hidden stage serves a group of tiles; keep enough of them in flight
    // to cover the W ring (groups may be one tile smaller than gmax).
    const int per = c->gmax > 1 ? (tight ? c->gmax : c->gmax - 1) : 1;
    return c->gmax == 1 ? stages : (stages + per - 1) / per + 1;
  };
  // Dynamic shared memory may use what the kernel's static shared memory leaves.
  cudaFuncAttributes head_attr{};
  if (cudaFuncGetAttributes(&head_attr, c->head_kernel) != cudaSuccess) {
    cudaGetLastError();
    delete c;
    return CAI_ERR_CUDA;
  }
  const size_t dyn_limit = static_cast<size_t>(smem_optin) - head_attr.sharedSizeBytes;
  const int scap = env_int("CAI_HEAD_STAGES");
  int stages = scap >= 2 && scap <= 16 ? scap : 12;
  while (stages > 2 && head_smem_bytes(stages, bslots_for(stages), c->b_slot_bytes,
                                       c->slot_cols) > dyn_limit)
    --stages;
  c->n_stages = stages;
  c->n_bslots = bslots_for(stages);
  c->head_smem = head_smem_bytes(stages, c->n_bslots, c->b_slot_bytes, c->slot_cols);
  // Single-kernel steps of up to 128 rows run lm_head_rows_kernel, the rows
  // as the MMA's A operand and up to 256 vocabulary rows as N, which consumes
  // W twice as fast per MMA as the swapped kernel (CAI_ROWS_HEAD=0: the
  // swapped kernel instead).  W is packed by pack_weight_rows_kernel.
  const char* rh_env = std::getenv("CAI_ROWS_HEAD");
  if (c->fused && c->BP <= kRowsM && !(rh_env && rh_env[0] == '0')) {
    c->rows_head = true;
    c->head_kernel = c->norm ? lm_head_rows_kernel<true> : lm_head_rows_kernel<false>;
    cudaFuncAttributes ra{};
    if (cudaFuncGetAttributes(&ra, c->head_kernel) != cudaSuccess) {
      cudaGetLastError();
      delete c;
      return CAI_ERR_CUDA;
    }
    const size_t rlimit = static_cast<size_t>(smem_optin) - ra.sharedSizeBytes;
    // As many W stages as fit next to a rows ring of the same depth (the
    // rows stages are small); CAI_ROWS_STAGES caps the W ring (tuning knob).
    // Four 32 KiB W stages in flight per SM: deeper rings stream faster on
    // most SMs but starve some (measured, LLaDA shape: finish spread 4 us at
    // 4 stages, 20 us at 6), and a step waits for its slowest CTA.
    const int hs = rows_h_stride(c->BP);
    const int scap2 = env_int("CAI_ROWS_STAGES");
    int st = scap2 >= 2 && scap2 <= 8 ? scap2 : 4;
    while (st > 2 && rows_smem_bytes(st, 2 * st, hs) > rlimit) --st;
    int bs = 2 * st;
    while (bs > 2 && rows_smem_bytes(st, bs, hs) > rlimit) --bs;
    c->n_stages = st;
    c->n_bslots = bs;
    c->tmem_cols = kRowsTmemCols;
    c->head_smem = rows_smem_bytes(st, bs, hs);
  }

  // Pair kernel launch shape: a persistent grid of as many 2-CTA clusters as
  // can be resident at once.
  if (c->use_pair) {
    c->n_vt = (cfg->V + kPairTileVocab - 1) / kPairTileVocab;
    cudaFuncAttributes pa{};
    if (cudaFuncGetAttributes(&pa, c->pair_kernel) != cudaSuccess) {
      cudaGetLastError();
      delete c;
      return CAI_ERR_CUDA;
    }
    const size_t plimit = static_cast<size_t>(smem_optin) - pa.sharedSizeBytes;
    // CAI_PAIR_STAGES caps the ring depth (tuning knob; results do not depend on it).
    const int pcap = env_int("CAI_PAIR_STAGES");
    int ps = pcap >= 2 && pcap < 6 ? pcap : 6;
    while (ps > 2 && pair_smem_bytes(ps, c->swap_max_n > 0) > plimit) --ps;
    c->pair_stages = ps;
    c->pair_smem = pair_smem_bytes(ps, c->swap_max_n > 0);
    const int rmax = env_int("CAI_PAIR_RING_MAX");
    if (rmax >= 2 && rmax <= kPairMaxRing) c->pair_ring_max = rmax;
    int clusters = 0;
    if (cudaFuncSetAttribute(c->pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(c->pair_smem)) != cudaSuccess) {
      cudaGetLastError();
      delete c;
      return CAI_ERR_CUDA;
    }
    cudaLaunchConfig_t qc = {};
    qc.gridDim = dim3(static_cast<unsigned>(sms & ~1));
    qc.blockDim = dim3(kPairThreads);
    qc.dynamicSmemBytes = c->pair_smem;
    if (cudaOccupancyMaxActiveClusters(&clusters, c->pair_kernel, &qc) != cudaSuccess ||
        clusters < 1) {
      cudaGetLastError();
      delete c;
      return CAI_ERR_CUDA;
    }
    // CAI_PAIR_CLUSTERS caps the grid (tests: per-tile partials at small M).
    const int cset = env_int("CAI_PAIR_CLUSTERS");
    if (cset > 0 && cset < clusters) clusters = cset;
    c->pair_grid = 2 * clusters;
    // Steps whose row-tile count does not divide the pairs leave one partial
    // per row and vocabulary tile to the reduce kernel; if no step size up to
    // B P does, that kernel is never launched.
    for (int rt = 1; rt <= (c->rows_cap + kPairTileRows - 1) / kPairTileRows; ++rt)
      if (clusters % rt != 0) c->need_reduce = true;
    const int warps_per_cta = kReduceThreads / 32;
    const int want = (c->rows_cap + warps_per_cta - 1) / warps_per_cta;
    c->reduce_grid = want < 4 * sms ? want : 4 * sms;
  }

  const size_t BL = static_cast<size_t>(cfg->B) * c->L;
  const size_t BN = static_cast<size_t>(cfg->B) * cfg->n_blocks;
  void* p;
#define CAI_ALLOC(field, type, count)                                  \
  if ((r = alloc_into(c, &p, sizeof(type) * (count))) != CAI_OK) {    \
    release(c);                                                        \
    delete c;                                                          \
    return r;                                                          \
  }                                                                    \
  field = static_cast<type*>(p);
  CAI_ALLOC(c->st.tok, int, BL)
  CAI_ALLOC(c->st.conf, float, BL)
  CAI_ALLOC(c->st.s0, float, BL)
  CAI_ALLOC(c->st.budget, uint8_t, BL)
  CAI_ALLOC(c->st.cstep, int16_t, BL)
  CAI_ALLOC(c->st.cand, int, BL)
  CAI_ALLOC(c->st.ell, int, cfg->B)
  CAI_ALLOC(c->st.eta, int, cfg->B)
  CAI_ALLOC(c->st.exit_reason, int, BN)
  CAI_ALLOC(c->st.exit_step, int, BN)
  CAI_ALLOC(c->st.unresolved, int, BN)
  CAI_ALLOC(c->st.m_hist, int, static_cast<size_t>(cfg->n_blocks) * cfg->T)
  CAI_ALLOC(c->st.run, uint8_t, BL)
  CAI_ALLOC(c->st.stable, int16_t, BL)
  CAI_ALLOC(c->st.drift, float, BN * cfg->T)
  if (cfg->flags & CAI_DIAGNOSTICS)
    CAI_ALLOC(c->h_prev, __nv_bfloat16, static_cast<size_t>(c->BP) * cfg->H)
  CAI_ALLOC(c->list, int, c->BP)
  CAI_ALLOC(c->row_of, int, c->BP)
  CAI_ALLOC(c->d_M, int, 1)
  CAI_ALLOC(c->ticket, unsigned, 1)
  CAI_ALLOC(c->pub, unsigned long long, 1)
  CAI_ALLOC(c->err, uint32_t, 1)
  CAI_ALLOC(c->hc, __nv_bfloat16, static_cast<size_t>(c->rows_cap) * cfg->H)
  // Partials per row: G (swapped-operand kernel), and with the pair kernel
  // n_vt (one per vocabulary tile) or up to n_pairs (one per pair).
  int part_cols = c->G;
  if (c->use_pair) {
    const int k = c->swap_max_n > 0 ? 2 : 1;  // swapped steps: one partial per CTA of a pair
    part_cols = k * c->n_vt > part_cols ? k * c->n_vt : part_cols;
    part_cols = k * (c->pair_grid / 2) > part_cols ? k * (c->pair_grid / 2) : part_cols;
  }
  CAI_ALLOC(c->part, float4, static_cast<size_t>(c->rows_cap) * part_cols)
  if (c->use_pair) {
    CAI_ALLOC(c->wt, uint8_t, static_cast<size_t>(2 * c->n_vt) * kPairHalf * 2 * cfg->H)
    CAI_ALLOC(c->rowres, float4, c->rows_cap)
  }
  CAI_ALLOC(c->hidden_stage, uint8_t, static_cast<size_t>(c->BP) * cfg->H * 2)
  if (!shard) {
    c->stage2[0] = c->hidden_stage;
    CAI_ALLOC(c->stage2[1], uint8_t, static_cast<size_t>(c->BP) * cfg->H * 2)
    CAI_ALLOC(c->stage_seq_dev, unsigned long long, 2)
    if (cudaMemset(c->stage_seq_dev, 0, 16) != cudaSuccess) {
      release(c);
      delete c;
      return CAI_ERR_CUDA;
    }
    c->stage_by_word = !(c->fused && c->norm) && !(cfg->flags & CAI_DIAGNOSTICS) &&
                       get_write_value64() != nullptr;
  }
  // The swapped-operand kernel's packed W, only where that kernel runs (every
  // single-kernel step; multi-kernel steps with CAI_PAIR_SWAP=0 or CAI_PAIR=0).
  if (c->head_in_step) CAI_ALLOC(c->wpk, uint8_t, static_cast<size_t>(units) * kUnitRows * 2 * cfg->H)
  if (c->norm) {
    CAI_ALLOC(c->inv_r, float, c->rows_cap)
    if (cudaMemset(c->inv_r, 0, sizeof(float) * c->rows_cap) != cudaSuccess) {
      release(c);
      delete c;
      return CAI_ERR_CUDA;
    }
  }
  // The norm weight, on the device for the pack kernels (staged if host).
  const __nv_bfloat16* g_dev = static_cast<const __nv_bfloat16*>(g);
  void* g_tmp = nullptr;
  if (g && !is_device_ptr(g)) {
    if ((r = dev_alloc(&g_tmp, static_cast<size_t>(cfg->H) * 2)) != CAI_OK) {
      release(c);
      delete c;
      return r;
    }
    if (cudaMemcpy(g_tmp, g, static_cast<size_t>(cfg->H) * 2, cudaMemcpyHostToDevice) !=
        cudaSuccess) {
      cudaFree(g_tmp);
      release(c);
      delete c;
      return CAI_ERR_CUDA;
    }
    g_dev = static_cast<const __nv_bfloat16*>(g_tmp);
  }
  const void* w_src = W;
  void* w_tmp = nullptr;
  if (!is_device_ptr(W)) {
    if ((r = dev_alloc(&w_tmp, static_cast<size_t>(cfg->V) * cfg->H * 2)) != CAI_OK) {
      if (g_tmp) cudaFree(g_tmp);
      release(c);
      delete c;
      return r;
    }
    if (cudaMemcpy(w_tmp, W, static_cast<size_t>(cfg->V) * cfg->H * 2, cudaMemcpyHostToDevice) !=
        cudaSuccess) {
      cudaFree(w_tmp);
      if (g_tmp) cudaFree(g_tmp);
      release(c);
      delete c;
      return CAI_ERR_CUDA;
    }
    w_src = w_tmp;
  }
  {
    const long long n_chunks = static_cast<long long>(units) * kUnitRows * cfg->H / 8;
    if (c->rows_head)
      pack_weight_rows_kernel<<<4 * sms, 256, 0, static_cast<cudaStream_t>(stream)>>>(
          static_cast<const uint4*>(w_src), static_cast<uint4*>(c->wpk), cfg->V, cfg->H, units,
          c->G, n_chunks, g_dev);
    else if (c->head_in_step)
      pack_weight_kernel<<<4 * sms, 256, 0, static_cast<cudaStream_t>(stream)>>>(
          static_cast<const uint4*>(w_src), static_cast<uint4*>(c->wpk), cfg->V, cfg->H, units,
          c->G, c->gmax, n_chunks, g_dev);
    if (c->use_pair)
      pack_w_tiles_kernel<<<4 * sms, 256, 0, static_cast<cudaStream_t>(stream)>>>(
          static_cast<const uint4*>(w_src), static_cast<uint4*>(c->wt), cfg->V, cfg->H,
          static_cast<long long>(2 * c->n_vt) * kPairHalf * cfg->H / 8, g_dev);
    const cudaError_t e1 = cudaGetLastError();
    const cudaError_t e2 = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    if (w_tmp) cudaFree(w_tmp);
    if (g_tmp) cudaFree(g_tmp);
    if (e1 != cudaSuccess || e2 != cudaSuccess) {
      release(c);
      delete c;
      return CAI_ERR_CUDA;
    }
  }
#undef CAI_ALLOC
  if (cudaHostAlloc(reinterpret_cast<void**>(&c->hf_host), sizeof(HostFlag), cudaHostAllocMapped) !=
          cudaSuccess ||
      cudaHostGetDevicePointer(reinterpret_cast<void**>(&c->hf_dev), c->hf_host, 0) != cudaSuccess) {
    cudaGetLastError();
    release(c);
    delete c;
    return CAI_ERR_NOMEM;
  }
  std::memset(c->hf_host, 0, sizeof(HostFlag));
  if (!make_map(&c->tm_h, c->hc, c->rows_cap, cfg->H, kBoxRowsB) ||
      (c->use_pair && !make_map(&c->tm_a, c->hc, c->rows_cap, cfg->H, kPairHalf)) ||
      (c->swap_max_n && !make_row_maps(c, cfg->H)) ||
      (c->use_pair &&
       !make_map(&c->tm_w, c->wt, static_cast<uint64_t>(2 * c->n_vt) * (cfg->H / kPairBlockK) *
                                      kPairHalf,
                 kPairBlockK, kPairHalf, CU_TENSOR_MAP_SWIZZLE_NONE))) {
    release(c);
    delete c;
    return CAI_ERR_CUDA;
  }
  if (!shard) {
    bool ok = (!c->fused || (make_map(&c->tm_stage[0], c->stage2[0], c->BP, cfg->H, kBoxRowsB) &&
                             make_map(&c->tm_stage[1], c->stage2[1], c->BP, cfg->H, kBoxRowsB))) &&
              cudaStreamCreateWithFlags(&c->copy_stream, cudaStreamNonBlocking) == cudaSuccess;
    for (int k = 0; ok && k < 2; ++k)
      ok = cudaEventCreateWithFlags(&c->ev_copied[k], cudaEventDisableTiming) == cudaSuccess &&
           cudaEventCreateWithFlags(&c->ev_read[k], cudaEventDisableTiming) == cudaSuccess;
    if (!ok) {
      cudaGetLastError();
      release(c);
      delete c;
      return CAI_ERR_CUDA;
    }
  }
  // All step kernels ask for the same (largest) shared-memory carveout, so the
  // small gather and merge CTAs can be resident on an SM beside an LM-head
  // CTA; under programmatic dependent launch they then start, and wait, while
  // the neighbouring kernel still runs.
  if (cudaFuncSetAttribute(c->head_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(c->head_smem)) != cudaSuccess ||
      cudaFuncSetAttribute(c->head_kernel,
                           cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared) != cudaSuccess ||
      cudaFuncSetAttribute(gather_rows_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared) != cudaSuccess ||
      cudaFuncSetAttribute(merge_commit_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared) != cudaSuccess) {
    cudaGetLastError();
    release(c);
    delete c;
    return CAI_ERR_CUDA;
  }
  c->stats.grid = c->G;
  c->stats.stages = c->n_stages;
  c->stats.n_max = c->n_max;
  c->stats.pair_grid = c->use_pair ? c->pair_grid : 0;
  c->stats.pair_swap_max_n = c->swap_max_n;
  c->stats.pair_stages = c->use_pair ? c->pair_stages : 0;
  c->stats.head_rows = c->rows_head ? 1 : 0;
  c->stats.kernels_per_step =
      c->fused ? 1
               : 2 + (c->head_in_step ? 1 : 0) + (c->use_pair ? 1 : 0) + (c->need_reduce ? 1 : 0) +
                     (c->shard ? 2 : 0);
  r = cai_reset(c, stream);
  if (r != CAI_OK) {
    release(c);
    delete c;
    return r;
  }
  *out = c;
  return CAI_OK;
}

}  // namespace

int cai_init(const cai_config* cfg, const void* W, void* stream, cai_ctx** out) {
  return init_impl(cfg, W, nullptr, 0.0, 0, 0, stream, out);
}

int cai_init_rmsnorm(const cai_config* cfg, const void* W, const void* norm_weight, double eps,
                     void* stream, cai_ctx** out) {
  if (!norm_weight || reinterpret_cast<uintptr_t>(norm_weight) % 2 != 0 || !(eps >= 0.0) ||
      !std::isfinite(eps))
    return CAI_ERR_ARG;
  return init_impl(cfg, W, norm_weight, eps, 0, 0, stream, out);
}

int cai_init_vocab_shard(const cai_config* cfg, const void* W_shard, int32_t v0, int32_t V_shard,
                         void* stream, cai_ctx** out) {
  if (V_shard < 1) return CAI_ERR_SHAPE;
  return init_impl(cfg, W_shard, nullptr, 0.0, v0, V_shard, stream, out);
}

int cai_reset(cai_ctx* c, void* stream_v) {
  if (!c) return CAI_ERR_ARG;
  if (c->sticky) return c->sticky;
  cudaStream_t s = static_cast<cudaStream_t>(stream_v);
  const cai_config& cfg = c->cfg;
  const size_t BL = static_cast<size_t>(cfg.B) * c->L;
  const size_t BN = static_cast<size_t>(cfg.B) * cfg.n_blocks;
  bool ok = cudaMemsetAsync(c->st.tok, 0xFF, BL * 4, s) == cudaSuccess &&
            cudaMemsetAsync(c->st.conf, 0, BL * 4, s) == cudaSuccess &&
            cudaMemsetAsync(c->st.s0, 0, BL * 4, s) == cudaSuccess &&
            cudaMemsetAsync(c->st.budget, 0, BL, s) == cudaSuccess &&
            cudaMemsetAsync(c->st.cstep, 0xFF, BL * 2, s) == cudaSuccess &&
            cudaMemsetAsync(c->st.cand, 0xFF, BL * 4, s) == cudaSuccess &&
            cudaMemsetAsync(c->st.ell, 0, cfg.B * 4, s) == cudaSuccess &&
            cudaMemsetAsync(c->st.eta, 0, cfg.B * 4, s) == cudaSuccess &&
            cudaMemsetAsync(c->st.exit_reason, 0, BN * 4, s) == cudaSuccess &&
            cudaMemsetAsync(c->st.exit_step, 0xFF, BN * 4, s) == cudaSuccess &&
            cudaMemsetAsync(c->st.unresolved, 0, BN * 4, s) == cudaSuccess &&
            cudaMemsetAsync(c->st.m_hist, 0, static_cast<size_t>(cfg.n_blocks) * cfg.T * 4, s) ==
                cudaSuccess &&
            cudaMemsetAsync(c->st.run, 0, BL, s) == cudaSuccess &&
            cudaMemsetAsync(c->st.stable, 0xFF, BL * 2, s) == cudaSuccess &&
            cudaMemsetAsync(c->st.drift, 0xFF, BN * cfg.T * 4, s) == cudaSuccess &&  // NaN
            cudaMemsetAsync(c->ticket, 0, 4, s) == cudaSuccess &&
            cudaMemsetAsync(c->pub, 0, 8, s) == cudaSuccess &&
            cudaMemsetAsync(c->err, 0, 4, s) == cudaSuccess &&
            cudaMemsetAsync(c->d_M, 0, 4, s) == cudaSuccess;
  if (!ok) return fail(c, CAI_ERR_CUDA);
  // Step ids keep increasing across resets, so a host-flag write still in
  // flight from the previous generation never satisfies a poll of this one.
  c->blk = 0;
  c->t_next = 0;
  c->block_done_seen = false;
  c->shard_pending = false;
  return CAI_OK;
}

int cai_first_step(cai_ctx* c, const void* hidden, void* stream) {
  if (!c || !hidden || c->shard) return CAI_ERR_ARG;
  if (c->sticky) return c->sticky;
  if (reinterpret_cast<uintptr_t>(hidden) % 16 != 0) return CAI_ERR_ARG;
  if (c->t_next != 0) return CAI_ERR_ORDER;
  c->block_done_seen = false;
  return step(c, hidden, stream, true);
}

int cai_denoise_step(cai_ctx* c, const void* hidden, void* stream) {
  if (!c || !hidden || c->shard) return CAI_ERR_ARG;
  if (c->sticky) return c->sticky;
  if (reinterpret_cast<uintptr_t>(hidden) % 16 != 0) return CAI_ERR_ARG;
  if (c->t_next < 1 || c->t_next >= c->cfg.T || c->block_done_seen) return CAI_ERR_ORDER;
  return step(c, hidden, stream, false);
}

int cai_block_advance(cai_ctx* c, void* stream) {
  (void)stream;
  if (!c) return CAI_ERR_ARG;
  if (c->sticky) return c->sticky;
  if (c->t_next < 1 || c->blk + 1 >= c->cfg.n_blocks || c->shard_pending) return CAI_ERR_ORDER;
  c->blk += 1;
  c->t_next = 0;
  c->block_done_seen = false;
  return CAI_OK;
}

int cai_shard_rows(const cai_ctx* c, int32_t* rows) {
  if (!c || !rows || !c->shard) return CAI_ERR_ARG;
  *rows = c->rows_cap;
  return CAI_OK;
}

int cai_shard_head(cai_ctx* c, const void* hidden, void* triples, void* stream_v) {
  if (!c || !hidden || !triples || !c->shard) return CAI_ERR_ARG;
  if (c->sticky) return c->sticky;
  if (reinterpret_cast<uintptr_t>(hidden) % 16 != 0 ||
      reinterpret_cast<uintptr_t>(triples) % 16 != 0 || !is_device_ptr(triples))
    return CAI_ERR_ARG;
  const bool first = c->t_next == 0;
  if (c->shard_pending || (!first && (c->t_next >= c->cfg.T || c->block_done_seen)))
    return CAI_ERR_ORDER;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_v);
  const void* hid = nullptr;
  int r = multi_kernel_rows(c, hidden, stream, &hid);
  if (r != CAI_OK) return r;
  if (first) c->block_done_seen = false;
  if ((r = launch_gather(c, hid, first, stream)) != CAI_OK) return r;
  if ((r = launch_pair_head(c, c->t_next, stream)) != CAI_OK) return r;
  ShardRowsParams sp{};
  sp.part = c->part;
  sp.rowres = c->rowres;
  sp.d_M = c->d_M;
  sp.out = static_cast<float4*>(triples);
  sp.rows_cap = c->rows_cap;
  sp.n_pairs = c->pair_grid / 2;
  sp.swap_max_n = c->swap_max_n;
  sp.v_off = c->v_off;
  const int warps = kShardThreads / 32;
  if (launch_pdl(c->pdl, shard_rows_kernel, (c->rows_cap + warps - 1) / warps, kShardThreads, 0,
                 stream, sp) != cudaSuccess)
    return check_launch(c);
  c->stats.launches++;
  c->stats.head_launches++;
  if ((r = check_launch(c)) != CAI_OK) return r;
  c->shard_pending = true;
  c->shard_first = first;
  return CAI_OK;
}

int cai_shard_commit(cai_ctx* c, const void* gathered, int32_t n_shards, void* stream_v) {
  if (!c || !gathered || !c->shard || n_shards < 1 || n_shards > 4096) return CAI_ERR_ARG;
  if (c->sticky) return c->sticky;
  if (reinterpret_cast<uintptr_t>(gathered) % 16 != 0 || !is_device_ptr(gathered))
    return CAI_ERR_ARG;
  if (!c->shard_pending) return CAI_ERR_ORDER;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_v);
  const int t = c->t_next;
  const int64_t step_id = c->last_step_id + 1;
  ShardMergeParams mp{};
  mp.gathered = static_cast<const float4*>(gathered);
  mp.rowres = c->rowres;
  mp.d_M = c->d_M;
  mp.rows_cap = c->rows_cap;
  mp.n_shards = n_shards;
  const int warps = kShardThreads / 32;
  if (launch_pdl(c->pdl, shard_merge_kernel, (c->rows_cap + warps - 1) / warps, kShardThreads, 0,
                 stream, mp) != cudaSuccess)
    return check_launch(c);
  c->stats.launches++;
  // The commit reads the one merged triple per row.
  CommitParams cp = commit_params(c, t, step_id);
  cp.part = c->rowres;
  cp.n_part = 1;
  cp.pair_min_M = INT_MAX;
  cp.prefetch_state = 0;  // the exchange before it is the caller's
  const int commit_threads = c->cfg.P < kCommitThreads / 32 ? 32 * c->cfg.P : kCommitThreads;
  if (launch_pdl(c->pdl, merge_commit_kernel, c->cfg.B, commit_threads, 0, stream, cp) !=
      cudaSuccess)
    return check_launch(c);
  c->stats.launches++;
  c->stats.steps++;
  const int r = check_launch(c);
  if (r != CAI_OK) return r;
  c->shard_pending = false;
  c->last_step_id = step_id;
  c->t_next = t + 1;
  return CAI_OK;
}

int cai_poll(cai_ctx* c, int32_t lag, int32_t timeout_ms, int32_t* all_done) {
  if (!c || !all_done || lag < 0) return CAI_ERR_ARG;
  if (c->sticky) return c->sticky;
  *all_done = 0;
  const int64_t target = c->last_step_id - lag;
  if (target < 0) return CAI_OK;
  volatile unsigned long long* word = &c->hf_host->word;
  const auto t0 = std::chrono::steady_clock::now();
  unsigned long long w = 0;
  for (uint32_t it = 0;; ++it) {
    w = *word;
    // The word holds step id + 1 (ids are kept since cai_init); 0 means "none yet".
    const bool seen = static_cast<int64_t>(w & 0xFFFFFFFFull) - 1 >= target;
    if ((w >> 33) & 1ull) return fail(c, CAI_ERR_DEVICE);
    if (seen) break;
    if ((it & 255u) == 255u) {
      const auto dt = std::chrono::steady_clock::now() - t0;
      if (std::chrono::duration_cast<std::chrono::milliseconds>(dt).count() >= timeout_ms)
        return CAI_ERR_TIMEOUT;
      std::this_thread::yield();
    }
  }
  const int blk = static_cast<int>((w >> 34) & 0x7FFFull);
  if (blk == (c->blk & 0x7FFF) && ((w >> 32) & 1ull)) {
    *all_done = 1;
    c->block_done_seen = true;
  }
  return CAI_OK;
}

int cai_get_state(cai_ctx* c, cai_state_view* v) {
  if (!c || !v) return CAI_ERR_ARG;
  v->tok = c->st.tok;
  v->conf = c->st.conf;
  v->s0 = c->st.s0;
  v->budget = c->st.budget;
  v->cstep = c->st.cstep;
  v->cand = c->st.cand;
  v->ell = c->st.ell;
  v->eta = c->st.eta;
  v->exit_reason = c->st.exit_reason;
  v->exit_step = c->st.exit_step;
  v->unresolved = c->st.unresolved;
  v->m_hist = c->st.m_hist;
  v->run = c->st.run;
  v->stable = c->st.stable;
  v->drift = c->st.drift;
  return CAI_OK;
}

static int transfer(cai_ctx* c, const cai_host_state* h, bool down) {
  const cai_config& cfg = c->cfg;
  const size_t BL = static_cast<size_t>(cfg.B) * c->L;
  const size_t BN = static_cast<size_t>(cfg.B) * cfg.n_blocks;
  struct F {
    void* host;
    void* dev;
    size_t bytes;
  } f[] = {
      {h->tok, c->st.tok, BL * 4},         {h->conf, c->st.conf, BL * 4},
      {h->s0, c->st.s0, BL * 4},           {h->budget, c->st.budget, BL},
      {h->cstep, c->st.cstep, BL * 2},     {h->cand, c->st.cand, BL * 4},
      {h->ell, c->st.ell, cfg.B * 4u},     {h->eta, c->st.eta, cfg.B * 4u},
      {h->exit_reason, c->st.exit_reason, BN * 4}, {h->exit_step, c->st.exit_step, BN * 4},
      {h->unresolved, c->st.unresolved, BN * 4},
      {h->m_hist, c->st.m_hist, static_cast<size_t>(cfg.n_blocks) * cfg.T * 4},
      {h->run, c->st.run, BL},
      {h->stable, c->st.stable, BL * 2},
      {h->drift, c->st.drift, BN * cfg.T * 4},
  };
  if (cudaDeviceSynchronize() != cudaSuccess) return fail(c, CAI_ERR_CUDA);
  for (const F& x : f) {
    if (!x.host) continue;
    cudaError_t e = down ? cudaMemcpy(x.host, x.dev, x.bytes, cudaMemcpyDeviceToHost)
                         : cudaMemcpy(x.dev, x.host, x.bytes, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return fail(c, CAI_ERR_CUDA);
  }
  return CAI_OK;
}

int cai_state_download(cai_ctx* c, cai_host_state* dst) {
  if (!c || !dst) return CAI_ERR_ARG;
  if (c->sticky) return c->sticky;
  int r = transfer(c, dst, true);
  if (r != CAI_OK) return r;
  dst->blk = c->blk;
  dst->t_next = c->t_next;
  uint32_t err = 0;
  if (cudaMemcpy(&err, c->err, 4, cudaMemcpyDeviceToHost) != cudaSuccess) return fail(c, CAI_ERR_CUDA);
  if (err) return fail(c, CAI_ERR_DEVICE);
  return CAI_OK;
}

int cai_state_upload(cai_ctx* c, const cai_host_state* src) {
  if (!c || !src) return CAI_ERR_ARG;
  if (c->sticky) return c->sticky;
  if (src->blk < 0 || src->blk >= c->cfg.n_blocks || src->t_next < 0 || src->t_next > c->cfg.T)
    return CAI_ERR_ARG;
  int r = transfer(c, src, false);
  if (r != CAI_OK) return r;
  // The uploaded state replaces what the last step published.
  if (cudaMemset(c->pub, 0, 8) != cudaSuccess) return fail(c, CAI_ERR_CUDA);
  c->blk = src->blk;
  c->t_next = src->t_next;
  c->block_done_seen = false;
  ListParams lp{};
  lp.tok = c->st.tok;
  lp.exit_reason = c->st.exit_reason;
  lp.list = c->list;
  lp.row_of = c->row_of;
  lp.d_M = c->d_M;
  lp.B = c->cfg.B;
  lp.P = c->cfg.P;
  lp.L = c->L;
  lp.n_blocks = c->cfg.n_blocks;
  lp.blk = c->blk;
  rebuild_list_kernel<<<1, kListThreads>>>(lp);
  c->stats.launches++;
  r = check_launch(c);
  if (r != CAI_OK) return r;
  if (cudaDeviceSynchronize() != cudaSuccess) return fail(c, CAI_ERR_CUDA);
  return CAI_OK;
}

int cai_read_tokens(cai_ctx* c, int32_t* host_tokens, void* stream) {
  if (!c || !host_tokens) return CAI_ERR_ARG;
  if (c->sticky) return c->sticky;
  if (cudaMemcpyAsync(host_tokens, c->st.tok, static_cast<size_t>(c->cfg.B) * c->L * 4,
                      cudaMemcpyDeviceToHost, static_cast<cudaStream_t>(stream)) != cudaSuccess)
    return fail(c, CAI_ERR_CUDA);
  return CAI_OK;
}

int cai_profile(cai_ctx* c, int32_t enable) {
  if (!c) return CAI_ERR_ARG;
  c->profiling = enable != 0;
  return CAI_OK;
}

int cai_device_error_bits(cai_ctx* c, uint32_t* bits) {
  if (!c || !bits) return CAI_ERR_ARG;
  static_assert(CAI_DEVERR_WAIT_EMPTY == kErrWaitEmpty && CAI_DEVERR_WAIT_FULL == kErrWaitFull &&
                    CAI_DEVERR_WAIT_ACC_FULL == kErrWaitAccFull &&
                    CAI_DEVERR_WAIT_ACC_EMPTY == kErrWaitAccEmpty && CAI_DEVERR_DRAIN == kErrDrain &&
                    CAI_DEVERR_BAD_ROW == kErrBadRow && CAI_DEVERR_WAIT_EPI == kErrWaitEpi &&
                    CAI_DEVERR_BOUNDS == kErrBounds && CAI_DEVERR_WAIT_ROWS == kErrWaitRows,
                "error bits of the header and the kernels");
  if (cudaMemcpy(bits, c->err, sizeof(uint32_t), cudaMemcpyDeviceToHost) != cudaSuccess) {
    cudaGetLastError();
    return CAI_ERR_CUDA;
  }
  return CAI_OK;
}

int cai_get_stats(cai_ctx* c, cai_stats* out) {
  if (!c || !out) return CAI_ERR_ARG;
  if (c->sticky) return c->sticky;
  double ms = 0.0, step_ms = 0.0;
  for (size_t i = 0; i < c->ev_used; i += 4) {
    if (cudaEventSynchronize(c->ev_pool[i + 3]) != cudaSuccess) return fail(c, CAI_ERR_CUDA);
    float m = 0.f, s = 0.f;
    if (cudaEventElapsedTime(&m, c->ev_pool[i + 1], c->ev_pool[i + 2]) != cudaSuccess ||
        cudaEventElapsedTime(&s, c->ev_pool[i], c->ev_pool[i + 3]) != cudaSuccess)
      return fail(c, CAI_ERR_CUDA);
    ms += m;
    step_ms += s;
  }
  c->stats.head_ms += ms;
  c->stats.step_ms += step_ms;
  c->stats.head_profiled += static_cast<int64_t>(c->ev_used / 4);
  c->ev_used = 0;
  *out = c->stats;
  return CAI_OK;
}

void cai_free(cai_ctx* c) {
  if (!c) return;
  cudaDeviceSynchronize();
  release(c);
  delete c;
}

const char* cai_strerror(int s) {
  switch (s) {
    case CAI_OK: return "ok";
    case CAI_ERR_ARG: return "invalid argument";
    case CAI_ERR_SHAPE: return "unsupported shape";
    case CAI_ERR_ORDER: return "call out of order";
    case CAI_ERR_CUDA: return "CUDA runtime error";
    case CAI_ERR_TIMEOUT: return "timed out waiting for the device";
    case CAI_ERR_DEVICE: return "a kernel gave up a bounded wait";
    case CAI_ERR_UNSUPPORTED: return "device is not compute capability 10.3";
    case CAI_ERR_NOMEM: return "out of memory";
    default: return "unknown status";
  }
}

int cai_test_check_guards(cai_ctx* c, int32_t* n_bad) {
  if (!c || !n_bad) return CAI_ERR_ARG;
  if (cudaDeviceSynchronize() != cudaSuccess) return fail(c, CAI_ERR_CUDA);
  unsigned char buf[kGuardBytes];
  int bad = 0;
  for (size_t i = 0; i < c->allocs.size(); ++i) {
    if (cudaMemcpy(buf, static_cast<char*>(c->allocs[i]) + c->alloc_bytes[i], kGuardBytes,
                   cudaMemcpyDeviceToHost) != cudaSuccess)
      return fail(c, CAI_ERR_CUDA);
    for (size_t k = 0; k < kGuardBytes; ++k) {
      if (buf[k] != kGuardByte) {
        ++bad;
        break;
      }
    }
  }
  *n_bad = bad;
  return CAI_OK;
}

int cai_test_head_grid_limit(int32_t n) {
  if (n < 0) return CAI_ERR_ARG;
  g_head_grid_limit.store(n);
  return CAI_OK;
}

int cai_test_wait_timeout(cai_ctx* c, void* stream) {
  if (!c) return CAI_ERR_ARG;
  if (c->sticky) return c->sticky;
  wait_timeout_probe_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(c->err, kErrWaitFull);
  c->stats.launches++;
  return check_launch(c);
}

int cai_test_pair_plan(int32_t M, int32_t n_pairs, int32_t swap_max_n, int32_t* out) {
  if (M < 1 || n_pairs < 1 || swap_max_n < 0 || !out) return CAI_ERR_ARG;
  const bool swap = pair_swapped(M, swap_max_n);
  const int n_rt = pair_row_tiles(M);
  out[0] = swap ? 1 : 0;
  out[1] = n_rt;
  out[2] = swap ? swap_tile_cols(M, n_rt) : kPairTileRows;
  out[3] = pair_partials_per_row(M, n_pairs, swap);
  return CAI_OK;
}

int cai_test_theta_table(const cai_config* cfg, int32_t blk, int32_t t, float* out) {
  if (!cfg || !out) return CAI_ERR_ARG;
  const int r = validate(cfg);
  if (r != CAI_OK) return r;
  if (blk < 0 || blk >= cfg->n_blocks || t < 0 || t >= cfg->T) return CAI_ERR_ARG;
  for (int p = 0; p < cfg->P; ++p) out[p] = theta_token_of(*cfg, blk + 1, t, p);
  return CAI_OK;
}

int cai_test_fail_alloc_after(int32_t n) {
  if (n < 0) return CAI_ERR_ARG;
  g_fail_alloc_after.store(n);
  return CAI_OK;
}

}  // extern "C"

// The allocation-free decoding head (cai_head_rows_static).
#include "static_head.cuh"
