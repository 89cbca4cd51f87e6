// cai_head_rows_static: the decoding head (confidence and argmax of every
// row) for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc at the point where they need the head:
// code running while a memory pool owns the whole device, allocator-free
// inference runtimes that reserve all memory up front, or a caller inside a
// region where a new allocation would synchronise the device.  This entry point
// allocates nothing.  The caller passes its own weight, rows and outputs; the
// only scratch (the per-CTA softmax partials) is a fixed, file-scope device
// array that every GPU loading this library holds until the process exits.
//
// Kernels: a variant of the LM-head kernel that reads the caller's row-major W
// in place through TMA boxes (the context path reads a packed copy instead),
// one tile of 128 vocabulary rows at a time, and writes its partials into the
// static scratch; then one warp per row merges them.
//
// Included once, at the end of cai.cu (it uses the device helpers of
// head_kernel.cuh, whose kernels must be defined in a single unit).
#pragma once

#include <atomic>
#include <mutex>

namespace cai {
namespace {

constexpr int kStaticMaxRows = 256;  // rows per call (one MMA chunk)
constexpr int kStaticMaxCtas = 160;  // LM-head CTAs per call
constexpr int kStaticStages = 4;     // W tile (16 KiB) + up to 256 rows (32 KiB) per stage
constexpr int kStaticMaxDevices = 64;

// The whole scratch of the entry point: partial triples [row][CTA], plus one
// error word.  640 KiB + 256 bytes on every device that loads the library.
static __device__ __align__(256) float4 g_static_part[kStaticMaxRows * kStaticMaxCtas];
static __device__ __align__(256) uint32_t g_static_err[64];

struct StaticSmem {
  uint8_t* stage;    // n_stages x (16 KiB W + 32 KiB rows)
  float4* epi;       // [4][256] cross-warp merge
  uint64_t* full;
  uint64_t* empty;
  uint64_t* accf;    // 2
  uint64_t* acce;    // 2
  uint64_t* epib;    // 1
  uint64_t* drain;   // 1
  uint32_t* tmem_slot;
  volatile int* abort;
};

constexpr int kStaticStageBytes = kATileBytes + kStaticMaxRows * 128;
constexpr size_t kStaticSmemBytes =
    1024 + static_cast<size_t>(kStaticStages) * kStaticStageBytes + 4 * 256 * 16 +
    (2 * kStaticStages + 6) * 8 + 16;

__device__ StaticSmem carve_static(uint8_t* raw) {
  StaticSmem s;
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  s.stage = base;
  s.epi = reinterpret_cast<float4*>(base + static_cast<size_t>(kStaticStages) * kStaticStageBytes);
  s.full = reinterpret_cast<uint64_t*>(s.epi + 4 * 256);
  s.empty = s.full + kStaticStages;
  s.accf = s.empty + kStaticStages;
  s.acce = s.accf + 2;
  s.epib = s.acce + 2;
  s.drain = s.epib + 1;
  s.tmem_slot = reinterpret_cast<uint32_t*>(s.drain + 1);
  s.abort = reinterpret_cast<volatile int*>(s.tmem_slot + 1);
  return s;
}

// LM head over M <= 256 caller rows against the caller's W [V, H]: CTA c
// takes 128-row tiles [c T / G, (c + 1) T / G) of the T = ceil(V / 128) tiles;
// rows >= V are filled with zeros by the TMA and masked in the epilogue.
__global__ void __launch_bounds__(kHeadThreads, 1)
    lm_head_rows_static_kernel(const __grid_constant__ CUtensorMap tm_w,
                               const __grid_constant__ CUtensorMap tm_r, float4* part,
                               uint32_t* err, int V, int H, int M, int n_tiles_total) {
  extern __shared__ uint8_t smem_raw[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  StaticSmem sm = carve_static(smem_raw);
  const int G = gridDim.x, cta = blockIdx.x;
  const int t0 = static_cast<int>((static_cast<long long>(cta) * n_tiles_total) / G);
  const int t1 = static_cast<int>((static_cast<long long>(cta + 1) * n_tiles_total) / G);
  const int KB = H / kBlockK;
  const int nq = (M + 15) & ~15;
  const int ngroups = (nq + 31) >> 5;
  constexpr int kTmemCols = 512;  // two 256-column accumulators

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStaticStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&sm.accf[a], 1);
      mbar_init(&sm.acce[a], 4);
    }
    mbar_init(sm.epib, 4);
    mbar_init(sm.drain, 1);
    *sm.abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(sm.tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *sm.tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      const uint64_t pol_w = policy_evict_first(), pol_r = policy_evict_last();
      Ring r;
      long long issued = 0;
      bool ok = true;
      for (int t = t0; t < t1 && ok; ++t) {
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(&sm.empty[r.slot], r.phase ^ 1u, sm.abort, err, kErrWaitEmpty)) {
            ok = false;
            break;
          }
          uint8_t* st = sm.stage + static_cast<size_t>(r.slot) * kStaticStageBytes;
          mbar_arrive_expect_tx(&sm.full[r.slot], static_cast<uint32_t>(kATileBytes + nq * 128));
          tma_load_2d(st, &tm_w, &sm.full[r.slot], kb * kBlockK, t * kRowsPerTile, pol_w);
          for (int i = 0; i < nq / kBoxRowsB; ++i)
            tma_load_2d(st + kATileBytes + i * kBoxRowsB * 128, &tm_r, &sm.full[r.slot],
                        kb * kBlockK, i * kBoxRowsB, pol_r);
          ++issued;
          r.next(kStaticStages);
        }
      }
      if (!ok) {
        const long long f = issued > kStaticStages ? issued - kStaticStages : 0;
        for (long long i = f; i < issued; ++i)
          mbar_drain(&sm.full[i % kStaticStages], static_cast<uint32_t>((i / kStaticStages) & 1),
                     err);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(kRowsPerTile, static_cast<uint32_t>(nq));
      Ring r, racc;
      bool ok = true;
      for (int t = t0; t < t1 && ok; ++t) {
        if (!mbar_wait(&sm.acce[racc.slot], racc.phase ^ 1u, sm.abort, err, kErrWaitAccEmpty)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(racc.slot * 256);
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(&sm.full[r.slot], r.phase, sm.abort, err, kErrWaitFull)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a = smem_addr(sm.stage + static_cast<size_t>(r.slot) * kStaticStageBytes);
          const uint32_t b = a + kATileBytes;
#pragma unroll
          for (int kk = 0; kk < kBlockK / 16; ++kk)
            mma_bf16(d_tmem, sdesc_k_sw128(a + kk * 32), sdesc_k_sw128(b + kk * 32), idesc,
                     (kb | kk) != 0 ? 1u : 0u);
          mma_commit(&sm.empty[r.slot]);
          r.next(kStaticStages);
        }
        if (!ok) break;
        mma_commit(&sm.accf[racc.slot]);
        racc.next(2);
      }
      if (!ok) {
        mma_commit(sm.drain);
        mbar_drain(sm.drain, 0, err);
      }
    }
    __syncwarp();
  } else {
    const int ew = warp - 2, quarter = warp & 3;
    const uint32_t lane_base = static_cast<uint32_t>(quarter * 32) << 16;
    float rm[8], rs[8];
    int ri[8];
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      rm[c] = kNegBig;
      rs[c] = 0.0f;
      ri[c] = INT_MAX;
    }
    Ring racc;
    bool ok = true;
    for (int t = t0; t < t1; ++t) {
      if (!mbar_wait(&sm.accf[racc.slot], racc.phase, sm.abort, err, kErrWaitAccFull)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const int vrow = t * kRowsPerTile + quarter * 32 + lane;
      const bool valid = vrow < V;
      const uint32_t tcol = tmem_base + lane_base + static_cast<uint32_t>(racc.slot * 256);
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        if (c < ngroups) {
          uint32_t v[32];
          tmem_ld_32cols(tcol + 32 * c, v);
          tmem_ld_wait();
          float m, s;
          int i;
          transpose_reduce32(v, valid, vrow, lane, m, s, i);
          merge_tri(rm[c], rs[c], ri[c], m, s, i);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.acce[racc.slot]);
      racc.next(2);
    }
    if (ok) {
#pragma unroll
      for (int c = 0; c < 8; ++c)
        if (c < ngroups)
          sm.epi[ew * 256 + 32 * c + lane] = make_float4(rm[c], rs[c], __int_as_float(ri[c]), 0.0f);
      __syncwarp();
      if (lane == 0) mbar_arrive(sm.epib);
      if (mbar_wait(sm.epib, 0, sm.abort, err, kErrWaitEpi)) {
        for (int col = ew * 32 + lane; col < M; col += 128) {
          const float4 a = sm.epi[col];
          float m = a.x, s = a.y;
          int i = __float_as_int(a.z);
#pragma unroll
          for (int w = 1; w < 4; ++w) {
            const float4 b = sm.epi[w * 256 + col];
            merge_tri(m, s, i, b.x, b.y, __float_as_int(b.z));
          }
          part[static_cast<size_t>(col) * G + cta] = make_float4(m, s, __int_as_float(i), 0.0f);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// One warp per row: merge the G partials, write c = 1 / S and the argmax.  If
// a bounded wait of the LM-head kernel gave up, every output is NaN / -1; the
// error word is then cleared for the next call.
__global__ void merge_rows_static_kernel(const float4* part, uint32_t* err, int M, int G,
                                         float* conf, int32_t* argmax) {
  const int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= M) return;
  float m = kNegBig, s = 0.0f;
  int ix = INT_MAX;
  for (int k = lane; k < G; k += 32) {
    const float4 q = part[static_cast<size_t>(row) * G + k];
    merge_tri(m, s, ix, q.x, q.y, __float_as_int(q.z));
  }
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) {
    const float mo = __shfl_xor_sync(0xffffffffu, m, off);
    const float so = __shfl_xor_sync(0xffffffffu, s, off);
    const int io = __shfl_xor_sync(0xffffffffu, ix, off);
    merge_tri(m, s, ix, mo, so, io);
  }
  if (lane == 0) {
    const bool bad = *reinterpret_cast<volatile uint32_t*>(err) != 0u;
    conf[row] = bad ? __int_as_float(0x7fc00000) : 1.0f / s;
    argmax[row] = bad ? -1 : ix;
  }
}

__global__ void clear_static_err_kernel(uint32_t* err) { *err = 0u; }

typedef CUresult (*EncodeFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                             const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                             const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                             CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

struct DeviceSetup {
  bool ready = false;
  float4* part = nullptr;
  uint32_t* err = nullptr;
  int sms = 0;
};
std::mutex g_setup_mutex;
DeviceSetup g_setup[kStaticMaxDevices];
EncodeFn g_encode = nullptr;

// Once per device, with that device current: the device addresses of the
// static scratch (a host-side name of a __device__ array is not a device
// address), the shared-memory opt-in of the LM-head variant, the SM count.
int setup_device(int dev, DeviceSetup** out) {
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  DeviceSetup& d = g_setup[dev];
  if (!d.ready) {
    if (!g_encode) {
      void* fn = nullptr;
      cudaDriverEntryPointQueryResult q;
      if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                           cudaEnableDefault, &q) != cudaSuccess ||
          q != cudaDriverEntryPointSuccess)
        return CAI_ERR_CUDA;
      g_encode = reinterpret_cast<EncodeFn>(fn);
    }
    if (cudaGetSymbolAddress(reinterpret_cast<void**>(&d.part), g_static_part) != cudaSuccess ||
        cudaGetSymbolAddress(reinterpret_cast<void**>(&d.err), g_static_err) != cudaSuccess ||
        cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaFuncSetAttribute(lm_head_rows_static_kernel,
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(kStaticSmemBytes)) != cudaSuccess) {
      cudaGetLastError();
      return CAI_ERR_CUDA;
    }
    d.ready = true;
  }
  *out = &d;
  return CAI_OK;
}

bool encode(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBlockK), box_rows};
  cuuint32_t estr[2] = {1, 1};
  return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Whether p is device (or managed) memory of device dev: the TMA maps and the
// kernels' stores must never be pointed at host memory.
bool on_device(const void* p, int dev) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) && a.device == dev;
}

// Test hook: the next call makes its error word record a failed bounded wait
// before the merge (see cai_test_static_wait_timeout).
std::atomic<int> g_static_fail_next{0};

}  // namespace
}  // namespace cai

extern "C" int cai_head_rows_static(const void* W, int32_t V, int32_t H, const void* rows,
                                    int32_t M, float* conf, int32_t* argmax, void* stream) {
  using namespace cai;
  if (!W || !rows || !conf || !argmax) return CAI_ERR_ARG;
  if (M < 1 || M > kStaticMaxRows || V < 128 || H < 64 || H > 16384 || (H % 64) != 0)
    return CAI_ERR_SHAPE;
  if (reinterpret_cast<uintptr_t>(W) % 16 != 0 || reinterpret_cast<uintptr_t>(rows) % 16 != 0)
    return CAI_ERR_ARG;
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kStaticMaxDevices ||
      cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess) {
    cudaGetLastError();
    return CAI_ERR_CUDA;
  }
  if (major != 10 || minor != 3) return CAI_ERR_UNSUPPORTED;
  if (!on_device(W, dev) || !on_device(rows, dev) || !on_device(conf, dev) ||
      !on_device(argmax, dev))
    return CAI_ERR_ARG;
  DeviceSetup* d = nullptr;
  int r = setup_device(dev, &d);
  if (r != CAI_OK) return r;
  const int n_tiles = (V + kRowsPerTile - 1) / kRowsPerTile;
  int G = d->sms < kStaticMaxCtas ? d->sms : kStaticMaxCtas;
  if (G > n_tiles) G = n_tiles;
  CUtensorMap tm_w, tm_r;
  if (!encode(&tm_w, W, static_cast<uint64_t>(V), static_cast<uint64_t>(H), kRowsPerTile) ||
      !encode(&tm_r, rows, static_cast<uint64_t>(M), static_cast<uint64_t>(H), kBoxRowsB))
    return CAI_ERR_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // An error left pending by earlier, unrelated work is not this call's.
  cudaGetLastError();
  lm_head_rows_static_kernel<<<G, kHeadThreads, kStaticSmemBytes, s>>>(tm_w, tm_r, d->part, d->err,
                                                                       V, H, M, n_tiles);
  // If the LM head did not launch, the merge would read a previous call's partials.
  if (cudaGetLastError() != cudaSuccess) return CAI_ERR_CUDA;
  if (g_static_fail_next.exchange(0) != 0)
    wait_timeout_probe_kernel<<<1, 32, 0, s>>>(d->err, kErrWaitFull);
  merge_rows_static_kernel<<<(M + 7) / 8, 256, 0, s>>>(d->part, d->err, M, G, conf, argmax);
  clear_static_err_kernel<<<1, 1, 0, s>>>(d->err);
  if (cudaGetLastError() != cudaSuccess) return CAI_ERR_CUDA;
  return CAI_OK;
}

extern "C" int cai_test_static_wait_timeout(void) {
  cai::g_static_fail_next.store(1);
  return CAI_OK;
}
