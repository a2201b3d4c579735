// spade_common.cu -- status strings, last-error message, device check and
// tensor-map encoding shared by the entry points.
#include <cstdarg>
#include <cstdio>
#include <mutex>

#include "internal.h"
#include "ptx.cuh"

namespace spade {

static thread_local char g_last_error[512] = "";

spade_status fail(spade_status s, const char *fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_last_error, sizeof(g_last_error), fmt, ap);
  va_end(ap);
  return s;
}

spade_status cuda_fail(cudaError_t e, const char *what) {
  return fail(SPADE_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

namespace {
constexpr int kMaxDevices = 64;
struct DevInfo {
  int checked = 0;
  int ok = 0;
  int sms = 0;
  int major = 0, minor = 0;
};
DevInfo g_dev[kMaxDevices];
std::mutex g_dev_mu;
}  // namespace

spade_status device_info(int *num_sms, int *device) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return fail(SPADE_ERR_UNSUPPORTED_DEVICE, "device %d", dev);
  std::lock_guard<std::mutex> lk(g_dev_mu);
  DevInfo &d = g_dev[dev];
  if (!d.checked) {
    e = cudaDeviceGetAttribute(&d.major, cudaDevAttrComputeCapabilityMajor, dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&d.minor, cudaDevAttrComputeCapabilityMinor, dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
    d.ok = (d.major == 10 && d.minor == 3);
    d.checked = 1;
  }
  if (!d.ok)
    return fail(SPADE_ERR_UNSUPPORTED_DEVICE, "device %d is sm_%d%d; this library runs on sm_103 only",
                dev, d.major, d.minor);
  if (num_sms) *num_sms = d.sms;
  if (device) *device = dev;
  return SPADE_OK;
}

namespace {
using EncodeFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                              const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                              const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                              CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeFn g_encode = nullptr;
std::once_flag g_encode_once;
}  // namespace

bool encode_tmap_bf16_sw128(CUtensorMap *map, const void *base, uint64_t inner, uint64_t rows,
                            uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_rows) {
  std::call_once(g_encode_once, [] {
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<EncodeFn>(fn);
  });
  if (!g_encode) {
    fail(SPADE_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
    return false;
  }
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {row_stride_bytes};
  cuuint32_t box[2] = {box_inner, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    fail(SPADE_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d) for [%llu x %llu] box %u x %u",
         static_cast<int>(r), (unsigned long long)rows, (unsigned long long)inner, box_rows,
         box_inner);
    return false;
  }
  return true;
}

bool encode_tmap_rows_by_slab(CUtensorMap *map, const void *base, uint64_t rows, uint32_t cols,
                              uint32_t box_rows, uint32_t box_slabs) {
  std::call_once(g_encode_once, [] {
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<EncodeFn>(fn);
  });
  if (!g_encode) {
    fail(SPADE_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
    return false;
  }
  cuuint64_t dims[3] = {64, rows, cols / 64};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(cols) * 2, 128};
  cuuint32_t box[3] = {64, box_rows, box_slabs ? box_slabs : cols / 64};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    fail(SPADE_ERR_CUDA, "cuTensorMapEncodeTiled (row slabs) failed (%d) for [%llu x %u]",
         static_cast<int>(r), (unsigned long long)rows, cols);
    return false;
  }
  return true;
}

// One thread waits on an mbarrier that nothing completes, bounded as every
// kernel's waits are, and reports the expiry in the status word.
__global__ void selftest_wait_kernel(int32_t *status, uint64_t limit_ns) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
    const uint64_t t0 = globaltimer();
    bool done = mbar_try_wait(&bar, 0);
    while (!done && globaltimer() - t0 <= limit_ns) done = mbar_try_wait(&bar, 0);
    if (!done) atomicOr(status, SPADE_DEV_TIMEOUT);
  }
}

}  // namespace spade

extern "C" {

spade_status spade_selftest_wait_timeout(int32_t *status, int32_t limit_us, spade_stream_t stream) {
  using namespace spade;
  if (!status) return fail(SPADE_ERR_INVALID_ARG, "spade_selftest_wait_timeout: null status");
  if (limit_us < 1 || limit_us > 1000000)
    return fail(SPADE_ERR_INVALID_ARG, "spade_selftest_wait_timeout: limit %d us out of [1, 1000000]", limit_us);
  spade_status st = device_info(nullptr, nullptr);
  if (st != SPADE_OK) return st;
  selftest_wait_kernel<<<1, 32, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      status, static_cast<uint64_t>(limit_us) * 1000u);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "selftest launch");
  return SPADE_OK;
}

const char *spade_status_string(spade_status s) {
  switch (s) {
    case SPADE_OK: return "SPADE_OK";
    case SPADE_ERR_INVALID_ARG: return "SPADE_ERR_INVALID_ARG";
    case SPADE_ERR_SHAPE: return "SPADE_ERR_SHAPE";
    case SPADE_ERR_CAPACITY: return "SPADE_ERR_CAPACITY";
    case SPADE_ERR_UNSUPPORTED_DEVICE: return "SPADE_ERR_UNSUPPORTED_DEVICE";
    case SPADE_ERR_CUDA: return "SPADE_ERR_CUDA";
    case SPADE_ERR_WORKSPACE: return "SPADE_ERR_WORKSPACE";
  }
  return "SPADE_ERR_UNKNOWN";
}

const char *spade_last_error(void) { return spade::g_last_error; }

const char *spade_version(void) { return "spade-gb300 0.1 sm_103a"; }

}  // extern "C"
