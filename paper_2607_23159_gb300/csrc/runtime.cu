// Library-wide host state: per-thread error message, launch counter, SM count and
// TMA tensor-map encoding (cuTensorMapEncodeTiled reached through the runtime's
// driver entry-point query, so the library needs no link against libcuda).
#include <atomic>
#include <cstring>
#include <mutex>

#include <cuda.h>

#include "common.cuh"
#include "ptx.cuh"
#include "tma_host.h"

namespace cs {

static thread_local std::string g_last_error;
static std::atomic<long long> g_launches{0};

void set_error(const char* fmt, ...) {
  char buf[1024];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_last_error = buf;
}

void count_launch(long long n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

int num_sms() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 1;
  return n > 0 ? n : 1;
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// bf16 tensor of `rank` dims (dims[0] innermost, contiguous), 128-byte swizzle.
cs_status make_tmap_bf16(CUtensorMap* map, const void* base, int rank, const uint64_t* dims,
                         const uint64_t* strides_bytes, const uint32_t* box) {
  return make_tmap(map, base, rank, dims, strides_bytes, box, false);
}

cs_status make_tmap(CUtensorMap* map, const void* base, int rank, const uint64_t* dims,
                    const uint64_t* strides_bytes, const uint32_t* box, bool f32) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) {
    set_error("cuTensorMapEncodeTiled is not available from the driver");
    return CS_ERR_CUDA;
  }
  if ((reinterpret_cast<uintptr_t>(base) & 15) != 0) {
    set_error("TMA base address %p is not 16-byte aligned", base);
    return CS_ERR_ARG;
  }
  cuuint64_t gd[5], gs[4];
  cuuint32_t bx[5], es[5];
  for (int i = 0; i < rank; ++i) {
    gd[i] = dims[i];
    bx[i] = box[i];
    es[i] = 1;
  }
  for (int i = 0; i + 1 < rank; ++i) {
    gs[i] = strides_bytes[i];
    if (gs[i] % 16 != 0) {
      set_error("TMA stride %llu bytes is not a multiple of 16", (unsigned long long)gs[i]);
      return CS_ERR_ARG;
    }
  }
  CUresult r = fn(map, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void*>(base), gd, gs, bx, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    set_error("cuTensorMapEncodeTiled failed (CUresult %d, rank %d, dims %llu x %llu, box %u x %u)", (int)r, rank,
              (unsigned long long)gd[0], (unsigned long long)(rank > 1 ? gd[1] : 1), bx[0], rank > 1 ? bx[1] : 1);
    return CS_ERR_CUDA;
  }
  return CS_OK;
}

// One thread waits on an mbarrier that nothing arrives on: the bounded wait that every
// kernel of this library uses gives up after CS_WAIT_TIMEOUT_NS and records the timeout
// in the device error word, and the kernel returns normally.
__global__ void bounded_wait_selftest_kernel(int* err) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  block_sync();
  if (threadIdx.x == 0) mbar_wait(&bar, 0, &abort_flag, err);   // phase 0 never completes
}

}  // namespace cs

extern "C" cs_status cs_selftest_bounded_wait(int* err_dev, cudaStream_t stream) {
  CS_REQUIRE(err_dev, "cs_selftest_bounded_wait: null error word");
  cs::bounded_wait_selftest_kernel<<<1, 32, 0, stream>>>(err_dev);
  CS_LAUNCHED();
  return CS_OK;
}

extern "C" const char* cs_last_error(void) { return cs::g_last_error.c_str(); }
extern "C" const char* cs_version(void) { return "cachedsearch-gb300 0.1 (sm_103a)"; }

extern "C" int cs_build_flags(void) {
#ifdef CS_DEBUG_CHECKS
  return 1;
#else
  return 0;
#endif
}
extern "C" long long cs_launch_count(void) { return cs::g_launches.load(); }
