// Host-side plumbing shared by the library's translation units: status codes, the
// per-thread error message, the launch counter and CUDA error checks.
#pragma once
#include <cstdarg>
#include <cstdio>
#include <string>

#include <cuda_runtime.h>

#include "../../include/cachedsearch.h"
#include "../../include/cachedsearch_kernels.h"

namespace cs {

void set_error(const char* fmt, ...);
void count_launch(long long n = 1);
int num_sms();

}  // namespace cs

#define CS_REQUIRE(cond, ...)              \
  do {                                     \
    if (!(cond)) {                         \
      cs::set_error(__VA_ARGS__);          \
      return CS_ERR_ARG;                   \
    }                                      \
  } while (0)

#define CS_CUDA(expr)                                                                            \
  do {                                                                                           \
    cudaError_t e_ = (expr);                                                                     \
    if (e_ != cudaSuccess) {                                                                     \
      cs::set_error("%s failed: %s (%s:%d)", #expr, cudaGetErrorString(e_), __FILE__, __LINE__); \
      return CS_ERR_CUDA;                                                                        \
    }                                                                                            \
  } while (0)

// After a kernel launch: count it and surface launch-configuration errors.
#define CS_LAUNCHED()                                                                           \
  do {                                                                                          \
    cs::count_launch();                                                                         \
    cudaError_t e_ = cudaGetLastError();                                                        \
    if (e_ != cudaSuccess) {                                                                    \
      cs::set_error("kernel launch failed: %s (%s:%d)", cudaGetErrorString(e_), __FILE__, __LINE__); \
      return CS_ERR_CUDA;                                                                       \
    }                                                                                           \
  } while (0)

#define CS_TRY(expr)                 \
  do {                               \
    cs_status s_ = (expr);           \
    if (s_ != CS_OK) return s_;      \
  } while (0)
