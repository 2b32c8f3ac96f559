// Host-side helpers of the C ABI: error messages, device error word, limits.
#include <cstdarg>
#include <cstdio>
#include <cstring>

#include "common.cuh"

namespace om {

int read_clear_err_route(unsigned long long* out);
int read_clear_err_dispatch(unsigned long long* out);
int read_clear_err_gemm(unsigned long long* out);
int read_clear_err_sim(unsigned long long* out);
int read_clear_err_cost(unsigned long long* out);
int read_clear_err_simtc(unsigned long long* out);
int selftest_wait_timeout(uint64_t limit_ns, cudaStream_t stream);

static thread_local char t_msg[512] = "";
static thread_local uint64_t t_wait_limit_ns = 2000000000ull;

int fail(int code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(t_msg, sizeof t_msg, fmt, ap);
  va_end(ap);
  return code;
}

int cuda_fail(cudaError_t e, const char* what) {
  return fail(ORDERMOE_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorString(e), cudaGetErrorName(e));
}

uint64_t wait_limit_ns() { return t_wait_limit_ns; }

int num_sms() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
    return 1;
  return n;
}

}  // namespace om

using namespace om;

extern "C" const char* ordermoe_last_error(void) { return t_msg; }

extern "C" int ordermoe_version(void) { return 100; }

extern "C" int ordermoe_set_wait_limit_ns(uint64_t limit_ns) {
  if (limit_ns == 0) return fail(ORDERMOE_ERR_INVALID_ARG, "set_wait_limit_ns: limit must be > 0");
  t_wait_limit_ns = limit_ns;
  return ORDERMOE_OK;
}

extern "C" int ordermoe_device_error(int* code, int* detail) {
  OM_TRACE();
  if (!code) return fail(ORDERMOE_ERR_INVALID_ARG, "device_error: null code");
  OM_CUDA(cudaDeviceSynchronize());
  unsigned long long words[6] = {0, 0, 0, 0, 0, 0};
  int rc;
  if ((rc = read_clear_err_route(&words[0]))) return rc;
  if ((rc = read_clear_err_dispatch(&words[1]))) return rc;
  if ((rc = read_clear_err_gemm(&words[2]))) return rc;
  if ((rc = read_clear_err_sim(&words[3]))) return rc;
  if ((rc = read_clear_err_cost(&words[4]))) return rc;
  if ((rc = read_clear_err_simtc(&words[5]))) return rc;
  *code = 0;
  if (detail) *detail = 0;
  for (unsigned long long w : words) {
    if (w != 0) {
      *code = static_cast<int>(w & 0xFFFFFFFFull);
      if (detail) *detail = static_cast<int>(w >> 32);
      return fail(ORDERMOE_ERR_DEVICE_CHECK, "device error %d (detail %d)", *code,
                  static_cast<int>(w >> 32));
    }
  }
  return ORDERMOE_OK;
}

extern "C" int ordermoe_selftest_wait_timeout(uint64_t limit_ns, ordermoe_stream_t stream) {
  OM_TRACE();
  if (limit_ns == 0 || limit_ns > 10000000000ull)
    return fail(ORDERMOE_ERR_INVALID_ARG, "selftest_wait_timeout: need 0 < limit <= 10 s");
  return selftest_wait_timeout(limit_ns, stream);
}
