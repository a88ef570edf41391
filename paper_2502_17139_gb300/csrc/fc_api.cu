// Library-wide entry points: status names, version, device error word.
#include "fc_common.cuh"

extern "C" unsigned int fc_take_error_sa(cudaStream_t s);
extern "C" unsigned int fc_take_error_ret(cudaStream_t s);
extern "C" unsigned int fc_take_error_tree(cudaStream_t s);
extern "C" unsigned int fc_take_error_step(cudaStream_t s);
extern "C" unsigned int fc_take_error_attn(cudaStream_t s);
extern "C" unsigned int fc_take_error_cache(cudaStream_t s);
extern "C" unsigned int fc_take_error_dec(cudaStream_t s);
extern "C" unsigned int fc_take_error_gemm(cudaStream_t s);

namespace {
thread_local unsigned int* t_error_slot = nullptr;
}

unsigned int* fc_error_slot() { return t_error_slot; }

FcErrorScope::FcErrorScope(unsigned int* word) : prev(t_error_slot) { t_error_slot = word; }

FcErrorScope::~FcErrorScope() { t_error_slot = prev; }

extern "C" const char* fc_status_string(fc_status s) {
  switch (s) {
    case FC_OK: return "FC_OK";
    case FC_ERR_INVALID_ARG: return "FC_ERR_INVALID_ARG";
    case FC_ERR_UNSUPPORTED: return "FC_ERR_UNSUPPORTED";
    case FC_ERR_WORKSPACE: return "FC_ERR_WORKSPACE";
    case FC_ERR_CAPACITY: return "FC_ERR_CAPACITY";
    case FC_ERR_TIMEOUT: return "FC_ERR_TIMEOUT";
    case FC_ERR_CUDA: return "FC_ERR_CUDA";
    case FC_ERR_INTERNAL: return "FC_ERR_INTERNAL";
    case FC_ERR_IO: return "FC_ERR_IO";
  }
  return "FC_ERR_UNKNOWN";
}

extern "C" const char* fc_version(void) { return "0.1.0"; }

extern "C" fc_status fc_get_error(fc_stream stream) {
  FC_NVTX_RANGE();
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) return FC_ERR_CUDA;
  unsigned int e = fc_take_error_sa(s) | fc_take_error_ret(s) | fc_take_error_tree(s) | fc_take_error_step(s) |
                   fc_take_error_attn(s) | fc_take_error_cache(s) |
                   fc_take_error_dec(s) | fc_take_error_gemm(s);
  return fc_status_of_bits(e);
}
