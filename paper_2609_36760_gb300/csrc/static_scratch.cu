// qmla_mla_decode_static: the packed-cache decode without a caller-provided
// workspace, for callers that cannot allocate device memory at the point of
// the call (for example code running inside an allocator-free region of a
// serving loop, or a host library that is handed finished buffers and must
// not call cudaMalloc, whose synchronising behaviour and pool growth it does
// not control). The scratch the decode needs (tile plan, split partials and
// query images) lives in one fixed, file-scope device array instead.
//
// The array takes kStaticScratchBytes of device memory on every GPU that
// loads this library, for the life of the process. Its device address is
// looked up once per device (cudaGetSymbolAddress) the first time this entry
// point runs on that device.
#include <cuda_runtime.h>

#include <mutex>

#include "kernels.h"
#include "qmla.h"

namespace {

constexpr size_t kStaticScratchBytes = size_t(32) << 20;  // 32 MiB

static __device__ __align__(256) unsigned char g_decode_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_ptr[kMaxDevices] = {};
int g_scratch_sms[kMaxDevices] = {};

// Device address of g_decode_scratch on the current device (and its SM
// count); looked up once per device with that device current.
int scratch_for_current_device(void** ptr, int* sms, int* cuda_err) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    *cuda_err = static_cast<int>(e);
    return QMLA_ERR_CUDA;
  }
  if (dev < 0 || dev >= kMaxDevices) return QMLA_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    int major = 0, minor = 0, n = 0;
    if ((e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) {
      *cuda_err = static_cast<int>(e);
      return QMLA_ERR_CUDA;
    }
    if (!(major == 10 && minor == 3)) return QMLA_ERR_UNSUPPORTED;
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_decode_scratch);
    if (e != cudaSuccess || p == nullptr) {
      *cuda_err = static_cast<int>(e);
      return QMLA_ERR_CUDA;
    }
    g_scratch_ptr[dev] = p;
    g_scratch_sms[dev] = n;
  }
  *ptr = g_scratch_ptr[dev];
  *sms = g_scratch_sms[dev];
  return QMLA_OK;
}

bool aligned_to(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

}  // namespace

extern "C" {

size_t qmla_static_scratch_bytes(void) { return kStaticScratchBytes; }

int qmla_mla_decode_static(const void* pool_dev, int c_bits, int num_blocks, const uint16_t* q_latent_dev,
                           const uint16_t* q_pe_dev, int batch, int heads, const int32_t* block_table_dev,
                           int max_blocks, const int32_t* seq_lens_dev, float softmax_scale, float* out_dev,
                           float* lse_dev, uint32_t* dev_err_dev, qmla_stream_t stream) {
  if (c_bits != 4 && c_bits != 2) return QMLA_ERR_INVALID_ARG;
  if (pool_dev == nullptr || q_latent_dev == nullptr || q_pe_dev == nullptr || block_table_dev == nullptr ||
      seq_lens_dev == nullptr || out_dev == nullptr)
    return QMLA_ERR_INVALID_ARG;
  if (batch <= 0 || heads < 1 || heads > 128 || num_blocks <= 0 || max_blocks <= 0) return QMLA_ERR_INVALID_ARG;
  if (!(softmax_scale > 0.0f) || softmax_scale > 1e30f) return QMLA_ERR_INVALID_ARG;
  if (!aligned_to(pool_dev, 16) || !aligned_to(q_latent_dev, 16) || !aligned_to(q_pe_dev, 16) ||
      !aligned_to(block_table_dev, 4) || !aligned_to(seq_lens_dev, 4) || !aligned_to(out_dev, 16) ||
      (lse_dev != nullptr && !aligned_to(lse_dev, 4)))
    return QMLA_ERR_INVALID_ARG;
  if (static_cast<long long>(max_blocks) * 64 > 0x7fffffffLL) return QMLA_ERR_INVALID_ARG;
  void* scratch = nullptr;
  int sms = 0;
  int cuda_err = 0;
  const int st = scratch_for_current_device(&scratch, &sms, &cuda_err);
  if (st != QMLA_OK) {
    if (st == QMLA_ERR_CUDA) qmla::record_cuda_error(cuda_err);
    return st;
  }
  // The same layout the workspace of qmla_mla_decode uses; reject what does
  // not fit the fixed array.
  if (qmla::decode_workspace_layout(batch, heads, sms).total > kStaticScratchBytes) return QMLA_ERR_WORKSPACE_TOO_SMALL;
  qmla::DecodeArgs a;
  a.pool = pool_dev;
  a.cache_kind = c_bits;
  a.num_blocks = num_blocks;
  a.q_latent = q_latent_dev;
  a.q_pe = q_pe_dev;
  a.batch = batch;
  a.heads = heads;
  a.table = block_table_dev;
  a.max_blocks = max_blocks;
  a.seq_lens = seq_lens_dev;
  a.softmax_scale = softmax_scale;
  a.out = out_dev;
  a.lse = lse_dev;
  a.workspace = scratch;
  a.dev_err = dev_err_dev;
  a.grid = sms;
  const cudaError_t e = qmla::launch_decode(a, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) {
    qmla::record_cuda_error(static_cast<int>(e));
    return QMLA_ERR_CUDA;
  }
  return QMLA_OK;
}

}  // extern "C"
