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
// point runs on that device; the decode itself is qmla_mla_decode_ex with the
// array as its workspace.
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

// Device address of g_decode_scratch on the current device, looked up once
// per device with that device current.
int scratch_for_current_device(void** ptr, int* cuda_err) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    *cuda_err = static_cast<int>(e);
    return QMLA_ERR_CUDA;
  }
  if (dev < 0 || dev >= kMaxDevices) return QMLA_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_decode_scratch);
    if (e != cudaSuccess || p == nullptr) {
      *cuda_err = static_cast<int>(e);
      return QMLA_ERR_CUDA;
    }
    g_scratch_ptr[dev] = p;
  }
  *ptr = g_scratch_ptr[dev];
  return QMLA_OK;
}

}  // namespace

extern "C" {

size_t qmla_static_scratch_bytes(void) { return kStaticScratchBytes; }

int qmla_mla_decode_static(const void* pool_dev, int c_bits, int num_blocks, const uint16_t* q_latent_dev,
                           const uint16_t* q_pe_dev, int batch, int heads, const int32_t* block_table_dev,
                           int max_blocks, const int32_t* seq_lens_dev, float softmax_scale, float* out_dev,
                           float* lse_dev, uint32_t* dev_err_dev, qmla_stream_t stream) {
  if (c_bits != 4 && c_bits != 2) return QMLA_ERR_INVALID_ARG;
  // The workspace entry point with the fixed array as its workspace: the same
  // argument checks (run here first, before any device call), device lookup
  // and launches; a batch x heads whose workspace layout exceeds the array
  // gets QMLA_ERR_WORKSPACE_TOO_SMALL.
  qmla_decode_desc d{};
  d.pool = pool_dev;
  d.cache_kind = c_bits;
  d.num_blocks = num_blocks;
  d.q_latent = q_latent_dev;
  d.q_pe = q_pe_dev;
  d.batch = batch;
  d.q_tokens = 1;
  d.heads = heads;
  d.block_table = block_table_dev;
  d.max_blocks = max_blocks;
  d.seq_lens = seq_lens_dev;
  d.softmax_scale = softmax_scale;
  d.out = out_dev;
  d.lse = lse_dev;
  d.workspace_bytes = kStaticScratchBytes;
  d.dev_err = dev_err_dev;
  int st = qmla::check_decode_desc(&d, false);
  if (st != QMLA_OK) return st;
  void* scratch = nullptr;
  int cuda_err = 0;
  st = scratch_for_current_device(&scratch, &cuda_err);
  if (st != QMLA_OK) {
    if (st == QMLA_ERR_CUDA) qmla::record_cuda_error(cuda_err);
    return st;
  }
  d.workspace = scratch;
  return qmla_mla_decode_ex(&d, stream);
}

}  // extern "C"
