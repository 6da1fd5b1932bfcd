// Host side of the C ABI declared in include/qmla.h: argument validation,
// device checks and kernel launches. Nothing here allocates device memory.
#include <cuda_runtime.h>

#include <cstdint>

#include "common.cuh"
#include "kernels.h"
#include "qmla.h"

namespace {

thread_local int g_last_cuda_error = 0;

int cuda_fail(cudaError_t e) {
  g_last_cuda_error = static_cast<int>(e);
  return QMLA_ERR_CUDA;
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

// SM count and architecture of each device, looked up once.
struct DevInfo {
  int sms = -1;
  bool supported = false;
};
DevInfo g_dev[64];

int current_device_info(DevInfo& out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e);
  if (dev < 0 || dev >= 64) return QMLA_ERR_UNSUPPORTED;
  if (g_dev[dev].sms < 0) {
    int major = 0, minor = 0, sms = 0;
    if ((e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev)) != cudaSuccess) return cuda_fail(e);
    if ((e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev)) != cudaSuccess) return cuda_fail(e);
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return cuda_fail(e);
    g_dev[dev].supported = (major == 10 && minor == 3);
    g_dev[dev].sms = sms;
  }
  out = g_dev[dev];
  return out.supported ? QMLA_OK : QMLA_ERR_UNSUPPORTED;
}

int append_common_checks(const void* pool, int num_blocks, const uint16_t* latent, const uint16_t* k_pe,
                         const int32_t* positions, int n, const int32_t* table, int num_seqs,
                         int max_blocks) {
  if (n < 0 || num_blocks <= 0 || num_seqs <= 0 || max_blocks <= 0) return QMLA_ERR_INVALID_ARG;
  if (n == 0) return QMLA_OK;
  if (pool == nullptr || latent == nullptr || k_pe == nullptr || positions == nullptr || table == nullptr)
    return QMLA_ERR_INVALID_ARG;
  if (!aligned(pool, 32) || !aligned(latent, 4) || !aligned(k_pe, 4) || !aligned(positions, 4) ||
      !aligned(table, 4))
    return QMLA_ERR_INVALID_ARG;
  if (static_cast<long long>(max_blocks) * qmla::kBlockTokens > INT32_MAX) return QMLA_ERR_INVALID_ARG;
  return QMLA_OK;
}

// Host checks of a decode call (no device access). heads counts every query
// row of a sequence (q_tokens x heads per token).
int decode_checks(const void* pool, int num_blocks, const uint16_t* q_latent, const uint16_t* q_pe, int batch,
                  int heads, const int32_t* table, int max_blocks, const int32_t* seq_lens, float softmax_scale,
                  const float* out, const float* lse, const void* workspace, const void* prot, int q_tokens,
                  bool need_workspace = true) {
  if (pool == nullptr || q_latent == nullptr || q_pe == nullptr || table == nullptr || seq_lens == nullptr ||
      out == nullptr || (need_workspace && workspace == nullptr))
    return QMLA_ERR_INVALID_ARG;
  if (prot != nullptr && !aligned(prot, 16)) return QMLA_ERR_INVALID_ARG;
  if (q_tokens < 1 || q_tokens > QMLA_MAX_Q_TOKENS || heads % q_tokens != 0) return QMLA_ERR_INVALID_ARG;
  if (batch <= 0 || heads < 1 || heads / q_tokens > 128 || num_blocks <= 0 || max_blocks <= 0)
    return QMLA_ERR_INVALID_ARG;
  if (!(softmax_scale > 0.0f) || softmax_scale > 1e30f) return QMLA_ERR_INVALID_ARG;
  if (!aligned(pool, 32) || !aligned(q_latent, 16) || !aligned(q_pe, 16) || !aligned(table, 4) ||
      !aligned(seq_lens, 4) || !aligned(out, 16) || (lse != nullptr && !aligned(lse, 4)) ||
      (need_workspace && !aligned(workspace, 256)))
    return QMLA_ERR_INVALID_ARG;
  if (static_cast<long long>(max_blocks) * qmla::kBlockTokens > INT32_MAX) return QMLA_ERR_INVALID_ARG;
  return QMLA_OK;
}

int decode_common(const void* pool, int kind, int num_blocks, const uint16_t* q_latent, const uint16_t* q_pe,
                  int batch, int heads, const int32_t* table, int max_blocks, const int32_t* seq_lens,
                  float softmax_scale, float* out, float* lse, void* workspace, size_t workspace_bytes,
                  uint32_t* dev_err, qmla_stream_t stream, const void* prot = nullptr, int q_tokens = 1,
                  void* ev_before_main = nullptr, void* ev_after_main = nullptr) {
  int st = decode_checks(pool, num_blocks, q_latent, q_pe, batch, heads, table, max_blocks, seq_lens, softmax_scale,
                         out, lse, workspace, prot, q_tokens);
  if (st != QMLA_OK) return st;
  DevInfo di;
  st = current_device_info(di);
  if (st != QMLA_OK) return st;
  const qmla::DecodeWorkspace w = qmla::decode_workspace_layout(batch, heads, di.sms);
  if (workspace_bytes < w.total) return QMLA_ERR_WORKSPACE_TOO_SMALL;
  qmla::DecodeArgs a;
  a.pool = pool;
  a.cache_kind = kind;
  a.num_blocks = num_blocks;
  a.q_latent = q_latent;
  a.q_pe = q_pe;
  a.batch = batch;
  a.heads = heads;
  a.table = table;
  a.max_blocks = max_blocks;
  a.seq_lens = seq_lens;
  a.softmax_scale = softmax_scale;
  a.out = out;
  a.lse = lse;
  a.workspace = workspace;
  a.dev_err = dev_err;
  a.grid = di.sms;
  a.prot = prot;
  a.q_tokens = q_tokens;
  a.ev_before_main = static_cast<cudaEvent_t>(ev_before_main);
  a.ev_after_main = static_cast<cudaEvent_t>(ev_after_main);
  cudaError_t e = qmla::launch_decode(a, reinterpret_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? QMLA_OK : cuda_fail(e);
}

// Descriptor-level checks of qmla_mla_decode_ex before the common ones.
int desc_checks(const qmla_decode_desc* d) {
  if (d == nullptr) return QMLA_ERR_INVALID_ARG;
  const int kind = d->cache_kind;
  if (kind != 4 && kind != 2 && kind != QMLA_CACHE_C4R4 && kind != QMLA_CACHE_BF16) return QMLA_ERR_INVALID_ARG;
  if (kind == QMLA_CACHE_BF16 && (d->prot != nullptr || d->q_tokens != 1)) return QMLA_ERR_INVALID_ARG;
  if (kind == QMLA_CACHE_C4R4 && d->q_tokens != 1) return QMLA_ERR_INVALID_ARG;
  if (d->q_tokens < 1 || d->q_tokens > QMLA_MAX_Q_TOKENS || d->heads < 1 || d->heads > 128)
    return QMLA_ERR_INVALID_ARG;
  return QMLA_OK;
}

}  // namespace

namespace qmla {
void record_cuda_error(int err) { g_last_cuda_error = err; }

int check_decode_desc(const qmla_decode_desc* d, bool check_workspace) {
  int st = desc_checks(d);
  if (st != QMLA_OK) return st;
  return decode_checks(d->pool, d->num_blocks, d->q_latent, d->q_pe, d->batch, d->q_tokens * d->heads,
                       d->block_table, d->max_blocks, d->seq_lens, d->softmax_scale, d->out, d->lse, d->workspace,
                       d->prot, d->q_tokens, check_workspace);
}
}  // namespace qmla

extern "C" {

size_t qmla_block_bytes(int c_bits) {
  if (c_bits == 4) return qmla::BlockLayout<4>::kBytes;
  if (c_bits == 2) return qmla::BlockLayout<2>::kBytes;
  return 0;
}

size_t qmla_bf16_block_bytes(void) { return qmla::kBf16BlockBytes; }

int qmla_quant_append(void* pool_dev, int c_bits, int num_blocks, const uint16_t* latent_dev,
                      const uint16_t* k_pe_dev, const int32_t* seq_ids_dev, const int32_t* positions_dev,
                      int n, const int32_t* block_table_dev, int num_seqs, int max_blocks,
                      uint32_t* dev_err_dev, qmla_stream_t stream) {
  if (c_bits != 4 && c_bits != 2) return QMLA_ERR_INVALID_ARG;
  int st = append_common_checks(pool_dev, num_blocks, latent_dev, k_pe_dev, positions_dev, n, block_table_dev,
                                num_seqs, max_blocks);
  if (st != QMLA_OK || n == 0) return st;
  DevInfo di;
  if ((st = current_device_info(di)) != QMLA_OK) return st;
  cudaError_t e = qmla::launch_quant_append(pool_dev, c_bits, num_blocks, latent_dev, k_pe_dev, seq_ids_dev,
                                            positions_dev, n, block_table_dev, num_seqs, max_blocks,
                                            dev_err_dev, reinterpret_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? QMLA_OK : cuda_fail(e);
}

size_t qmla_protect_bytes_per_seq(void) { return static_cast<size_t>(qmla::kProtRows) * qmla::kDqk * 2; }

int qmla_quant_append_protected(void* pool_dev, int c_bits, int num_blocks, const uint16_t* latent_dev,
                                const uint16_t* k_pe_dev, const int32_t* seq_ids_dev,
                                const int32_t* positions_dev, int n, const int32_t* block_table_dev,
                                int num_seqs, int max_blocks, const int32_t* seq_lens_dev, void* prot_dev,
                                uint32_t* dev_err_dev, qmla_stream_t stream) {
  if (c_bits != 4 && c_bits != 2) return QMLA_ERR_INVALID_ARG;
  int st = append_common_checks(pool_dev, num_blocks, latent_dev, k_pe_dev, positions_dev, n, block_table_dev,
                                num_seqs, max_blocks);
  if (st != QMLA_OK) return st;
  if (prot_dev == nullptr || seq_lens_dev == nullptr || !aligned(prot_dev, 16) || !aligned(seq_lens_dev, 4) ||
      !aligned(latent_dev, 16) || !aligned(k_pe_dev, 16))
    return QMLA_ERR_INVALID_ARG;
  if (n == 0) return QMLA_OK;
  DevInfo di;
  if ((st = current_device_info(di)) != QMLA_OK) return st;
  cudaError_t e = qmla::launch_quant_append(pool_dev, c_bits, num_blocks, latent_dev, k_pe_dev, seq_ids_dev,
                                            positions_dev, n, block_table_dev, num_seqs, max_blocks,
                                            dev_err_dev, reinterpret_cast<cudaStream_t>(stream), prot_dev,
                                            seq_lens_dev);
  return e == cudaSuccess ? QMLA_OK : cuda_fail(e);
}

int qmla_bf16_append(void* pool_dev, int num_blocks, const uint16_t* latent_dev, const uint16_t* k_pe_dev,
                     const int32_t* seq_ids_dev, const int32_t* positions_dev, int n,
                     const int32_t* block_table_dev, int num_seqs, int max_blocks, uint32_t* dev_err_dev,
                     qmla_stream_t stream) {
  int st = append_common_checks(pool_dev, num_blocks, latent_dev, k_pe_dev, positions_dev, n, block_table_dev,
                                num_seqs, max_blocks);
  if (st != QMLA_OK || n == 0) return st;
  DevInfo di;
  if ((st = current_device_info(di)) != QMLA_OK) return st;
  cudaError_t e = qmla::launch_bf16_append(pool_dev, num_blocks, latent_dev, k_pe_dev, seq_ids_dev, positions_dev,
                                           n, block_table_dev, num_seqs, max_blocks, dev_err_dev,
                                           reinterpret_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? QMLA_OK : cuda_fail(e);
}

size_t qmla_decode_workspace_bytes(int batch, int heads) {
  if (batch <= 0 || heads < 1 || heads > 128 * QMLA_MAX_Q_TOKENS) return 0;
  DevInfo di;
  if (current_device_info(di) != QMLA_OK) return 0;
  return qmla::decode_workspace_layout(batch, heads, di.sms).total;
}

int qmla_mla_decode(const void* pool_dev, int c_bits, int num_blocks, const uint16_t* q_latent_dev,
                    const uint16_t* q_pe_dev, int batch, int heads, const int32_t* block_table_dev, int max_blocks,
                    const int32_t* seq_lens_dev, float softmax_scale, float* out_dev, float* lse_dev,
                    void* workspace_dev, size_t workspace_bytes, uint32_t* dev_err_dev, qmla_stream_t stream) {
  if (c_bits != 4 && c_bits != 2) return QMLA_ERR_INVALID_ARG;
  return decode_common(pool_dev, c_bits, num_blocks, q_latent_dev, q_pe_dev, batch, heads, block_table_dev,
                       max_blocks, seq_lens_dev, softmax_scale, out_dev, lse_dev, workspace_dev, workspace_bytes,
                       dev_err_dev, stream);
}

int qmla_mla_decode_protected(const void* pool_dev, int c_bits, int num_blocks, const uint16_t* q_latent_dev,
                              const uint16_t* q_pe_dev, int batch, int heads, const int32_t* block_table_dev,
                              int max_blocks, const int32_t* seq_lens_dev, const void* prot_dev,
                              float softmax_scale, float* out_dev, float* lse_dev, void* workspace_dev,
                              size_t workspace_bytes, uint32_t* dev_err_dev, qmla_stream_t stream) {
  if (c_bits != 4 && c_bits != 2) return QMLA_ERR_INVALID_ARG;
  if (prot_dev == nullptr) return QMLA_ERR_INVALID_ARG;
  return decode_common(pool_dev, c_bits, num_blocks, q_latent_dev, q_pe_dev, batch, heads, block_table_dev,
                       max_blocks, seq_lens_dev, softmax_scale, out_dev, lse_dev, workspace_dev, workspace_bytes,
                       dev_err_dev, stream, prot_dev);
}

size_t qmla_c4r4_page_bytes(void) { return qmla::BlockLayout<qmla::kC4R4>::kBytes; }

int qmla_quant_append_c4r4(void* pool_dev, int num_blocks, const uint16_t* latent_dev, const uint16_t* k_pe_dev,
                           const int32_t* seq_ids_dev, const int32_t* positions_dev, int n,
                           const int32_t* block_table_dev, int num_seqs, int max_blocks,
                           const int32_t* seq_lens_dev, void* prot_dev, uint32_t* dev_err_dev,
                           qmla_stream_t stream) {
  int st = append_common_checks(pool_dev, num_blocks, latent_dev, k_pe_dev, positions_dev, n, block_table_dev,
                                num_seqs, max_blocks);
  if (st != QMLA_OK) return st;
  if (prot_dev != nullptr &&
      (seq_lens_dev == nullptr || !aligned(prot_dev, 16) || !aligned(seq_lens_dev, 4) ||
       !aligned(latent_dev, 16) || !aligned(k_pe_dev, 16)))
    return QMLA_ERR_INVALID_ARG;
  if (n == 0) return QMLA_OK;
  DevInfo di;
  if ((st = current_device_info(di)) != QMLA_OK) return st;
  cudaError_t e = qmla::launch_quant_append(pool_dev, qmla::kC4R4, num_blocks, latent_dev, k_pe_dev, seq_ids_dev,
                                            positions_dev, n, block_table_dev, num_seqs, max_blocks,
                                            dev_err_dev, reinterpret_cast<cudaStream_t>(stream), prot_dev,
                                            prot_dev != nullptr ? seq_lens_dev : nullptr);
  return e == cudaSuccess ? QMLA_OK : cuda_fail(e);
}

int qmla_mla_decode_c4r4(const void* pool_dev, int num_blocks, const uint16_t* q_latent_dev,
                         const uint16_t* q_pe_dev, int batch, int heads, const int32_t* block_table_dev,
                         int max_blocks, const int32_t* seq_lens_dev, const void* prot_dev, float softmax_scale,
                         float* out_dev, float* lse_dev, void* workspace_dev, size_t workspace_bytes,
                         uint32_t* dev_err_dev, qmla_stream_t stream) {
  return decode_common(pool_dev, qmla::kC4R4, num_blocks, q_latent_dev, q_pe_dev, batch, heads, block_table_dev,
                       max_blocks, seq_lens_dev, softmax_scale, out_dev, lse_dev, workspace_dev, workspace_bytes,
                       dev_err_dev, stream, prot_dev);
}

int qmla_mla_decode_multi(const void* pool_dev, int c_bits, int num_blocks, const uint16_t* q_latent_dev,
                          const uint16_t* q_pe_dev, int batch, int q_tokens, int heads,
                          const int32_t* block_table_dev, int max_blocks, const int32_t* seq_lens_dev,
                          const void* prot_dev, float softmax_scale, float* out_dev, float* lse_dev,
                          void* workspace_dev, size_t workspace_bytes, uint32_t* dev_err_dev, qmla_stream_t stream) {
  if (c_bits != 4 && c_bits != 2) return QMLA_ERR_INVALID_ARG;
  if (q_tokens < 1 || q_tokens > QMLA_MAX_Q_TOKENS || heads < 1 || heads > 128) return QMLA_ERR_INVALID_ARG;
  return decode_common(pool_dev, c_bits, num_blocks, q_latent_dev, q_pe_dev, batch, q_tokens * heads,
                       block_table_dev, max_blocks, seq_lens_dev, softmax_scale, out_dev, lse_dev, workspace_dev,
                       workspace_bytes, dev_err_dev, stream, prot_dev, q_tokens);
}

int qmla_mla_decode_bf16cache(const void* pool_dev, int num_blocks, const uint16_t* q_latent_dev,
                              const uint16_t* q_pe_dev, int batch, int heads, const int32_t* block_table_dev,
                              int max_blocks, const int32_t* seq_lens_dev, float softmax_scale, float* out_dev,
                              float* lse_dev, void* workspace_dev, size_t workspace_bytes, uint32_t* dev_err_dev,
                              qmla_stream_t stream) {
  return decode_common(pool_dev, 16, num_blocks, q_latent_dev, q_pe_dev, batch, heads, block_table_dev, max_blocks,
                       seq_lens_dev, softmax_scale, out_dev, lse_dev, workspace_dev, workspace_bytes, dev_err_dev,
                       stream);
}

int qmla_debug_tile(const void* pool_dev, int cache_kind, int num_blocks, const int32_t* block_table_dev,
                    int max_blocks, const int32_t* seq_lens_dev, int batch, int b, int j, const void* prot_dev,
                    uint16_t* tile_dev, uint32_t* dev_err_dev, qmla_stream_t stream) {
  static_assert(QMLA_CACHE_C4R4 == qmla::kC4R4, "kind code of the paper's page");
  if (cache_kind != 4 && cache_kind != 2 && cache_kind != QMLA_CACHE_C4R4 && cache_kind != QMLA_CACHE_BF16)
    return QMLA_ERR_INVALID_ARG;
  if (pool_dev == nullptr || block_table_dev == nullptr || seq_lens_dev == nullptr || tile_dev == nullptr)
    return QMLA_ERR_INVALID_ARG;
  if (num_blocks <= 0 || max_blocks <= 0 || batch <= 0 || b < 0 || b >= batch || j < 0 ||
      static_cast<long long>(j) * 2 >= max_blocks)
    return QMLA_ERR_INVALID_ARG;
  if (!aligned(pool_dev, 32) || !aligned(tile_dev, 16) || (prot_dev != nullptr && !aligned(prot_dev, 16)))
    return QMLA_ERR_INVALID_ARG;
  if (prot_dev != nullptr && cache_kind == QMLA_CACHE_BF16) return QMLA_ERR_INVALID_ARG;
  DevInfo di;
  int st = current_device_info(di);
  if (st != QMLA_OK) return st;
  qmla::DecodeArgs a;
  a.pool = pool_dev;
  a.cache_kind = cache_kind;
  a.num_blocks = num_blocks;
  a.batch = batch;
  a.table = block_table_dev;
  a.max_blocks = max_blocks;
  a.seq_lens = seq_lens_dev;
  a.dev_err = dev_err_dev;
  a.prot = prot_dev;
  cudaError_t e = qmla::launch_tile_dump(a, b, j, tile_dev, reinterpret_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? QMLA_OK : cuda_fail(e);
}

int qmla_debug_wait_timeout(uint32_t limit_us, uint32_t* dev_err_dev, qmla_stream_t stream) {
  if (dev_err_dev == nullptr || limit_us < 1u || limit_us > 1000000u) return QMLA_ERR_INVALID_ARG;
  DevInfo di;
  int st = current_device_info(di);
  if (st != QMLA_OK) return st;
  cudaError_t e = qmla::launch_wait_timeout(dev_err_dev, static_cast<unsigned long long>(limit_us) * 1000ull,
                                            reinterpret_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? QMLA_OK : cuda_fail(e);
}

int qmla_read_dev_err(const uint32_t* dev_err_dev, uint32_t* host_out, qmla_stream_t stream) {
  if (dev_err_dev == nullptr || host_out == nullptr) return QMLA_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemcpyAsync(host_out, dev_err_dev, sizeof(uint32_t), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  return e == cudaSuccess ? QMLA_OK : cuda_fail(e);
}

int qmla_mla_decode_ex(const qmla_decode_desc* d, qmla_stream_t stream) {
  const int st = desc_checks(d);
  if (st != QMLA_OK) return st;
  return decode_common(d->pool, d->cache_kind, d->num_blocks, d->q_latent, d->q_pe, d->batch, d->q_tokens * d->heads,
                       d->block_table, d->max_blocks, d->seq_lens, d->softmax_scale, d->out, d->lse, d->workspace,
                       d->workspace_bytes, d->dev_err, stream, d->prot, d->q_tokens, d->ev_before_main,
                       d->ev_after_main);
}

int qmla_last_cuda_error(void) { return g_last_cuda_error; }

#ifdef QMLA_TRACE_BUILD
// Trace builds only (libqmla_trace.so): device buffer that receives the
// decode kernel's per-CTA event timeline; NULL disables.
int qmla_trace_set(void* buf_dev) {
  cudaError_t e = qmla::set_trace_buffer(buf_dev);
  return e == cudaSuccess ? QMLA_OK : cuda_fail(e);
}
#endif

const char* qmla_status_string(int status) {
  switch (status) {
    case QMLA_OK: return "ok";
    case QMLA_ERR_INVALID_ARG: return "invalid argument";
    case QMLA_ERR_UNSUPPORTED: return "unsupported device or shape";
    case QMLA_ERR_WORKSPACE_TOO_SMALL: return "workspace too small";
    case QMLA_ERR_CUDA: return "CUDA error";
    default: return "unknown status";
  }
}

int qmla_num_sms(void) {
  DevInfo di;
  if (current_device_info(di) != QMLA_OK) return -1;
  return di.sms;
}

}  // extern "C"
