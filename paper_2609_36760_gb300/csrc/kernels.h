// Internal launchers shared by the C ABI (api.cu) and the kernel files.
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "qmla.h"

namespace qmla {

// c_bits: 4 or 2 (this library's block) or kC4R4 (the paper's page).
cudaError_t launch_quant_append(void* pool, int c_bits, int num_blocks, const uint16_t* latent,
                                const uint16_t* k_pe, const int32_t* seq_ids,
                                const int32_t* positions, int n, const int32_t* table, int num_seqs,
                                int max_blocks, uint32_t* dev_err, cudaStream_t stream,
                                void* prot = nullptr, const int32_t* lens = nullptr);

cudaError_t launch_bf16_append(void* pool, int num_blocks, const uint16_t* latent,
                               const uint16_t* k_pe, const int32_t* seq_ids,
                               const int32_t* positions, int n, const int32_t* table, int num_seqs,
                               int max_blocks, uint32_t* dev_err, cudaStream_t stream);

// Heads handled by one CTA (the N of every MMA): 16, 32 or 64.
int head_group_size(int heads);

// Workspace carve-up of the decode path for `grid` CTAs.
struct DecodeWorkspace {
  size_t prefix_off, cta_off, part_o_off, part_ml_off, qimg_off, total;
};
DecodeWorkspace decode_workspace_layout(int batch, int heads, int grid);

struct DecodeArgs {
  const void* pool;
  int cache_kind;  // 4 or 2: packed content bits; kC4R4: the paper's page; 16: BF16 cache
  int num_blocks;
  const uint16_t* q_latent;
  const uint16_t* q_pe;
  int batch, heads;  // heads: all query rows of a sequence (q_tokens x heads per token)
  int q_tokens = 1;  // query tokens per sequence (the last q_tokens positions, causal among them)
  const int32_t* table;
  int max_blocks;
  const int32_t* seq_lens;
  float softmax_scale;
  float* out;
  float* lse;
  void* workspace;
  uint32_t* dev_err;
  int grid;  // CTAs of the main kernel (one per SM)
  const void* prot = nullptr;  // sink4/local128 protection buffer, or null
  cudaEvent_t ev_before_main = nullptr;  // optional, recorded around the main kernel
  cudaEvent_t ev_after_main = nullptr;
};
cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t stream);
// Test hook: tile j of sequence b as the decode kernel builds it, [128][576] fp16.
cudaError_t launch_tile_dump(const DecodeArgs& a, int b, int j, uint16_t* out, cudaStream_t stream);
// Test hook: a decode wait that runs out after limit_ns (see qmla_debug_wait_timeout).
cudaError_t launch_wait_timeout(uint32_t* dev_err, unsigned long long limit_ns, cudaStream_t stream);

// Records a failed CUDA call for qmla_last_cuda_error (calling thread).
void record_cuda_error(int err);
// The host checks of qmla_mla_decode_ex (no device access); the workspace
// fields are checked only with check_workspace.
int check_decode_desc(const qmla_decode_desc* d, bool check_workspace);

#ifdef QMLA_TRACE_BUILD
// Trace builds only: device buffer of [8 CTAs][96 events][32 tiles] u64 clock64 stamps.
cudaError_t set_trace_buffer(void* buf);
#endif

}  // namespace qmla
