// Quantise-and-pack cache writer (App. C.4 quantiser; App. C.5 cache update:
// content- and RoPE-cache quantisation, integer packing and slot-mapped page
// insertion) for this library's block and for the paper's own page, and the
// plain BF16 writer for the comparison cache.
//
// One warp per (token, group): the 9 groups of 64 coordinates of a token are
// quantised by 9 independent warps, so a decode step's few tokens are not a
// chain of 9 dependent reductions. Lane l holds coordinates 2l and 2l+1 of its
// group; the extrema come from warp reductions, every lane quantises its two
// values, and the packed code words are assembled with shuffles and stored by
// the lanes that own them.
#include <cuda_runtime.h>

#include "common.cuh"
#include "kernels.h"

namespace qmla {
namespace {

__device__ __forceinline__ float warp_min_f32(float v) {
  float r;
  asm volatile("redux.sync.min.f32 %0, %1, 0xffffffff;" : "=f"(r) : "f"(v));
  return r;
}
__device__ __forceinline__ float warp_max_f32(float v) {
  float r;
  asm volatile("redux.sync.max.f32 %0, %1, 0xffffffff;" : "=f"(r) : "f"(v));
  return r;
}

// Stored fp16 scale and integer zero point of one group (App. C.4 with the
// fp16 staging of include/qmla.h): s = RN_f16(RN_f32(max(d, 1e-8) / m)),
// clamped to [2^-24, 65504]; z = clip(rne(-x_min / s), 0, m).
__device__ __forceinline__ void group_scale(float xmin, float xmax, int m, float& s, float& z) {
  const float d = xmax - xmin;
  const float s32 = __fdiv_rn(fmaxf(d, 1e-8f), static_cast<float>(m));
  s = __half2float(__float2half_rn(s32));
  if (s == 0.0f) s = 5.9604644775390625e-08f;  // 2^-24, the smallest fp16 subnormal
  if (isinf(s)) s = 65504.0f;
  z = fminf(fmaxf(rintf(__fdiv_rn(-xmin, s)), 0.0f), static_cast<float>(m));
}

// Scales of the paper's page (App. C.4 with that format's staging): content
// s = RN_bf16(RN_f32(max(d, 1e-8) / 15)), RoPE s = RN_f32(max(d, 1e-8) / 15);
// z = clip(rne(-x_min / s), 0, 15) from an fp32 quotient. A bf16 scale and a
// bf16 input carry 8 significant bits each, so the fp32 quotients of the
// content path round to the same codes as exact arithmetic would.
__device__ __forceinline__ void paper_scale(float xmin, float xmax, bool content, float& s, float& z) {
  const float s32 = __fdiv_rn(fmaxf(xmax - xmin, 1e-8f), 15.0f);
  s = content ? __bfloat162float(__float2bfloat16_rn(s32)) : s32;
  z = fminf(fmaxf(rintf(__fdiv_rn(-xmin, s)), 0.0f), 15.0f);
}

__device__ __forceinline__ uint32_t quant_code(float x, float s, float z, int m) {
  // q = clip(rne(x / s + z), 0, m): z is added before rounding.
  return static_cast<uint32_t>(fminf(fmaxf(rintf(__fdiv_rn(x, s) + z), 0.0f), static_cast<float>(m)));
}

// Looks up and validates the destination of token i. Returns null (after
// recording the error) when the token cannot be written.
__device__ __forceinline__ uint8_t* token_block(uint8_t* pool, size_t block_bytes, int num_blocks,
                                                const int32_t* seq_ids, const int32_t* positions,
                                                int i, const int32_t* table, int num_seqs,
                                                int max_blocks, uint32_t* dev_err, int& slot) {
  const int seq = seq_ids != nullptr ? seq_ids[i] : i;
  const int pos = positions[i];
  if (seq < 0 || seq >= num_seqs) {
    report(dev_err, QMLA_DEVERR_BAD_SEQ);
    return nullptr;
  }
  if (pos < 0 || pos >= max_blocks * kBlockTokens) {
    report(dev_err, QMLA_DEVERR_BAD_POSITION);
    return nullptr;
  }
  const int blk = table[static_cast<size_t>(seq) * max_blocks + pos / kBlockTokens];
  if (blk < 0 || blk >= num_blocks) {
    report(dev_err, QMLA_DEVERR_BAD_BLOCK);
    return nullptr;
  }
  slot = pos % kBlockTokens;
  return pool + static_cast<size_t>(blk) * block_bytes;
}

// Sink/recent BF16 protection rows (App. C.5, "BF16 protection and cache
// lifecycle"): position p of a request whose length after this write is L goes
// to row p when p < 4 and to row 4 + p mod 128 when p >= L - 128. The warp
// copies the token's 576 bf16 values (1152 bytes) as 16-byte vectors.
__device__ __forceinline__ void protect_row(uint4* prot, const uint4* latent, const uint4* k_pe, int tok, int seq,
                                            int pos, int L, int lane) {
  uint4* base = prot + static_cast<size_t>(seq) * kProtRows * (kDqk * 2 / 16);
  const uint4* lat = latent + static_cast<size_t>(tok) * (kDc * 2 / 16);  // 64 vectors
  const uint4* kp = k_pe + static_cast<size_t>(tok) * (kDr * 2 / 16);     // 8 vectors
  const uint4 a = lat[lane], b = lat[32 + lane];
  const uint4 c = lane < 8 ? kp[lane] : make_uint4(0, 0, 0, 0);
#pragma unroll
  for (int which = 0; which < 2; ++which) {
    int row = -1;
    if (which == 0 && pos < kSinkTokens) row = pos;
    if (which == 1 && pos >= L - kRecentTokens) row = kSinkTokens + pos % kRecentTokens;
    if (row < 0) continue;
    uint4* dst = base + static_cast<size_t>(row) * (kDqk * 2 / 16);
    dst[lane] = a;
    dst[32 + lane] = b;
    if (lane < 8) dst[64 + lane] = c;
  }
}

// prot / lens: the protection buffer [num_seqs][132][576] bf16 and the
// requests' lengths after this write, or null for an unprotected cache.
// CB: content bits (4, 2) or kC4R4 for the paper's page (INT4 codes).
template <int CB>
__global__ void __launch_bounds__(256) quant_append_kernel(
    uint8_t* __restrict__ pool, int num_blocks, const __nv_bfloat162* __restrict__ latent,
    const __nv_bfloat162* __restrict__ k_pe, const int32_t* __restrict__ seq_ids,
    const int32_t* __restrict__ positions, int n, const int32_t* __restrict__ table, int num_seqs,
    int max_blocks, uint32_t* dev_err, uint4* __restrict__ prot, const int32_t* __restrict__ lens) {
  using L = BlockLayout<CB>;
  const long long wid = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (wid >= static_cast<long long>(n) * kGroups) return;
  const int tok = static_cast<int>(wid / kGroups);
  const int g = static_cast<int>(wid - static_cast<long long>(tok) * kGroups);
  // Quantise first: the group's loads and arithmetic do not wait for the
  // dependent seq_ids -> block-table lookup, which only the stores need.
  const int bits = g < 8 ? (CB == kC4R4 ? 4 : CB) : kPeBits;
  const int m = (1 << bits) - 1;
  const __nv_bfloat162 v = g < 8 ? latent[static_cast<size_t>(tok) * (kDc / 2) + g * 32 + lane]
                                 : k_pe[static_cast<size_t>(tok) * (kDr / 2) + lane];
  const float x0 = __low2float(v), x1 = __high2float(v);
  const float xmin = warp_min_f32(fminf(x0, x1));
  const float xmax = warp_max_f32(fmaxf(x0, x1));
  float s, z;
  if constexpr (CB == kC4R4) {
    paper_scale(xmin, xmax, g < 8, s, z);
  } else {
    group_scale(xmin, xmax, m, s, z);
  }
  const uint32_t code = quant_code(x0, s, z, m) | (quant_code(x1, s, z, m) << bits);
  // Lane l's 2*bits bits sit at bit offset 2*bits*l of the group's code string.
  const int lane_bits = 2 * bits;
  const int lanes_per_word = 32 / lane_bits;
  uint32_t word = code << ((lane % lanes_per_word) * lane_bits);
  for (int off = 1; off < lanes_per_word; off <<= 1) word |= __shfl_xor_sync(0xffffffffu, word, off);

  int slot = 0;
  // errors are reported once per token, by its group-0 warp
  uint8_t* blk = token_block(pool, L::kBytes, num_blocks, seq_ids, positions, tok, table, num_seqs,
                             max_blocks, lane == 0 && g == 0 ? dev_err : nullptr, slot);
  if (blk == nullptr) return;
  if (prot != nullptr && g == 0) {
    const int seq = seq_ids != nullptr ? seq_ids[tok] : tok;
    protect_row(prot, reinterpret_cast<const uint4*>(latent), reinterpret_cast<const uint4*>(k_pe), tok, seq,
                positions[tok], lens[seq], lane);
  }
  if (lane % lanes_per_word == 0) {
    reinterpret_cast<uint32_t*>(blk + L::code_off(g, slot))[lane / lanes_per_word] = word;
  }
  if (lane == 0) {
    if constexpr (CB == kC4R4) {
      if (g < 8) {
        *reinterpret_cast<__nv_bfloat16*>(blk + L::c_scale_off(g, slot)) = __float2bfloat16_rn(s);  // exact
      } else {
        *reinterpret_cast<float*>(blk + L::pe_scale_off(slot)) = s;
      }
      blk[L::zero_off(g, slot)] = static_cast<uint8_t>(z);
    } else {
      *reinterpret_cast<__half2*>(blk + L::sz_off(g, slot)) = __halves2half2(__float2half_rn(s), __float2half_rn(z));
    }
  }
}

__global__ void __launch_bounds__(256) bf16_append_kernel(
    uint8_t* __restrict__ pool, int num_blocks, const uint32_t* __restrict__ latent,
    const uint32_t* __restrict__ k_pe, const int32_t* __restrict__ seq_ids,
    const int32_t* __restrict__ positions, int n, const int32_t* __restrict__ table, int num_seqs,
    int max_blocks, uint32_t* dev_err) {
  const int tok = static_cast<int>((blockIdx.x * blockDim.x + threadIdx.x) >> 5);
  const int lane = threadIdx.x & 31;
  if (tok >= n) return;
  int slot = 0;
  uint8_t* blk = token_block(pool, kBf16BlockBytes, num_blocks, seq_ids, positions, tok, table,
                             num_seqs, max_blocks, lane == 0 ? dev_err : nullptr, slot);
  if (blk == nullptr) return;
  uint32_t* dst = reinterpret_cast<uint32_t*>(blk + slot * kDqk * 2);
  for (int w = lane; w < kDc / 2; w += 32) dst[w] = latent[static_cast<size_t>(tok) * (kDc / 2) + w];
  dst[kDc / 2 + lane] = k_pe[static_cast<size_t>(tok) * (kDr / 2) + lane];
}

}  // namespace

cudaError_t launch_quant_append(void* pool, int c_bits, int num_blocks, const uint16_t* latent,
                                const uint16_t* k_pe, const int32_t* seq_ids,
                                const int32_t* positions, int n, const int32_t* table, int num_seqs,
                                int max_blocks, uint32_t* dev_err, cudaStream_t stream, void* prot,
                                const int32_t* lens) {
  if (n == 0) return cudaSuccess;
  const dim3 block(256);
  const dim3 grid(static_cast<unsigned>((static_cast<long long>(n) * kGroups * 32 + 255) / 256));
  auto* lat = reinterpret_cast<const __nv_bfloat162*>(latent);
  auto* kp = reinterpret_cast<const __nv_bfloat162*>(k_pe);
  if (c_bits == kC4R4) {
    quant_append_kernel<kC4R4><<<grid, block, 0, stream>>>(static_cast<uint8_t*>(pool), num_blocks, lat,
                                                           kp, seq_ids, positions, n, table, num_seqs,
                                                           max_blocks, dev_err, static_cast<uint4*>(prot), lens);
  } else if (c_bits == 4) {
    quant_append_kernel<4><<<grid, block, 0, stream>>>(static_cast<uint8_t*>(pool), num_blocks, lat,
                                                       kp, seq_ids, positions, n, table, num_seqs,
                                                       max_blocks, dev_err, static_cast<uint4*>(prot), lens);
  } else {
    quant_append_kernel<2><<<grid, block, 0, stream>>>(static_cast<uint8_t*>(pool), num_blocks, lat,
                                                       kp, seq_ids, positions, n, table, num_seqs,
                                                       max_blocks, dev_err, static_cast<uint4*>(prot), lens);
  }
  return cudaGetLastError();
}

cudaError_t launch_bf16_append(void* pool, int num_blocks, const uint16_t* latent,
                               const uint16_t* k_pe, const int32_t* seq_ids,
                               const int32_t* positions, int n, const int32_t* table, int num_seqs,
                               int max_blocks, uint32_t* dev_err, cudaStream_t stream) {
  if (n == 0) return cudaSuccess;
  const dim3 block(256);
  const dim3 grid(static_cast<unsigned>((static_cast<long long>(n) * 32 + 255) / 256));
  bf16_append_kernel<<<grid, block, 0, stream>>>(
      static_cast<uint8_t*>(pool), num_blocks, reinterpret_cast<const uint32_t*>(latent),
      reinterpret_cast<const uint32_t*>(k_pe), seq_ids, positions, n, table, num_seqs, max_blocks,
      dev_err);
  return cudaGetLastError();
}

}  // namespace qmla
