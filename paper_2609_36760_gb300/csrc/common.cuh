// Shared device-side constants of the packed cache block and error reporting.
#pragma once
#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "qmla.h"

namespace qmla {

constexpr int kDc = 512;           // content latent width d_c
constexpr int kDr = 64;            // RoPE key width d_r
constexpr int kDqk = kDc + kDr;    // 576 channels take part in QK
constexpr int kGroup = 64;         // quantisation group (App. C.4)
constexpr int kGroups = 9;         // 8 content groups + 1 RoPE-key group
constexpr int kBlockTokens = 64;   // tokens per cache block (page)
constexpr int kPeBits = 4;         // RoPE key bit width
// sink4/local128 protection buffer: rows 0..3 sink positions, 4 + p mod 128 recent p.
constexpr int kSinkTokens = 4;
constexpr int kRecentTokens = 128;
constexpr int kProtRows = kSinkTokens + kRecentTokens;

// Block layout for content bit width CB (see include/qmla.h).
template <int CB>
struct BlockLayout {
  static constexpr int kCodeBytes = kGroup * CB / 8;                    // per token and group
  static constexpr int kPeCodesOff = 8 * kBlockTokens * kCodeBytes;     // RoPE-key codes
  static constexpr int kSzOff = kPeCodesOff + kBlockTokens * 32;        // scale/zero pairs
  static constexpr int kBytes = kSzOff + kGroups * kBlockTokens * 4;
  __host__ __device__ static constexpr int code_off(int g, int slot) {
    return g < 8 ? g * kBlockTokens * kCodeBytes + slot * kCodeBytes : kPeCodesOff + slot * 32;
  }
  __host__ __device__ static constexpr int sz_off(int g, int slot) {
    return kSzOff + (g * kBlockTokens + slot) * 4;
  }
};
// Cache kind of the paper's own INT4 page (App. C.5 storage layout; App. C.4:
// BF16 content scales, FP32 RoPE scale). A kind code, not a bit width.
constexpr int kC4R4 = 5;

// The paper's page: the same code regions as BlockLayout<4>, then bf16 content
// scales [8][64], fp32 RoPE scales [64], uint8 zero points [9][64] (group 8 is
// the RoPE key) and 192 bytes of padding to 20,480 bytes (320 per token).
template <>
struct BlockLayout<kC4R4> {
  static constexpr int kCodeBytes = 32;
  static constexpr int kPeCodesOff = 8 * kBlockTokens * kCodeBytes;   // 16384
  static constexpr int kCScaleOff = kPeCodesOff + kBlockTokens * 32;  // 18432
  static constexpr int kPeScaleOff = kCScaleOff + 8 * kBlockTokens * 2;  // 19456
  static constexpr int kZeroOff = kPeScaleOff + kBlockTokens * 4;        // 19712
  static constexpr int kBytes = 20480;
  __host__ __device__ static constexpr int code_off(int g, int slot) {
    return g < 8 ? g * kBlockTokens * kCodeBytes + slot * kCodeBytes : kPeCodesOff + slot * 32;
  }
  __host__ __device__ static constexpr int c_scale_off(int g, int slot) { return kCScaleOff + (g * kBlockTokens + slot) * 2; }
  __host__ __device__ static constexpr int pe_scale_off(int slot) { return kPeScaleOff + slot * 4; }
  __host__ __device__ static constexpr int zero_off(int g, int slot) { return kZeroOff + g * kBlockTokens + slot; }
};
static_assert(BlockLayout<kC4R4>::kZeroOff + kGroups * kBlockTokens <= BlockLayout<kC4R4>::kBytes, "C4R4 page");
static_assert(BlockLayout<4>::kBytes == 20736, "INT4 block size");
static_assert(BlockLayout<2>::kBytes == 12544, "INT2 block size");
constexpr int kBf16BlockBytes = kBlockTokens * kDqk * 2;  // 73728

__device__ __forceinline__ void report(uint32_t* dev_err, uint32_t bits) {
  if (dev_err != nullptr) atomicOr(dev_err, bits);
}

}  // namespace qmla
