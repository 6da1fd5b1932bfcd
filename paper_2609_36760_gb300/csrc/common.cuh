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
static_assert(BlockLayout<4>::kBytes == 20736, "INT4 block size");
static_assert(BlockLayout<2>::kBytes == 12544, "INT2 block size");
constexpr int kBf16BlockBytes = kBlockTokens * kDqk * 2;  // 73728

__device__ __forceinline__ void report(uint32_t* dev_err, uint32_t bits) {
  if (dev_err != nullptr) atomicOr(dev_err, bits);
}

}  // namespace qmla
