// Split-KV MLA decode over the low-bit paged cache (Eq. mla_compact; App. C.5
// "cache update and tile reuse" and "global attention normalization").
//
// Three kernels run per decode call:
//   prep_kernel    block 0: per-sequence tile counts -> prefix over (sequence,
//                  head group) units; the flattened tile list is cut into one
//                  equal range per SM ("metadata construction", App. F.1).
//                  Other blocks: query preparation, bf16 -> fp16 in the exact
//                  swizzled shared-memory image the MMA reads, one image per
//                  unit, later copied into each CTA by the bulk-copy engine.
//   decode_main    one persistent CTA per SM walks its tile range. A tile is 128
//                  cached tokens (two 64-token blocks) for one head group of HG
//                  heads. Per tile:
//                    dequant warps  gather packed codes + fp16 (s, z) from global
//                                   memory (prefetched a tile ahead), unpack and
//                                   dequantise RN_f16(s (q - z)) into nine
//                                   swizzled fp16 chunks of 128 tokens x 64
//                                   channels in shared memory;
//                    MMA issuers    S^T[t,h] = C_hat[t,:] . q[h,:] over 576
//                                   channels (tcgen05, M=128 tokens, N=HG,
//                                   K-major A and B) into TMEM;
//                    softmax warps  read S^T from TMEM (one token per thread),
//                                   keep a per-head reference max (rescaling O
//                                   only when a score exceeds it by 2^8), write
//                                   P^T = 2^(S*scale*log2e - m) as fp16;
//                    MMA issuers    O^T[c,h] += C_hat[:,c]^T P^T (M = 128
//                                   channels x 4, N=HG, K = 128 tokens; the same
//                                   shared-memory chunks read MN-major).
//                  The reconstructed content tile serves both QK and PV and a
//                  chunk is overwritten only after the PV that reads it commits.
//                  At a segment end the softmax warps write the final output, or
//                  an unnormalised partial (m, l, o) when the unit is split.
//   combine_kernel merges the partials of split units with
//                  m = max m_j, l = sum e^(m_j - m) l_j, O = sum e^(m_j - m) o_j / l
//                  (combine_wide_kernel for a few long units).
#include <cuda_runtime.h>

#include <cstddef>

#include "common.cuh"
#include "kernels.h"
#include "ptx.cuh"

namespace qmla {
namespace {

constexpr int kTileTokens = 128;                 // tokens per tile (M of QK)
constexpr int kChunkBytes = kTileTokens * 128;   // 128 tokens x 64 fp16 channels
constexpr int kNumChunks = 9;                    // 8 content chunks + RoPE-key chunk
constexpr int kWorkers = 8;                      // warps 0..7: dequantise, softmax, epilogue
// Warps 8..11 each keep one thread that issues MMAs, one per SM sub-partition
// (warp w runs on sub-partition w mod 4). A tcgen05.mma occupies its issuing
// thread until the tensor core takes it, so a single issuer stalls the tensor
// pipe whenever the scheduler of its sub-partition serves the busy worker
// warps there; four issuers with their own accumulators keep it fed.
constexpr int kIssuers = 4;
constexpr int kThreads = (kWorkers + kIssuers) * 32;  // 384
// S^T is accumulated in kQkParts partial sums, issuer j (< kQkParts) taking
// the K-steps kk = j mod kQkParts of every chunk; the softmax adds them.
constexpr int kQkParts = 2;
static_assert(4 % kQkParts == 0 && kQkParts <= kIssuers, "QK split");
constexpr uint64_t kWaitNs = 2000000000ull;      // bound of every on-chip wait (2 s)
constexpr float kRescaleLog2 = 8.0f;             // rescale O only above 2^8 growth
constexpr float kLn2 = 0.6931471805599453f;

// Optional per-CTA timeline (clock64 at pipeline events), compiled in only
// for trace builds (-DQMLA_TRACE_BUILD); see qmla_trace_set in api.cu.
#ifdef QMLA_TRACE_BUILD
constexpr int kTraceCtas = 8, kTraceEvents = 128, kTraceTiles = 32;
// The buffer pointer travels in the kernel parameters (constant bank), so an
// event costs one clock read and one global store, no load.
#define QMLA_TRACE(ev, tile)                                                                     \
  do {                                                                                           \
    if (p.trace != nullptr && blockIdx.x < kTraceCtas && (tile) < kTraceTiles)                   \
      p.trace[(static_cast<size_t>(blockIdx.x) * kTraceEvents + (ev)) * kTraceTiles + (tile)] = \
          clock64();                                                                             \
  } while (0)
// All CTAs: wall-clock start/end (%globaltimer), SM id and tile count after the event area.
#define QMLA_TRACE_CTA(slot, value)                                                                       \
  do {                                                                                                    \
    if (p.trace != nullptr)                                                                               \
      p.trace[static_cast<size_t>(kTraceCtas) * kTraceEvents * kTraceTiles + blockIdx.x * 4 + (slot)] = \
          (value);                                                                                        \
  } while (0)
#else
#define QMLA_TRACE(ev, tile) \
  do {                       \
  } while (0)
#define QMLA_TRACE_CTA(slot, value) \
  do {                              \
  } while (0)
#endif

struct Params {
  const uint8_t* pool;
  // sink4/local128 protection buffer [batch][132][576] bf16, or null (unprotected).
  const uint8_t* prot;
  int num_blocks;
  const __nv_bfloat16* q_lat;
  const __nv_bfloat16* q_pe;
  // heads = q_tokens * hpt "virtual heads" (query token t, head h) -> t * hpt + h;
  // one query token per sequence: q_tokens = 1, hpt = heads.
  int batch, heads, n_hg;
  int q_tokens, hpt;
  const int32_t* table;
  int max_blocks;
  const int32_t* seq_lens;
  float scale_log2;  // softmax_scale * log2(e)
  float* out;
  float* lse;
  const int32_t* prefix;
  int32_t* prefix_w;
  // [grid] per CTA, written by the prep kernel with the prefix: {unit of the first
  // tile, prefix[unit], prefix[unit + 1], total tiles} and, for the first tile,
  // {table entry of rows 0..63, of rows 64..127, sequence length, tile index}.
  int4* cta_info;
  int4* cta_first;
  int32_t* cta_t0;  // [grid + 1]: first tile of each CTA's range (cta_t0[grid] = total tiles)
  float* part_o;   // [(grid + units)][HG][512]
  float* part_ml;  // [(grid + units)][HG][2]
  uint8_t* qimg;   // [units][9][HG][128 B]: swizzled fp16 query tiles
  uint32_t* dev_err;
  int grid;
  unsigned long long* trace;  // trace builds only: per-CTA event clocks, else null
};

struct __align__(16) Ctrl {
  // chunk_full[k]: chunk k of the current tile is written (one arrive per warp of its parity).
  // pv_done: a tile's whole PV has completed (one commit per issuer, each its
  // 128-channel block): every chunk slot and the P tile are free and O^T holds
  // the sum through that tile.
  uint64_t chunk_full[kNumChunks];
  uint64_t pv_done;
  // rs_done: a tile's row-sum MMAs (issued after its PV, own commit) have completed.
  // s_full: every partial of S^T is complete (one commit per QK issuer).
  // p_full: every worker wrote its part of P (one arrive per warp). p_fixed: after a
  // rescale, P was rewritten against the raised reference.
  uint64_t rs_done, s_full, p_full, p_fixed, o_free, q_full, fin;
  uint64_t grp;  // barrier among the worker warps (one arrive per warp, reused in sequence)
  uint32_t tmem_base;
  uint32_t abort;
  uint32_t resc_tile;  // it + 1 when tile it needs a rescale (written before p_full)
  alignas(16) float m_ref[64];  // read as float4
  alignas(16) float alpha[64];
  alignas(16) float inv[64];  // 1 / l per head at a segment end, read as float4
  alignas(16) float red[4][64];
};
static_assert(offsetof(Ctrl, m_ref) % 16 == 0 && offsetof(Ctrl, alpha) % 16 == 0 && offsetof(Ctrl, inv) % 16 == 0,
              "float4 access alignment");
static_assert(sizeof(Ctrl) % 16 == 0, "Ctrl size");

template <int HG>
struct Cfg {
  static constexpr int kQBytes = kNumChunks * HG * 128;
  // O^T (4 HG columns), the kQkParts partials of S^T (HG each), the row sums
  // of P (HG) and the all-ones A operand of their MMAs (8), rounded up to a power of 2.
  static constexpr uint32_t kTmemCols = HG >= 64 ? 512 : (HG == 32 ? 256 : 128);
  static constexpr uint32_t kColL = (4 + kQkParts) * HG;
  static constexpr uint32_t kColOnes = kColL + HG;
  static_assert(HG > 64 || kColOnes + 8 <= kTmemCols, "TMEM columns");
  static constexpr int kSmem = 1024 + kNumChunks * kChunkBytes + kQBytes + (int)sizeof(Ctrl);
  static constexpr uint32_t kPRowBytes = 2 * HG;  // P^T tile row (one token, HG fp16)
};

// Channel order inside each 8-channel (16-byte) piece of a reconstructed row:
// the unpacking below yields nibble/crumb pairs in this order, and the query
// tile and the output mapping use the same permutation.
template <int CB>
struct Perm {
  // position p of a piece holds channel at(p): INT4 swaps bits 0 and 1 of p
  // ([0,2,1,3,4,6,5,7]); INT2 rotates them ([0,4,1,5,2,6,3,7]); BF16 keeps p.
  __host__ __device__ static constexpr int at(int p) {
    if constexpr (CB == 4 || CB == kC4R4) {
      return (p & 4) | ((p & 1) << 1) | ((p >> 1) & 1);
    } else if constexpr (CB == 2) {
      return ((p & 1) << 2) | (p >> 1);
    } else {
      return p;
    }
  }
};
static_assert(Perm<4>::at(1) == 2 && Perm<4>::at(2) == 1 && Perm<4>::at(5) == 6 && Perm<4>::at(7) == 7, "INT4 order");
static_assert(Perm<2>::at(1) == 4 && Perm<2>::at(2) == 1 && Perm<2>::at(6) == 3 && Perm<2>::at(7) == 7, "INT2 order");

// --------------------------------------------------------------- helpers
__device__ __forceinline__ uint4 ldg_nc_v4(const void* ptr) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(ptr));
  return r;
}
// 32 bytes in one request (the address is 32-byte aligned).
__device__ __forceinline__ void ldg_nc_v8(const void* ptr, uint4& a, uint4& b) {
  asm volatile("ld.global.nc.L1::no_allocate.v8.u32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=r"(a.x), "=r"(a.y), "=r"(a.z), "=r"(a.w), "=r"(b.x), "=r"(b.y), "=r"(b.z), "=r"(b.w)
               : "l"(ptr));
}
__device__ __forceinline__ uint32_t ldg_nc_u32(const void* ptr) {
  uint32_t r;
  asm volatile("ld.global.nc.L1::no_allocate.u32 %0, [%1];" : "=r"(r) : "l"(ptr));
  return r;
}
__device__ __forceinline__ uint32_t ldg_nc_u16(const void* ptr) {
  uint16_t r;
  asm volatile("ld.global.nc.L1::no_allocate.u16 %0, [%1];" : "=h"(r) : "l"(ptr));
  return r;
}
__device__ __forceinline__ uint32_t ldg_nc_u8(const void* ptr) {
  uint32_t r;
  asm volatile("ld.global.nc.L1::no_allocate.u8 %0, [%1];" : "=r"(r) : "l"(ptr));
  return r;
}
__device__ __forceinline__ void sts_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d)
               : "memory");
}
// RN_f16((x - zz) * s) per half: the subtraction of two integers below 2048 is
// exact, so this is a single rounding of s (q - z).
__device__ __forceinline__ uint32_t dq2(uint32_t x, uint32_t zz, uint32_t ss) {
  uint32_t t, r;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(t) : "r"(x), "r"(zz));
  asm("mul.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(t), "r"(ss));
  return r;
}
__device__ __forceinline__ uint32_t pack_h2(float lo, float hi) {
  const __half2 h = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ float warp_max_f32(float v) {
  float r;
  asm volatile("redux.sync.max.f32 %0, %1, 0xffffffff;" : "=f"(r) : "f"(v));
  return r;
}

// Wait sites, reported in bits 8.. of the error word when a wait runs out.
enum WaitSite : uint32_t {
  kSiteDqSlot = 0, kSiteMmaQFull, kSiteMmaChunk, kSiteMmaPFull, kSiteMmaOFree,
  kSiteSmSFull, kSiteGrp, kSitePvEpi, kSiteMmaFin
};

// Marks the CTA aborted; a wait that ran out (rather than saw the abort)
// also records its site.
__device__ __forceinline__ void set_abort(Ctrl& c, uint32_t* dev_err) {
  *reinterpret_cast<volatile uint32_t*>(&c.abort) = 1u;
  report(dev_err, QMLA_DEVERR_TIMEOUT);
}
__device__ __forceinline__ bool wait_ok(int r, uint32_t site, Ctrl& c, uint32_t* dev_err) {
  if (r == 0) {
    report(dev_err, QMLA_DEVERR_TIMEOUT | (0x100u << site));
    *reinterpret_cast<volatile uint32_t*>(&c.abort) = 1u;
  }
  return r == 1;
}
// Warp-uniform bounded wait: every lane waits on the barrier itself. Letting
// one lane poll while the others sit at a warp-synchronising instruction was
// measured to be much slower on sm_103a: the parked warp delayed the draining
// of other warps' shared-memory stores by thousands of cycles, and its own
// wake-up after the phase completed took ~2k cycles.
__device__ __forceinline__ bool wwait(uint64_t* bar, uint32_t parity, Ctrl& c, uint32_t site,
                                      uint32_t* dev_err, uint64_t limit_ns = kWaitNs) {
  const int r = mbar_wait(bar, parity, limit_ns, &c.abort);
  const bool all_ok = __all_sync(0xffffffffu, r == 1);
  if (r == 0) wait_ok(r, site, c, dev_err);
  return all_ok;
}
// Barrier among the worker warps (one arrive per warp), bounded. Every worker
// passes the same sequence of these, so one mbarrier serves them all: a warp
// cannot arrive for phase n + 2 before every warp has arrived for n + 1.
__device__ __forceinline__ bool group_sync(Ctrl& c, uint32_t& phase, uint32_t* dev_err) {
  __syncwarp();
  mbar_arrive_if((threadIdx.x & 31) == 0 ? 1u : 0u, &c.grp);
  const bool ok = wwait(&c.grp, phase & 1u, c, kSiteGrp, dev_err);
  ++phase;
  return ok;
}

// ------------------------------------------------------------- schedule
struct Sched {
  const int32_t* prefix;
  int t0, t1, t, u, pu0, pu1;
  int units;
  // info = {unit holding tile t0, prefix[unit], prefix[unit + 1], total tiles}
  // for this CTA (found once by the prep kernel).
  __device__ void init(const int32_t* pf, int4 info, int units_, int cta, int grid) {
    prefix = pf;
    units = units_;
    const int T = info.w;
    t0 = static_cast<int>(static_cast<long long>(cta) * T / grid);
    t1 = static_cast<int>(static_cast<long long>(cta + 1) * T / grid);
    t = t0;
    u = info.x;
    pu0 = info.y;
    pu1 = info.z;
  }
  __device__ bool valid() const { return t < t1; }
  __device__ void next() {
    ++t;
    while (t < t1 && t >= pu1 && u + 1 < units) {
      ++u;
      pu0 = pu1;
      pu1 = prefix[u + 1];
    }
  }
};

struct TileInfo {
  int b, hg, j, ntok, len;
  bool first, last;
};
// Segment position of the current tile, from the schedule alone (no loads).
struct TileFlags {
  bool first, last;
};
__device__ __forceinline__ TileFlags tile_flags(const Sched& s) {
  TileFlags f;
  f.first = (s.t == s.t0) || (s.t == s.pu0);
  f.last = (s.t + 1 == s.t1) || (s.t + 1 == s.pu1);
  return f;
}
__device__ __forceinline__ TileInfo tile_info(const Sched& s, const Params& p) {
  TileInfo ti;
  ti.b = s.u / p.n_hg;
  ti.hg = s.u - ti.b * p.n_hg;
  ti.j = s.t - s.pu0;
  ti.len = p.seq_lens[ti.b];
  ti.ntok = min(kTileTokens, ti.len - kTileTokens * ti.j);
  ti.first = (s.t == s.t0) || (ti.j == 0);
  ti.last = (s.t + 1 == s.t1) || (s.t + 1 == s.pu1);
  return ti;
}

// -------------------------------------------------------- dequant warps
// Packed data of one token row for one chunk, fetched ahead of use.
struct Fetch {
  uint4 a, b;
  uint32_t sz;  // fp16 (s, z) pair; for the paper's page the scale as fp32 bits
  uint32_t z;   // the paper's page: the uint8 zero point
  bool ok;
};

// Block-table entry and sequence length of one token row of a tile, loaded a
// tile before they are needed (nothing branches on them until resolve_row).
// The table column is clamped so that rows past the sequence end never read
// beyond the sequence's table row.
struct RowRef {
  int entry, len, j, b;
  bool has;
};
__device__ __forceinline__ RowRef row_ref(const Params& p, const Sched& s, int row) {
  RowRef r;
  r.has = s.valid();
  r.entry = -1;
  r.len = 0;
  r.j = 0;
  r.b = 0;
  if (!r.has) return r;
  const int b = s.u / p.n_hg;
  r.b = b;
  r.j = s.t - s.pu0;
  r.len = p.seq_lens[b];
  const int lb = min(2 * r.j + (row >> 6), p.max_blocks - 1);
  r.entry = p.table[static_cast<size_t>(b) * p.max_blocks + lb];
  return r;
}
template <int CB>
__device__ __forceinline__ const uint8_t* resolve_row(const Params& p, const RowRef& r, int row, bool& valid) {
  valid = false;
  if (!r.has || row >= min(kTileTokens, r.len - kTileTokens * r.j)) return nullptr;
  if (r.entry < 0 || r.entry >= p.num_blocks) {
    report(p.dev_err, QMLA_DEVERR_BAD_BLOCK);
    return nullptr;
  }
  valid = true;
  constexpr size_t kBlk = CB == 16 ? static_cast<size_t>(kBf16BlockBytes) : BlockLayout<CB == 16 ? 4 : CB>::kBytes;
  return p.pool + static_cast<size_t>(r.entry) * kBlk;
}

// The protection-buffer row a tile row attends with (App. C.5, "BF16
// protection and cache lifecycle": position p of a length-L request is
// protected iff p < min(4, L) or p >= L - 128), or null when the row is read
// from the packed cache. Sink positions read their sink row, which the writer
// always fills; recent ones the ring row 4 + p mod 128.
__device__ __forceinline__ const uint8_t* prot_row(const Params& p, const RowRef& r, int row) {
  if (p.prot == nullptr || !r.has) return nullptr;
  const int pos = kTileTokens * r.j + row;
  if (pos >= r.len) return nullptr;
  int pr;
  if (pos < kSinkTokens) {
    pr = pos;
  } else if (pos >= r.len - kRecentTokens) {
    pr = kSinkTokens + pos % kRecentTokens;
  } else {
    return nullptr;
  }
  return p.prot + (static_cast<size_t>(r.b) * kProtRows + pr) * (kDqk * 2);
}

template <int CB>
__device__ __forceinline__ Fetch fetch_chunk(const uint8_t* blk, bool valid, int k, int slot) {
  Fetch f;
  f.ok = valid;
  f.a = make_uint4(0, 0, 0, 0);
  f.b = f.a;
  f.sz = 0;
  f.z = 0;
  if (!valid) return f;
  using L = BlockLayout<CB>;
  const uint8_t* c = blk + L::code_off(k, slot);
  // a 32-byte code row in one request (half the requests of two 16-byte
  // loads, which made the next tile's fetch a quarter of the kernel's time)
  if (CB == 4 || CB == kC4R4 || k == 8) {
    ldg_nc_v8(c, f.a, f.b);
  } else {
    f.a = ldg_nc_v4(c);
  }
  if constexpr (CB == kC4R4) {
    // bf16 content scale -> fp32 bits by a 16-bit shift; the RoPE scale is fp32
    f.sz = k < 8 ? ldg_nc_u16(blk + L::c_scale_off(k, slot)) << 16 : ldg_nc_u32(blk + L::pe_scale_off(slot));
    f.z = ldg_nc_u8(blk + L::zero_off(k, slot));
  } else {
    f.sz = ldg_nc_u32(blk + L::sz_off(k, slot));
  }
  return f;
}

// Half h of a token row of the RoPE-key chunk (INT4 codes of channels 32 h ..
// 32 h + 31, bytes 16 h .. 16 h + 15): the two worker warps that share a row
// quarter split that chunk, so each dequantises 4.5 chunks per tile.
template <int CB>
__device__ __forceinline__ Fetch fetch_rope_half(const uint8_t* blk, bool valid, int slot, int h) {
  Fetch f;
  f.ok = valid;
  f.a = make_uint4(0, 0, 0, 0);
  f.b = f.a;
  f.sz = 0;
  f.z = 0;
  if (!valid) return f;
  using L = BlockLayout<CB>;
  f.a = ldg_nc_v4(blk + L::code_off(8, slot) + 16 * h);
  if constexpr (CB == kC4R4) {
    f.sz = ldg_nc_u32(blk + L::pe_scale_off(slot));  // the fp32 RoPE scale
    f.z = ldg_nc_u8(blk + L::zero_off(8, slot));
  } else {
    f.sz = ldg_nc_u32(blk + L::sz_off(8, slot));
  }
  return f;
}

// Unpacks one row (64 codes) of chunk k and stores RN_f16(s (q - z)) into the
// swizzled chunk tile. The code nibbles / crumbs are placed into the mantissa
// of 1024.0 (0x6400), giving 1024 + q exactly; subtracting 1024 + z is exact.
template <int CB>
__device__ __forceinline__ void store_row(uint32_t chunk_base, int row, const Fetch& f, bool int4) {
  if (!f.ok) {
#pragma unroll
    for (int i = 0; i < 8; ++i) sts_v4(chunk_base + swz_off(row, i, 128), 0, 0, 0, 0);
    return;
  }
  const __half2 sz = *reinterpret_cast<const __half2*>(&f.sz);
  const __half2 s2 = __half2half2(__low2half(sz));
  const __half2 zz2 = __half2half2(__hadd(__high2half(sz), __float2half_rn(1024.0f)));
  const uint32_t ss = *reinterpret_cast<const uint32_t*>(&s2);
  const uint32_t zz = *reinterpret_cast<const uint32_t*>(&zz2);
  constexpr uint32_t K = 0x64646464u;
  if (int4) {
    const uint32_t w[8] = {f.a.x, f.a.y, f.a.z, f.a.w, f.b.x, f.b.y, f.b.z, f.b.w};
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint32_t lo = w[i] & 0x0F0F0F0Fu;          // e0 e2 e4 e6
      const uint32_t hi = (w[i] >> 4) & 0x0F0F0F0Fu;   // e1 e3 e5 e7
      sts_v4(chunk_base + swz_off(row, i, 128), dq2(__byte_perm(lo, K, 0x4140), zz, ss),
             dq2(__byte_perm(hi, K, 0x4140), zz, ss), dq2(__byte_perm(lo, K, 0x4342), zz, ss),
             dq2(__byte_perm(hi, K, 0x4342), zz, ss));
    }
  } else {
    const uint32_t w[4] = {f.a.x, f.a.y, f.a.z, f.a.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const uint32_t c0 = w[i] & 0x03030303u;          // e0 e4 e8 e12
      const uint32_t c1 = (w[i] >> 2) & 0x03030303u;   // e1 e5 e9 e13
      const uint32_t c2 = (w[i] >> 4) & 0x03030303u;   // e2 e6 e10 e14
      const uint32_t c3 = (w[i] >> 6) & 0x03030303u;   // e3 e7 e11 e15
      sts_v4(chunk_base + swz_off(row, 2 * i, 128), dq2(__byte_perm(c0, K, 0x4140), zz, ss),
             dq2(__byte_perm(c1, K, 0x4140), zz, ss), dq2(__byte_perm(c2, K, 0x4140), zz, ss),
             dq2(__byte_perm(c3, K, 0x4140), zz, ss));
      sts_v4(chunk_base + swz_off(row, 2 * i + 1, 128), dq2(__byte_perm(c0, K, 0x4342), zz, ss),
             dq2(__byte_perm(c1, K, 0x4342), zz, ss), dq2(__byte_perm(c2, K, 0x4342), zz, ss),
             dq2(__byte_perm(c3, K, 0x4342), zz, ss));
    }
  }
}

// store_row split around the slot wait for the decode workers: dq_regs
// dequantises a packed row into registers before the wait, store_regs writes
// it into the swizzled chunk after it, so that only the stores remain between
// the slot's release and the chunk's arrival. Same arithmetic as store_row; a
// row that is not fetched (f.ok false) has zero codes, scale and zero point,
// so it dequantises to zeros without a branch.
__device__ __forceinline__ void dq_regs(uint32_t (&o)[32], const Fetch& f, bool int4) {
  const __half2 sz = *reinterpret_cast<const __half2*>(&f.sz);
  const __half2 s2 = __half2half2(__low2half(sz));
  const __half2 zz2 = __half2half2(__hadd(__high2half(sz), __float2half_rn(1024.0f)));
  const uint32_t ss = *reinterpret_cast<const uint32_t*>(&s2);
  const uint32_t zz = *reinterpret_cast<const uint32_t*>(&zz2);
  constexpr uint32_t K = 0x64646464u;
  const uint32_t w[8] = {f.a.x, f.a.y, f.a.z, f.a.w, f.b.x, f.b.y, f.b.z, f.b.w};
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    if (int4) {
      const uint32_t lo = w[i] & 0x0F0F0F0Fu;
      const uint32_t hi = (w[i] >> 4) & 0x0F0F0F0Fu;
      o[4 * i + 0] = dq2(__byte_perm(lo, K, 0x4140), zz, ss);
      o[4 * i + 1] = dq2(__byte_perm(hi, K, 0x4140), zz, ss);
      o[4 * i + 2] = dq2(__byte_perm(lo, K, 0x4342), zz, ss);
      o[4 * i + 3] = dq2(__byte_perm(hi, K, 0x4342), zz, ss);
    } else {  // INT2: pieces 2m and 2m + 1 come from word m
      const uint32_t x = w[i >> 1];
      const uint32_t sel = (i & 1) ? 0x4342u : 0x4140u;
      o[4 * i + 0] = dq2(__byte_perm(x & 0x03030303u, K, sel), zz, ss);
      o[4 * i + 1] = dq2(__byte_perm((x >> 2) & 0x03030303u, K, sel), zz, ss);
      o[4 * i + 2] = dq2(__byte_perm((x >> 4) & 0x03030303u, K, sel), zz, ss);
      o[4 * i + 3] = dq2(__byte_perm((x >> 6) & 0x03030303u, K, sel), zz, ss);
    }
  }
}
__device__ __forceinline__ void store_regs(uint32_t chunk_base, int row, const uint32_t (&o)[32]) {
#pragma unroll
  for (int i = 0; i < 8; ++i)
    sts_v4(chunk_base + swz_off(row, i, 128), o[4 * i], o[4 * i + 1], o[4 * i + 2], o[4 * i + 3]);
}
// Half h of a RoPE-key row (fetch_rope_half): o[0..15] from the 32 INT4 codes
// of f.a, the same arithmetic as dq_regs; stored as pieces 4 h .. 4 h + 3.
__device__ __forceinline__ void dq_half(uint32_t (&o)[32], const Fetch& f) {
  const __half2 sz = *reinterpret_cast<const __half2*>(&f.sz);
  const __half2 s2 = __half2half2(__low2half(sz));
  const __half2 zz2 = __half2half2(__hadd(__high2half(sz), __float2half_rn(1024.0f)));
  const uint32_t ss = *reinterpret_cast<const uint32_t*>(&s2);
  const uint32_t zz = *reinterpret_cast<const uint32_t*>(&zz2);
  constexpr uint32_t K = 0x64646464u;
  const uint32_t w[4] = {f.a.x, f.a.y, f.a.z, f.a.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t lo = w[i] & 0x0F0F0F0Fu;
    const uint32_t hi = (w[i] >> 4) & 0x0F0F0F0Fu;
    o[4 * i + 0] = dq2(__byte_perm(lo, K, 0x4140), zz, ss);
    o[4 * i + 1] = dq2(__byte_perm(hi, K, 0x4140), zz, ss);
    o[4 * i + 2] = dq2(__byte_perm(lo, K, 0x4342), zz, ss);
    o[4 * i + 3] = dq2(__byte_perm(hi, K, 0x4342), zz, ss);
  }
}
__device__ __forceinline__ void store_half(uint32_t chunk_base, int row, const uint32_t (&o)[32], int h) {
#pragma unroll
  for (int i = 0; i < 4; ++i)
    sts_v4(chunk_base + swz_off(row, 4 * h + i, 128), o[4 * i], o[4 * i + 1], o[4 * i + 2], o[4 * i + 3]);
}

// Rows of the paper's page. store_row_c4r4 writes one row (64 INT4 codes) of
// chunk k as RN_f16(s (q - z)) with the stored bf16 (content) or fp32 (RoPE)
// scale. q - z is exact in fp16 (as in store_row); a bf16 scale in [2^-14,
// 65504] is an fp16 value, so the fp16 product is the single rounding of the
// exact product. Any other scale (the fp32 RoPE scale, a tiny or huge content
// scale) multiplies in fp32 and rounds to fp16 after (store_row_c4r4_f32): one
// rounding for content, whose fp32 product is exact, and
// RN_f16(RN_f32(s (q - z))) for the RoPE key.
__device__ __forceinline__ void store_row_c4r4_f32(uint32_t chunk_base, int row, const uint4& a, const uint4& b,
                                                   float s, uint32_t zz) {
  constexpr uint32_t K = 0x64646464u;
  const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
  auto dqf = [&](uint32_t x) {
    uint32_t t;
    asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(t) : "r"(x), "r"(zz));
    const float2 d = __half22float2(*reinterpret_cast<const __half2*>(&t));
    return pack_h2(d.x * s, d.y * s);
  };
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint32_t lo = w[i] & 0x0F0F0F0Fu;
    const uint32_t hi = (w[i] >> 4) & 0x0F0F0F0Fu;
    sts_v4(chunk_base + swz_off(row, i, 128), dqf(__byte_perm(lo, K, 0x4140)), dqf(__byte_perm(hi, K, 0x4140)),
           dqf(__byte_perm(lo, K, 0x4342)), dqf(__byte_perm(hi, K, 0x4342)));
  }
}

template <bool kContent>
__device__ __forceinline__ void store_row_c4r4(uint32_t chunk_base, int row, const Fetch& f) {
  if (!f.ok) {
#pragma unroll
    for (int i = 0; i < 8; ++i) sts_v4(chunk_base + swz_off(row, i, 128), 0, 0, 0, 0);
    return;
  }
  const float s = __uint_as_float(f.sz);
  const __half2 zz2 = __half2half2(__float2half_rn(1024.0f + static_cast<float>(f.z)));
  const uint32_t zz = *reinterpret_cast<const uint32_t*>(&zz2);
  if constexpr (!kContent) {
    store_row_c4r4_f32(chunk_base, row, f.a, f.b, s, zz);
  } else {
    const __half sh = __float2half_rn(s);
    if (__half2float(sh) != s) {  // only a content scale outside fp16's normal range
      store_row_c4r4_f32(chunk_base, row, f.a, f.b, s, zz);
      return;
    }
    const __half2 s2 = __half2half2(sh);
    const uint32_t ss = *reinterpret_cast<const uint32_t*>(&s2);
    constexpr uint32_t K = 0x64646464u;
    const uint32_t w[8] = {f.a.x, f.a.y, f.a.z, f.a.w, f.b.x, f.b.y, f.b.z, f.b.w};
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint32_t lo = w[i] & 0x0F0F0F0Fu;
      const uint32_t hi = (w[i] >> 4) & 0x0F0F0F0Fu;
      sts_v4(chunk_base + swz_off(row, i, 128), dq2(__byte_perm(lo, K, 0x4140), zz, ss),
             dq2(__byte_perm(hi, K, 0x4140), zz, ss), dq2(__byte_perm(lo, K, 0x4342), zz, ss),
             dq2(__byte_perm(hi, K, 0x4342), zz, ss));
    }
  }
}

// The paper's page into registers (the decode workers compute a chunk row
// before its stores, as dq_regs does for this library's block): NW code words
// of f (8 for a row, 4 for half a RoPE row) into o[0 .. 4 NW). Same arithmetic
// as store_row_c4r4: fp16 subtract-and-multiply for a content row whose bf16
// scale is an fp16 value, else (the RoPE key, or a content scale outside
// fp16's normal range) the fp32 product rounded once to fp16.
template <int NW>
__device__ __forceinline__ void dq_regs_c4r4(uint32_t (&o)[32], const Fetch& f, bool content) {
  const float s = __uint_as_float(f.sz);
  const __half2 zz2 = __half2half2(__float2half_rn(1024.0f + static_cast<float>(f.z)));
  const uint32_t zz = *reinterpret_cast<const uint32_t*>(&zz2);
  constexpr uint32_t K = 0x64646464u;
  const uint32_t w[8] = {f.a.x, f.a.y, f.a.z, f.a.w, f.b.x, f.b.y, f.b.z, f.b.w};
  const __half sh = __float2half_rn(s);
  if (content && __half2float(sh) == s) {
    const __half2 s2 = __half2half2(sh);
    const uint32_t ss = *reinterpret_cast<const uint32_t*>(&s2);
#pragma unroll
    for (int i = 0; i < NW; ++i) {
      const uint32_t lo = w[i] & 0x0F0F0F0Fu;
      const uint32_t hi = (w[i] >> 4) & 0x0F0F0F0Fu;
      o[4 * i + 0] = dq2(__byte_perm(lo, K, 0x4140), zz, ss);
      o[4 * i + 1] = dq2(__byte_perm(hi, K, 0x4140), zz, ss);
      o[4 * i + 2] = dq2(__byte_perm(lo, K, 0x4342), zz, ss);
      o[4 * i + 3] = dq2(__byte_perm(hi, K, 0x4342), zz, ss);
    }
  } else {
    auto dqf = [&](uint32_t x) {
      uint32_t t;
      asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(t) : "r"(x), "r"(zz));
      const float2 d = __half22float2(*reinterpret_cast<const __half2*>(&t));
      return pack_h2(d.x * s, d.y * s);
    };
#pragma unroll
    for (int i = 0; i < NW; ++i) {
      const uint32_t lo = w[i] & 0x0F0F0F0Fu;
      const uint32_t hi = (w[i] >> 4) & 0x0F0F0F0Fu;
      o[4 * i + 0] = dqf(__byte_perm(lo, K, 0x4140));
      o[4 * i + 1] = dqf(__byte_perm(hi, K, 0x4140));
      o[4 * i + 2] = dqf(__byte_perm(lo, K, 0x4342));
      o[4 * i + 3] = dqf(__byte_perm(hi, K, 0x4342));
    }
  }
}

// A protected row's chunk k: 64 bf16 values (8 x 16 bytes) rounded to fp16 and
// placed in the same within-piece channel order as the packed rows
// (bf16 -> fp16 is exact for magnitudes in [2^-14, 65504]).
template <int CB>
__device__ __forceinline__ void store_row_prot(uint32_t chunk_base, int row, const uint4 (&v)[8], int k) {
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint32_t w[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
    float f[8];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      f[2 * e] = bf16_lo(w[e]);
      f[2 * e + 1] = bf16_hi(w[e]);
    }
    uint32_t o[4];
    if (k < 8) {
#pragma unroll
      for (int e = 0; e < 4; ++e) o[e] = pack_h2(f[Perm<CB>::at(2 * e)], f[Perm<CB>::at(2 * e + 1)]);
    } else {
#pragma unroll
      for (int e = 0; e < 4; ++e) o[e] = pack_h2(f[Perm<4>::at(2 * e)], f[Perm<4>::at(2 * e + 1)]);
    }
    sts_v4(chunk_base + swz_off(row, i, 128), o[0], o[1], o[2], o[3]);
  }
}

// BF16 comparison cache: the row is copied and rounded to fp16.
__device__ __forceinline__ void store_row_bf16(uint32_t chunk_base, int row, const uint4 (&v)[8], bool ok) {
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    uint32_t o[4] = {0, 0, 0, 0};
    if (ok) {
      const uint32_t w[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) o[e] = pack_h2(bf16_lo(w[e]), bf16_hi(w[e]));
    }
    sts_v4(chunk_base + swz_off(row, i, 128), o[0], o[1], o[2], o[3]);
  }
}

// One row's chunk k of a packed cache (this library's block or the paper's
// page) as dq_row would store it (the eight 16-byte pieces in order),
// computed into registers: the protected bf16 row when ps is set, else the
// packed row f. The decode workers compute it ahead of its stores.
template <int CB, bool PROT>
__device__ __forceinline__ void row_regs(uint32_t (&o)[32], const Fetch& f, int k, const uint8_t* ps) {
  if (PROT && ps != nullptr) {
    uint4 pv[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) pv[i] = __ldg(reinterpret_cast<const uint4*>(ps + k * 128) + i);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint32_t w[4] = {pv[i].x, pv[i].y, pv[i].z, pv[i].w};
      float v[8];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        v[2 * e] = bf16_lo(w[e]);
        v[2 * e + 1] = bf16_hi(w[e]);
      }
      if (k < 8) {
#pragma unroll
        for (int e = 0; e < 4; ++e) o[4 * i + e] = pack_h2(v[Perm<CB>::at(2 * e)], v[Perm<CB>::at(2 * e + 1)]);
      } else {
#pragma unroll
        for (int e = 0; e < 4; ++e) o[4 * i + e] = pack_h2(v[Perm<4>::at(2 * e)], v[Perm<4>::at(2 * e + 1)]);
      }
    }
  } else if constexpr (CB == kC4R4) {
    dq_regs_c4r4<8>(o, f, k < 8);
  } else {
    dq_regs(o, f, CB == 4 || k == 8);
  }
  // Pin the results here: the (volatile) slot wait that follows must not be
  // hoisted above the arithmetic.
#pragma unroll
  for (int i = 0; i < 32; ++i) asm volatile("" : "+r"(o[i]));
}
// Half h of a RoPE-key row into o[0..15] (pieces 4 h .. 4 h + 3): the
// protection row's bf16 channels 32 h .. 32 h + 31 rounded to fp16 when the
// row is protected, else dq_half of the packed codes.
template <int CB, bool PROT>
__device__ __forceinline__ void row_regs_half(uint32_t (&o)[32], const Fetch& f, const uint8_t* ps, int h) {
  if (PROT && ps != nullptr) {
    uint4 pv[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) pv[i] = __ldg(reinterpret_cast<const uint4*>(ps + 8 * 128 + h * 64) + i);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const uint32_t w[4] = {pv[i].x, pv[i].y, pv[i].z, pv[i].w};
      float v[8];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        v[2 * e] = bf16_lo(w[e]);
        v[2 * e + 1] = bf16_hi(w[e]);
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) o[4 * i + e] = pack_h2(v[Perm<4>::at(2 * e)], v[Perm<4>::at(2 * e + 1)]);
    }
  } else if constexpr (CB == kC4R4) {
    dq_regs_c4r4<4>(o, f, false);
  } else {
    dq_half(o, f);
  }
#pragma unroll
  for (int i = 0; i < 16; ++i) asm volatile("" : "+r"(o[i]));
}

// BF16 cache rows read coalesced: lane l of a warp handles piece l & 7 (16
// bytes) of rows r0 + 4 i + (l >> 3), i = 0..7, so every load instruction
// reads four whole 128-byte lines (32 rows x one chunk per warp). r0 is the
// warp's first row (its rows share a block, slots slot0 ..); vmask bit m is
// set when row r0 + m is to be read (else zeros).
__device__ __forceinline__ void bf16_load_t(uint4 (&v)[8], const uint8_t* blk, uint32_t vmask, int slot0, int k,
                                            int lane) {
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int m = 4 * i + (lane >> 3);
    v[i] = (vmask >> m) & 1u ? ldg_nc_v4(blk + (slot0 + m) * (kDqk * 2) + k * 128 + (lane & 7) * 16)
                             : make_uint4(0, 0, 0, 0);
  }
}
// Writes those pieces rounded to fp16 into the swizzled chunk.
__device__ __forceinline__ void bf16_store_t(uint32_t chunk_base, int r0, const uint4 (&v)[8], int lane) {
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int m = 4 * i + (lane >> 3);
    const uint32_t w[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
    uint32_t o[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) o[e] = pack_h2(bf16_lo(w[e]), bf16_hi(w[e]));
    sts_v4(chunk_base + swz_off(r0 + m, lane & 7, 128), o[0], o[1], o[2], o[3]);
  }
}

// Query image of one unit: HG heads x 576 channels in fp16 laid out exactly as
// the K-major, 128-byte-swizzled shared-memory operand ([chunk][head][128 B]),
// channels permuted within each 8-channel piece like the cache rows. Piece
// (k, h, i) is 8 channels of chunk k, head h. bf16 -> fp16 is exact for
// magnitudes in [2^-14, 65504].
template <int CB, int HG>
__device__ __forceinline__ void query_piece(const Params& p, uint8_t* img, int b, int h0, int idx) {
  const int i = idx & 7;
  const int kh = idx >> 3;
  const int h = kh % HG;
  const int k = kh / HG;
  uint4 raw = make_uint4(0, 0, 0, 0);
  if (h0 + h < p.heads) {
    const size_t bh = static_cast<size_t>(b) * p.heads + h0 + h;
    const __nv_bfloat16* src = k < 8 ? p.q_lat + bh * kDc + k * 64 + i * 8 : p.q_pe + bh * kDr + i * 8;
    raw = *reinterpret_cast<const uint4*>(src);
  }
  const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
  float f[8];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    f[2 * e] = bf16_lo(w[e]);
    f[2 * e + 1] = bf16_hi(w[e]);
  }
  uint4 o;
  uint32_t* ov = reinterpret_cast<uint32_t*>(&o);
  if (k < 8 || CB == 16) {
#pragma unroll
    for (int e = 0; e < 4; ++e) ov[e] = pack_h2(f[Perm<CB>::at(2 * e)], f[Perm<CB>::at(2 * e + 1)]);
  } else {
#pragma unroll
    for (int e = 0; e < 4; ++e) ov[e] = pack_h2(f[Perm<4>::at(2 * e)], f[Perm<4>::at(2 * e + 1)]);
  }
  *reinterpret_cast<uint4*>(img + k * HG * 128 + swz_off(h, i, 128)) = o;
}

// ------------------------------------------------------------ worker warps
// Eight worker warps dequantise each tile, compute its softmax and write the
// segment results. Warp w owns token rows 32 (w & 3) .. 32 (w & 3) + 31 (its
// TMEM lane quarter), dequantises the chunks of parity w >> 2 and, in the
// softmax and epilogue, the heads [(w >> 2) HG/2, (w >> 2 + 1) HG/2).
template <int HG>
struct Cols {
  static constexpr int kPerWarp = HG / 2;       // heads per worker warp
  static constexpr int kW = HG >= 32 ? 16 : 8;  // TMEM columns per load
  static constexpr int kN = kPerWarp / kW;      // loads per column set
  static_assert(kN * kW == kPerWarp, "column split");
};


__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// A thread's row admits the warp's head columns i >= lim (lim = kPerWarp for a
// row past the sequence end; with several query tokens per sequence, the
// heads of earlier query tokens do not see the last positions: Eq. mla_compact's
// causal mask, see row_limit).

// W columns of this thread's row of S^T starting at t_s: the sum of the
// kQkParts partials (HG columns apart), added in a fixed order.
template <int HG, int W>
__device__ __forceinline__ void load_s(uint32_t t_s, uint32_t (&r)[W]) {
  tmem_ld(t_s, r);
  if constexpr (kQkParts > 1) {
    uint32_t a[kQkParts - 1][W];
#pragma unroll
    for (int q = 1; q < kQkParts; ++q) tmem_ld(t_s + q * HG, a[q - 1]);
    tmem_ld_wait();
#pragma unroll
    for (int jj = 0; jj < W; ++jj) {
      float v = __uint_as_float(r[jj]);
#pragma unroll
      for (int q = 1; q < kQkParts; ++q) v += __uint_as_float(a[q - 1][jj]);
      r[jj] = __float_as_uint(v);
    }
  } else {
    tmem_ld_wait();
  }
}

// Tile max of the scaled scores of this warp's heads over its 32 rows into red_q[h].
template <int HG>
__device__ __forceinline__ void warp_tile_max(uint32_t t_s, float sl2, int lim, float* red_q, int lane) {
  using C = Cols<HG>;
#pragma unroll
  for (int c = 0; c < C::kN; ++c) {
    uint32_t r[C::kW];
    load_s<HG>(t_s + c * C::kW, r);
#pragma unroll
    for (int jj = 0; jj < C::kW; ++jj) {
      const float x = c * C::kW + jj >= lim ? __uint_as_float(r[jj]) * sl2 : -INFINITY;
      const float mx = warp_max_f32(x);
      if (lane == jj) red_q[c * C::kW + jj] = mx;
    }
  }
}

// P^T[t, h] = 2^(S * scale * log2e - m_ref[h]) in fp16 for this warp's heads,
// into row t of the P tile and into pk; returns whether a weight exceeds 2^8.
template <int HG>
__device__ __forceinline__ bool compute_p(uint32_t t_s, const float* mr, float sl2, int lim, uint32_t ptile,
                                          int row, int piece0, uint32_t (&pk)[Cols<HG>::kPerWarp / 2]) {
  using C = Cols<HG>;
  constexpr uint32_t kRB = Cfg<HG>::kPRowBytes;
  bool over = false;
#pragma unroll
  for (int c = 0; c < C::kN; ++c) {
    float m[C::kW];
#pragma unroll
    for (int v4 = 0; v4 < C::kW / 4; ++v4) {
      const float4 mv = reinterpret_cast<const float4*>(mr)[c * (C::kW / 4) + v4];
      m[4 * v4] = mv.x;
      m[4 * v4 + 1] = mv.y;
      m[4 * v4 + 2] = mv.z;
      m[4 * v4 + 3] = mv.w;
    }
    uint32_t r[C::kW];
    load_s<HG>(t_s + c * C::kW, r);
#pragma unroll
    for (int jj = 0; jj < C::kW; jj += 2) {
      const float x0 = __uint_as_float(r[jj]) * sl2 - m[jj];
      const float x1 = __uint_as_float(r[jj + 1]) * sl2 - m[jj + 1];
      const bool ok0 = c * C::kW + jj >= lim, ok1 = c * C::kW + jj + 1 >= lim;
      over |= (ok0 && x0 > kRescaleLog2) || (ok1 && x1 > kRescaleLog2);
      pk[c * (C::kW / 2) + (jj >> 1)] = pack_h2(ok0 ? ex2_approx(x0) : 0.0f, ok1 ? ex2_approx(x1) : 0.0f);
    }
#pragma unroll
    for (int pc = 0; pc < C::kW / 8; ++pc) {
      const uint32_t* w = &pk[c * (C::kW / 2) + 4 * pc];
      sts_v4(ptile + swz_off(row, piece0 + c * (C::kW / 8) + pc, kRB), w[0], w[1], w[2], w[3]);
    }
  }
  return over;
}

// lim of a tile row: kPerWarp past the sequence end; else the number of this
// warp's head columns whose query token precedes the row's position. Query
// token t of a sequence of len tokens sits at position len - q_tokens + t and
// sees positions <= its own, so row position pos is hidden from tokens
// t < d = pos - (len - q_tokens), i.e. from virtual heads v < d * hpt: a prefix
// of the head columns.
template <int HG>
__device__ __forceinline__ int row_limit(const Params& p, const TileInfo& ti, int row, int cb0) {
  constexpr int kPer = Cols<HG>::kPerWarp;
  if (row >= ti.ntok) return kPer;
  const int d = kTileTokens * ti.j + row - (ti.len - p.q_tokens);
  if (d <= 0) return 0;
  return min(max(d * p.hpt - (ti.hg * HG + cb0), 0), kPer);
}

// What a segment end needs once its last PV has completed.
struct SegEnd {
  int b, hg;
  bool whole;   // the segment is the whole unit: write out / lse, else a partial
  size_t pidx;  // partial slot (CTA index + unit)
};

// Segment end: l[h] from the row-sum accumulator (every TMEM lane holds the
// same sums; the warps of lane quarter 0 read theirs once the segment's last
// row-sum MMAs, phase rs_parity of rs_done, have completed), then out = O / l
// (or the partial o, m, l) for this warp's heads, then release O^T and the
// row sums to the next segment.
template <int CB, int HG>
__device__ bool epilogue(const Params& p, const SegEnd& e, Ctrl& ctl, uint32_t tmem, uint32_t& gph,
                         uint32_t rs_parity, int warp, int lane) {
  using C = Cols<HG>;
  const int q4 = warp & 3, half = warp >> 2, row = q4 * 32 + lane, cb0 = half * C::kPerWarp;
  const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
  const uint32_t t_o = tmem + cb0 + lane_off;
  if (q4 == 0) {
    if (!wwait(&ctl.rs_done, rs_parity, ctl, kSitePvEpi, p.dev_err)) return false;
    tc_fence_after();
#pragma unroll
    for (int c = 0; c < C::kN; ++c) {
      uint32_t r[C::kW];
      tmem_ld(tmem + Cfg<HG>::kColL + cb0 + c * C::kW, r);
      tmem_ld_wait();
      if (lane == 0) {
#pragma unroll
        for (int jj = 0; jj < C::kW; ++jj) ctl.red[0][cb0 + c * C::kW + jj] = __uint_as_float(r[jj]);
      }
    }
  }
  if (!group_sync(ctl, gph, p.dev_err)) return false;
  const int tid = threadIdx.x;  // 0 .. 255 over the worker warps
  if (tid < HG) {
    const float l = ctl.red[0][tid];
    ctl.alpha[tid] = l;
    ctl.inv[tid] = l > 0.0f ? 1.0f / l : 0.0f;  // one division per head; 0 for a head that saw no key
  }
  if (!group_sync(ctl, gph, p.dev_err)) return false;
  const int h0 = e.hg * HG;
  const int hn = min(HG, p.heads - h0);
  float* const obase =
      e.whole ? p.out + (static_cast<size_t>(e.b) * p.heads + h0) * kDc : p.part_o + e.pidx * HG * kDc;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int P = i * 128 + row;  // position in the reconstructed row
    float* const orow = obase + (P & ~7) + Perm<CB>::at(P & 7);
#pragma unroll
    for (int c = 0; c < C::kN; ++c) {
      uint32_t r[C::kW];
      tmem_ld(t_o + i * HG + c * C::kW, r);
      float f[C::kW];
#pragma unroll
      for (int v4 = 0; v4 < C::kW / 4; ++v4) {
        const float4 iv = e.whole ? reinterpret_cast<const float4*>(ctl.inv + cb0)[c * (C::kW / 4) + v4]
                                  : make_float4(1.f, 1.f, 1.f, 1.f);
        f[4 * v4] = iv.x;
        f[4 * v4 + 1] = iv.y;
        f[4 * v4 + 2] = iv.z;
        f[4 * v4 + 3] = iv.w;
      }
      tmem_ld_wait();
#pragma unroll
      for (int jj = 0; jj < C::kW; ++jj) {
        const int h = cb0 + c * C::kW + jj;
        if (h < hn) orow[static_cast<size_t>(h) * kDc] = __uint_as_float(r[jj]) * f[jj];
      }
    }
  }
  if (tid < HG && h0 + tid < p.heads) {
    if (e.whole) {
      if (p.lse != nullptr)
        p.lse[static_cast<size_t>(e.b) * p.heads + h0 + tid] = (ctl.m_ref[tid] + log2f(ctl.alpha[tid])) * kLn2;
    } else {
      p.part_ml[(e.pidx * HG + tid) * 2 + 0] = ctl.m_ref[tid];
      p.part_ml[(e.pidx * HG + tid) * 2 + 1] = ctl.alpha[tid];
    }
  }
  tc_fence_before();
  __syncwarp();
  mbar_arrive_if(lane == 0 ? 1u : 0u, &ctl.o_free);
  return true;
}

// Chunk k of one tile row of a packed cache: the protected bf16 row when ps is
// set, else the packed row f dequantised (the paper's page or this library's
// block). The decode workers and the tile dump share it.
template <int CB, bool PROT>
__device__ __forceinline__ void dq_row(uint32_t chunk_base, int row, int k, const uint8_t* ps, const Fetch& f) {
  if (PROT && ps != nullptr) {
    uint4 pv[8];  // the protected row's 64 bf16 values of chunk k
    // L1-allocating loads: the eight 16-byte pieces of the row's 128-byte line
    // come from one L1 fill instead of eight L2 reads.
#pragma unroll
    for (int i = 0; i < 8; ++i) pv[i] = __ldg(reinterpret_cast<const uint4*>(ps + k * 128) + i);
    store_row_prot<CB>(chunk_base, row, pv, k);
  } else if constexpr (CB == kC4R4) {
    if (k < 8) {
      store_row_c4r4<true>(chunk_base, row, f);
    } else {
      store_row_c4r4<false>(chunk_base, row, f);
    }
  } else {
    store_row<CB>(chunk_base, row, f, CB == 4 || k == 8);
  }
}

// PROT: the cache has sink4/local128 protection rows (a separate instantiation,
// so the unprotected kernel carries none of that code).
template <int CB, int HG, bool PROT>
__device__ void worker_role(const Params& p, Sched sc, uint32_t chunks, Ctrl& ctl, uint32_t tmem, int warp,
                            int lane) {
  using C = Cols<HG>;
  const int q4 = warp & 3;
  // dequantised chunks k = par, par + 2, ...; heads half `par` (the mask tells
  // the compiler par <= 1, so each unrolled chunk step knows whether k < 8)
  const int par = (warp >> 2) & 1;
  const int row = q4 * 32 + lane;
  const int slot = row & 63;
  const int cb0 = par * C::kPerWarp;
  const int piece0 = cb0 / 8;
  const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
  const uint32_t t_s = tmem + 4 * HG + cb0 + lane_off;
  const uint32_t t_o = tmem + cb0 + lane_off;
  const uint32_t ptile = chunks + 8 * kChunkBytes;
  const float sl2 = p.scale_log2;
  constexpr int kMyChunks = 5;  // chunk steps per warp (the paper's page and BF16: parity 1 has 4)
  // The packed caches (this library's INT4 / INT2 block and the paper's page):
  // each warp dequantises 4 content chunks and half of the RoPE-key chunk
  // (channels 32 par .. 32 par + 31), each row's arithmetic ahead of its stores.
  constexpr bool kEarly = CB == 4 || CB == 2 || CB == kC4R4;
  uint32_t it = 0, gph = 0, nresc = 0;
  int seg_j0 = 0;
  bool ok = true;
  bool pending = false;  // the previous tile ended a segment whose epilogue is still due
  SegEnd pend{};

  // Packed rows of the tile about to be dequantised (INT4/INT2), fetched a tile ahead.
  Fetch f[kMyChunks];
  // BF16 cache: one chunk row (8 x 16 B) of look-ahead.
  uint4 cur[CB == 16 ? 8 : 1];
  bool valid_cur = false;
  RowRef ref0;  // the first tile's reference, prepared by the prep kernel
  {
    const int4 fr = p.cta_first[blockIdx.x];
    ref0.has = sc.valid();
    ref0.entry = row < 64 ? fr.x : fr.y;
    ref0.len = fr.z;
    ref0.j = fr.w;
    ref0.b = sc.u / p.n_hg;
  }
  // A protected row reads its BF16 row instead of the packed cache.
  const uint8_t* psrc_cur = PROT ? prot_row(p, ref0, row) : nullptr;
  if constexpr (PROT) {
    if (psrc_cur != nullptr) {
#pragma unroll
      for (int i = 0; i < kDqk * 2 / 128; ++i) asm volatile("prefetch.global.L2 [%0];" ::"l"(psrc_cur + i * 128));
    }
  }
  const uint8_t* blk_cur = psrc_cur != nullptr ? nullptr : resolve_row<CB>(p, ref0, row, valid_cur);
  if constexpr (kEarly) {
#pragma unroll
    for (int kc = 0; kc < 4; ++kc) f[kc] = fetch_chunk<CB>(blk_cur, valid_cur, 2 * kc + par, slot);
    f[4] = fetch_rope_half<CB>(blk_cur, valid_cur, slot, par);
  } else if constexpr (CB != 16) {
#pragma unroll
    for (int kc = 0; kc < kMyChunks; ++kc) {
      const int k = 2 * kc + par;
      if (k < kNumChunks) f[kc] = fetch_chunk<CB>(blk_cur, valid_cur, k, slot);
    }
  } else {
    // (the warp's 32 rows share a block: lane 0's row is valid whenever any is)
    const uint8_t* wblk = reinterpret_cast<const uint8_t*>(
        __shfl_sync(0xffffffffu, reinterpret_cast<unsigned long long>(blk_cur), 0));
    bf16_load_t(cur, wblk, __ballot_sync(0xffffffffu, valid_cur), slot & ~31, par, lane);
  }
  // Table references run one tile ahead of the block pointer they resolve to.
  Sched nx = sc;
  nx.next();
  RowRef ref_nx = row_ref(p, nx, row);

  for (; ok && sc.valid(); sc.next()) {
    const TileFlags tf = tile_flags(sc);
    if (tf.first) seg_j0 = sc.t - sc.pu0;
    // The next tile's block pointer (its table entry was loaded a tile ago)
    // and the table entry of the tile after it.
    bool valid_nx = false;
    const uint8_t* psrc_nx = PROT ? prot_row(p, ref_nx, row) : nullptr;
    if constexpr (PROT) {
      // The next tile's protected rows into L2 now (no registers held): their
      // chunk loads come after each slot wait and would otherwise miss to DRAM.
      if (psrc_nx != nullptr) {
#pragma unroll
        for (int i = 0; i < kDqk * 2 / 128; ++i) asm volatile("prefetch.global.L2 [%0];" ::"l"(psrc_nx + i * 128));
      }
    }
    const uint8_t* blk_nx = psrc_nx != nullptr ? nullptr : resolve_row<CB>(p, ref_nx, row, valid_nx);
    if constexpr (CB != 16) {
      // The next tile's two packed blocks into L2 by the bulk-copy engine (one
      // request each, from the threads of rows 0 and 64), so that the register
      // fetch of its rows after this tile's chunk loop reads L2, not DRAM.
      if (lane == 0 && (q4 & 1) == 0 && par == 0 && valid_nx) bulk_prefetch_l2(blk_nx, BlockLayout<CB>::kBytes);
    }
    if constexpr (CB == 16) {
      // BF16 cache: its rows are read only one chunk ahead into registers, so
      // bring the next tile's lines of this thread's row and chunks into L2 now.
      if (valid_nx) {
#pragma unroll
        for (int kc = 0; kc < kMyChunks; ++kc) {
          const int k = 2 * kc + par;
          if (k < kNumChunks)
            asm volatile("prefetch.global.L2 [%0];" ::"l"(blk_nx + slot * (kDqk * 2) + k * 128));
        }
      }
    }
    Sched nn = nx;
    nn.next();
    const RowRef ref_nn = row_ref(p, nn, row);
    if (lane == 0 && warp == 0) QMLA_TRACE(0, it);

    // ---- dequantise this tile. The previous tile's four PV blocks (one issuer
    // each) complete together, so one wait frees every slot. For the packed
    // caches (protected rows included) the arithmetic of the first chunk and
    // of the RoPE half runs before that wait and each further chunk's while
    // the stores of the one before drain, ahead of its proxy fence.
    uint32_t dq[kEarly ? 32 : 1];
    uint32_t dqh[kEarly ? 32 : 1];  // the RoPE half (16 words), also computed before the wait
    if constexpr (kEarly) {
      row_regs<CB, PROT>(dq, f[0], par, psrc_cur);
      row_regs_half<CB, PROT>(dqh, f[4], psrc_cur, par);
    }
    if (lane == 0 && warp == 0) QMLA_TRACE(105, it);
    if (!(ok = wwait(&ctl.pv_done, (it & 1u) ^ 1u, ctl, kSiteDqSlot, p.dev_err))) break;
    if (lane == 0) QMLA_TRACE(88 + warp, it);
    if (lane == 0 && (warp & 3) == 0) QMLA_TRACE(warp == 0 ? 96 : 101, it);
#pragma unroll
    for (int kc = 0; kc < kMyChunks; ++kc) {
      // (packed caches: content chunks 2 kc + par, then half par of the RoPE chunk)
      const int k = kEarly && kc == 4 ? 8 : 2 * kc + par;
      if (k >= kNumChunks) break;
      // The RoPE chunk's slot held the previous tile's P, which its row-sum
      // MMAs (committed apart from the PV) may still be reading.
      if (k == 8 && !(ok = wwait(&ctl.rs_done, (it & 1u) ^ 1u, ctl, kSiteDqSlot, p.dev_err))) break;
      if constexpr (CB == 16) {
        // (a wait per chunk, as a scheduling barrier: without it the compiler
        // hoists the loads of later chunks and spills)
        if (kc > 0 && !(ok = wwait(&ctl.pv_done, (it & 1u) ^ 1u, ctl, kSiteDqSlot, p.dev_err))) break;
        uint4 nxt[8];
        const int kn = k + 2;
        const bool same = kn < kNumChunks;  // the next chunk of this tile, else the next tile's first
        const uint8_t* wblk = reinterpret_cast<const uint8_t*>(__shfl_sync(
            0xffffffffu, reinterpret_cast<unsigned long long>(same ? blk_cur : blk_nx), 0));
        bf16_load_t(nxt, wblk, __ballot_sync(0xffffffffu, same ? valid_cur : valid_nx), slot & ~31,
                    same ? kn : par, lane);
        bf16_store_t(chunks + k * kChunkBytes, q4 * 32, cur, lane);
#pragma unroll
        for (int i = 0; i < 8; ++i) cur[i] = nxt[i];
      } else if constexpr (kEarly) {
        if (kc < 4) {
          store_regs(chunks + k * kChunkBytes, row, dq);
        } else {
          store_half(chunks + 8 * kChunkBytes, row, dqh, par);
        }
        // the next chunk's arithmetic while these stores drain
        if (kc + 1 < 4) row_regs<CB, PROT>(dq, f[kc + 1], k + 2, psrc_cur);
      } else {
        dq_row<CB, PROT>(chunks + k * kChunkBytes, row, k, psrc_cur, f[kc]);
        f[kc] = fetch_chunk<CB>(blk_nx, valid_nx, k, slot);  // the next tile's rows of this chunk
      }
      fence_proxy_async_smem();
      __syncwarp();
      mbar_arrive_if(lane == 0 ? 1u : 0u, &ctl.chunk_full[k]);
      if (lane == 0) QMLA_TRACE(48 + warp * 5 + kc, it);
    }
    if (!ok) break;
    if constexpr (kEarly) {
      // The next tile's packed rows, issued once this tile's stores are out
      // (inside the chunk loop their issue queued behind the stores).
#pragma unroll
      for (int kc = 0; kc < 4; ++kc) f[kc] = fetch_chunk<CB>(blk_nx, valid_nx, 2 * kc + par, slot);
      f[4] = fetch_rope_half<CB>(blk_nx, valid_nx, slot, par);
    }
    if (lane == 0) QMLA_TRACE(32 + warp, it);
    blk_cur = blk_nx;
    valid_cur = valid_nx;
    psrc_cur = psrc_nx;
    nx = nn;
    ref_nx = ref_nn;
    const TileInfo ti = tile_info(sc, p);  // ntok of this tile for the softmax
    const int lim = row_limit<HG>(p, ti, row, cb0);

    // ---- the previous segment's results (its last PV completed: pv_done was waited for above)
    if (pending) {
      tc_fence_after();
      if (!(ok = epilogue<CB, HG>(p, pend, ctl, tmem, gph, (it - 1) & 1u, warp, lane))) break;
      pending = false;
      if (lane == 0 && warp == 0) QMLA_TRACE(20, it);
    }

    // ---- softmax of this tile
    if (!(ok = wwait(&ctl.s_full, it & 1u, ctl, kSiteSmSFull, p.dev_err))) break;
    tc_fence_after();
    if (lane == 0 && warp == 0) QMLA_TRACE(16, it);
    if (ti.first) {
      // New segment: the reference is this tile's max.
      warp_tile_max<HG>(t_s, sl2, lim, &ctl.red[q4][cb0], lane);
      if (!(ok = group_sync(ctl, gph, p.dev_err))) break;
      if (threadIdx.x < HG) {
        const int h = threadIdx.x;
        ctl.m_ref[h] = fmaxf(fmaxf(ctl.red[0][h], ctl.red[1][h]), fmaxf(ctl.red[2][h], ctl.red[3][h]));
      }
      if (!(ok = group_sync(ctl, gph, p.dev_err))) break;
    }
    uint32_t pk[C::kPerWarp / 2];
    const bool over = compute_p<HG>(t_s, ctl.m_ref + cb0, sl2, lim, ptile, row, piece0, pk);
    // A weight above 2^8 anywhere in the tile asks for a rescale; the flag is
    // written before p_full, so whoever has seen p_full complete reads it.
    if (__any_sync(0xffffffffu, over) && lane == 0) *reinterpret_cast<volatile uint32_t*>(&ctl.resc_tile) = it + 1;
    fence_proxy_async_smem();
    tc_fence_before();
    __syncwarp();
    mbar_arrive_if(lane == 0 ? 1u : 0u, &ctl.p_full);
    if (lane == 0 && warp == 0) QMLA_TRACE(19, it);
    // Off the MMA issuers' path from here: learn whether any warp asked for a rescale.
    if (!(ok = wwait(&ctl.p_full, it & 1u, ctl, kSiteGrp, p.dev_err))) break;
    if (lane == 0 && warp == 0) QMLA_TRACE(17, it);
    if (*reinterpret_cast<volatile uint32_t*>(&ctl.resc_tile) == it + 1) {
      // Raise the reference to the running max; O and the row sums were
      // accumulated against the old one and are scaled by alpha = 2^(m_old - m_new).
      // The previous PV has completed (its slots were waited for above); the
      // MMA issuers wait on p_fixed before this tile's PV.
      tc_fence_after();
      warp_tile_max<HG>(t_s, sl2, lim, &ctl.red[q4][cb0], lane);
      if (!(ok = group_sync(ctl, gph, p.dev_err))) break;
      if (threadIdx.x < HG) {
        const int h = threadIdx.x;
        const float mt = fmaxf(fmaxf(ctl.red[0][h], ctl.red[1][h]), fmaxf(ctl.red[2][h], ctl.red[3][h]));
        const float mo = ctl.m_ref[h];
        const float mn = fmaxf(mo, mt);
        ctl.alpha[h] = mo == mn ? 1.0f : exp2f(mo - mn);  // also when no key was seen yet (-inf)
        ctl.m_ref[h] = mn;
      }
      if (!(ok = group_sync(ctl, gph, p.dev_err))) break;
      if (!ti.first) {
        // (the previous tile's row-sum MMAs must have landed before L is rescaled)
        if (!(ok = wwait(&ctl.rs_done, (it - 1) & 1u, ctl, kSitePvEpi, p.dev_err))) break;
        tc_fence_after();
#pragma unroll
        for (int i = 0; i < 5; ++i) {  // O^T blocks 0..3 and the row sums
          const uint32_t col = i < 4 ? i * HG : Cfg<HG>::kColL;
#pragma unroll
          for (int c = 0; c < C::kN; ++c) {
            uint32_t r[C::kW];
            tmem_ld(t_o + col + c * C::kW, r);
            tmem_ld_wait();
#pragma unroll
            for (int jj = 0; jj < C::kW; ++jj)
              r[jj] = __float_as_uint(__uint_as_float(r[jj]) * ctl.alpha[cb0 + c * C::kW + jj]);
            tmem_st(t_o + col + c * C::kW, r);
          }
        }
        tmem_st_wait();
      }
      compute_p<HG>(t_s, ctl.m_ref + cb0, sl2, lim, ptile, row, piece0, pk);
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      mbar_arrive_if(lane == 0 ? 1u : 0u, &ctl.p_fixed);
      ++nresc;
    }
    // (the row sums of the fp16 weights are summed by the tensor core, see mma_issuer)
    if (lane == 0 && warp == 0) QMLA_TRACE(18, it);
    if (ti.last) {
      pending = true;
      pend.b = ti.b;
      pend.hg = ti.hg;
      pend.whole = (seg_j0 == 0) && (sc.t + 1 == sc.pu1);
      pend.pidx = static_cast<size_t>(blockIdx.x) + sc.u;
    }
    ++it;
  }
  // The last segment's results once its PV has completed.
  if (ok && pending) {
    if ((ok = wwait(&ctl.pv_done, (it - 1) & 1u, ctl, kSitePvEpi, p.dev_err))) {
      tc_fence_after();
      ok = epilogue<CB, HG>(p, pend, ctl, tmem, gph, (it - 1) & 1u, warp, lane);
    }
  }
  if (!ok && lane == 0) set_abort(ctl, p.dev_err);
}

// ------------------------------------------------------------ MMA warp
// Copies the query image of `unit` into shared memory with the bulk-copy
// engine, completing on q_full through its transaction count.
template <int HG>
__device__ __forceinline__ void issue_query(const Params& p, int unit, uint8_t* qsmem, Ctrl& ctl) {
  constexpr uint32_t kBytes = Cfg<HG>::kQBytes;
  mbar_arrive_expect_tx(&ctl.q_full, kBytes);
  const uint8_t* src = p.qimg + static_cast<size_t>(unit) * kBytes;
#pragma unroll 1
  for (int k = 0; k < kNumChunks; ++k) bulk_g2s(qsmem + k * HG * 128, src + k * HG * 128, HG * 128, &ctl.q_full);
}

// Bounded wait of an MMA-issuing thread (no warp-collective operations: the
// other lanes of its warp have exited).
__device__ __forceinline__ bool twait(uint64_t* bar, uint32_t parity, Ctrl& c, uint32_t site, uint32_t* dev_err) {
  return wait_ok(mbar_wait(bar, parity, kWaitNs, &c.abort), site, c, dev_err);
}

// Issuer j (0..3, one thread of warp 8 + j; the other lanes exit at the start:
// a warp whose lane 0 issues or waits while the other lanes sit at a
// re-convergence point was measured to issue MMAs and wake up far more slowly
// on sm_103a) issues K-steps kk = j mod kQkParts of every QK chunk into S^T
// partial j, and PV block j (channels 128 j .. 128 j + 127) into O^T block j.
// A commit tracks the MMAs issued by the committing thread, so each issuer
// commits its own: s_full counts the QK partials, pv_done the PV blocks. Issuer 0 also copies the query
// images. QK starts on each chunk as soon as it is written. Descriptors are
// advanced by adding (byte offset >> 4) to their start-address field.
template <int HG>
__device__ void mma_issuer(const Params& p, Sched sc, uint32_t chunks, uint8_t* qsmem, Ctrl& ctl, uint32_t tmem,
                           int j) {
  constexpr uint32_t kIdQK = idesc_f16_f32(128, HG, false, false);
  constexpr uint32_t kIdPV = idesc_f16_f32(128, HG, true, true);
  constexpr uint32_t kIdL = idesc_f16_f32(128, HG, false, true);  // A (ones) from TMEM, B = P^T
  constexpr uint32_t kRB = Cfg<HG>::kPRowBytes;
  constexpr uint32_t kSboP = 8 * kRB;
  constexpr int kSteps = 4 / kQkParts;  // QK K-steps per chunk and issuer
  const bool qk = j < kQkParts;
  const uint32_t qbase = smem_u32(qsmem);
  const uint32_t ptile = chunks + 8 * kChunkBytes;
  const uint32_t t_s = tmem + (4 + j) * HG;  // S^T partial j
  const uint32_t t_o = tmem + j * HG;        // O^T block j
  const uint64_t qk_a0 = smem_desc(chunks, 16, 1024, SWZ_128B) + static_cast<uint64_t>((j * 32) >> 4);
  const uint64_t qk_b0 = smem_desc(qbase, 16, 1024, SWZ_128B) + static_cast<uint64_t>((j * 32) >> 4);
  const uint64_t pv_a0 =
      smem_desc(chunks, kChunkBytes, 1024, SWZ_128B) + static_cast<uint64_t>((2 * j * kChunkBytes) >> 4);
  const uint64_t pv_b0 = smem_desc(ptile, 16 * kSboP, kSboP, swz_mode_for_row(kRB));
  uint32_t it = 0, seg = 0, nresc = 0;
  bool ok = true;
  if (j == 0 && sc.valid()) issue_query<HG>(p, sc.u, qsmem, ctl);
  for (; ok && sc.valid(); sc.next()) {
    const TileFlags ti = tile_flags(sc);
    if (j == 0) QMLA_TRACE(1, it);
    if (ti.first && !(ok = twait(&ctl.q_full, seg & 1u, ctl, kSiteMmaQFull, p.dev_err))) break;
    if (qk) {
      // S^T = C_hat . q^T over the nine 64-channel chunks (K = 576), chunk by
      // chunk. The next chunk's barrier is probed before this chunk's MMAs are
      // issued, so the probe's latency overlaps them; only a chunk that was not
      // yet written takes the (bounded) wait.
      // (Unrolled by three: fully unrolled, the first tile after a cold start
      // spends thousands of cycles fetching the loop's instructions.)
      bool ready = mbar_test(&ctl.chunk_full[0], it & 1u);
#pragma unroll 3
      for (int k = 0; k < kNumChunks; ++k) {
        if (!ready && !(ok = twait(&ctl.chunk_full[k], it & 1u, ctl, kSiteMmaChunk, p.dev_err))) break;
        tc_fence_after();
        if (j == 0) QMLA_TRACE(112 + k, it);
        if (k + 1 < kNumChunks) ready = mbar_test(&ctl.chunk_full[k + 1], it & 1u);
#pragma unroll
        for (int kk = 0; kk < kSteps; ++kk)
          umma_f16_ss(t_s, qk_a0 + static_cast<uint64_t>((k * kChunkBytes + kk * kQkParts * 32) >> 4),
                      qk_b0 + static_cast<uint64_t>((k * HG * 128 + kk * kQkParts * 32) >> 4), kIdQK,
                      (k | kk) != 0 ? 1u : 0u);
      }
      if (!ok) break;
      umma_commit(&ctl.s_full);
    }
    if (j == 0) QMLA_TRACE(12, it);
    if (!(ok = twait(&ctl.p_full, it & 1u, ctl, kSiteMmaPFull, p.dev_err))) break;
    if (*reinterpret_cast<volatile uint32_t*>(&ctl.resc_tile) == it + 1) {
      if (!(ok = twait(&ctl.p_fixed, nresc & 1u, ctl, kSiteMmaPFull, p.dev_err))) break;
      ++nresc;
    }
    if (j == 0) QMLA_TRACE(14, it);
    if (j == 0 && ti.last) {
      // The softmax only signals P after every QK partial of this tile has
      // completed, so the query tile is free: start copying the next
      // segment's query now.
      Sched nx = sc;
      nx.next();
      if (nx.valid()) issue_query<HG>(p, nx.u, qsmem, ctl);
    }
    if (ti.first && seg > 0 && !(ok = twait(&ctl.o_free, (seg - 1) & 1u, ctl, kSiteMmaOFree, p.dev_err))) break;
    tc_fence_after();
    // O^T[c, h] += sum_t C_hat[t, c] P^T[t, h] for this issuer's 128 channels, K = 128 tokens.
    const uint32_t acc0 = ti.first ? 0u : 1u;
#pragma unroll
    for (int kk = 0; kk < 8; ++kk)
      umma_f16_ss(t_o, pv_a0 + static_cast<uint64_t>((kk * 2048) >> 4),
                  pv_b0 + static_cast<uint64_t>((kk * 2 * kSboP) >> 4), kIdPV, kk == 0 ? acc0 : 1u);
    umma_commit(&ctl.pv_done);
    if (j == kIssuers - 1) {
      // Row sums of P: L[m, h] += sum_t 1 * P^T[t, h] for every row m, with an
      // all-ones A operand in TMEM. Committed on their own barrier so that the
      // PV completion the dequantisation waits for does not wait for them; they
      // run while the next tile's first chunks are written.
#pragma unroll
      for (int kk = 0; kk < 8; ++kk)
        umma_f16_ts(tmem + Cfg<HG>::kColL, tmem + Cfg<HG>::kColOnes,
                    pv_b0 + static_cast<uint64_t>((kk * 2 * kSboP) >> 4), kIdL, kk == 0 ? acc0 : 1u);
      umma_commit(&ctl.rs_done);
    }
    QMLA_TRACE(24 + j, it);
    if (j == 0) QMLA_TRACE(15, it);
    ++it;
    if (ti.last) ++seg;
  }
  if (!ok) set_abort(ctl, p.dev_err);
  // Every MMA and copy must have landed before TMEM and shared memory are
  // released; this wait ignores the abort flag.
  umma_commit(&ctl.fin);
  wait_ok(mbar_wait(&ctl.fin, 0, kWaitNs, nullptr), kSiteMmaFin, ctl, p.dev_err);
}

template <int CB, int HG, bool PROT>
__global__ void __launch_bounds__(kThreads, 1) decode_main(const Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t chunks = smem_u32(smem);
  uint8_t* qsmem = smem + kNumChunks * kChunkBytes;
  Ctrl& ctl = *reinterpret_cast<Ctrl*>(smem + kNumChunks * kChunkBytes + Cfg<HG>::kQBytes);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    QMLA_TRACE(22, 0);
    QMLA_TRACE_CTA(0, globaltimer_ns());
    uint32_t smid;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(smid));
    QMLA_TRACE_CTA(2, smid);
  }

  if (threadIdx.x == 0) {
    // chunk k is written by the 4 warps of its parity; the packed caches split
    // the RoPE chunk (k = 8) over all 8 workers
    for (int k = 0; k < kNumChunks; ++k) mbar_init(&ctl.chunk_full[k], k == 8 && CB != 16 ? 8 : 4);
    mbar_init(&ctl.pv_done, kIssuers);
    mbar_init(&ctl.s_full, kQkParts);
    mbar_init(&ctl.rs_done, 1);
    mbar_init(&ctl.p_full, kWorkers);
    mbar_init(&ctl.p_fixed, kWorkers);
    ctl.resc_tile = 0u;
    mbar_init(&ctl.o_free, kWorkers);
    mbar_init(&ctl.q_full, 1);
    mbar_init(&ctl.fin, kIssuers);
    mbar_init(&ctl.grp, kWorkers);
    ctl.abort = 0u;
    fence_mbar_init();
  }
  if (warp == 0) {  // worker warp 0 owns the TMEM allocation
    tmem_alloc(&ctl.tmem_base, Cfg<HG>::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctl.tmem_base;
  if (warp < 4) {  // the all-ones A operand of the row-sum MMAs, each warp its lane quarter
    uint32_t r[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) r[i] = 0x3c003c00u;  // fp16 pair (1, 1)
    tmem_st(tmem + (static_cast<uint32_t>(warp * 32) << 16) + Cfg<HG>::kColOnes, r);
    tmem_st_wait();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp >= kWorkers && lane != 0) return;  // each MMA role is a single thread
  // The set-up above may overlap the prep kernel; everything below reads what
  // prep and the cache writer before it produced.
  griddep_wait();

  Sched sc;
  sc.init(p.prefix, p.cta_info[blockIdx.x], p.batch * p.n_hg, blockIdx.x, gridDim.x);
  if (warp < kWorkers) {
    worker_role<CB, HG, PROT>(p, sc, chunks, ctl, tmem, warp, lane);
  } else {
    mma_issuer<HG>(p, sc, chunks, qsmem, ctl, tmem, warp - kWorkers);
  }
  griddep_launch_dependents();  // the merge may be scheduled as CTAs finish
  tc_fence_before();
  __syncthreads();  // the exited lanes of the MMA warps do not take part
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, Cfg<HG>::kTmemCols);
  }
  if (threadIdx.x == 0) {
    QMLA_TRACE(23, 0);
    QMLA_TRACE_CTA(1, globaltimer_ns());
    QMLA_TRACE_CTA(3, static_cast<unsigned long long>(sc.t1 - sc.t0));
  }
}

// ------------------------------------------------------------ prep / combine
constexpr int kPrepThreads = 1024;

// Block 0: tile prefix over units (u = b * n_hg + hg), tiles = ceil(len / 128).
// Blocks 1..: one query-image piece (16 bytes) per thread.
template <int CB, int HG>
__global__ void __launch_bounds__(kPrepThreads) prep_kernel(const Params p) {
  griddep_launch_dependents();  // the main kernel may start its set-up meanwhile
  if (blockIdx.x > 0) {
    const long long idx = static_cast<long long>(blockIdx.x - 1) * kPrepThreads + threadIdx.x;
    constexpr int kPieces = kNumChunks * HG * 8;
    const long long units = static_cast<long long>(p.batch) * p.n_hg;
    if (idx >= units * kPieces) return;
    const int u = static_cast<int>(idx / kPieces);
    const int b = u / p.n_hg;
    query_piece<CB, HG>(p, p.qimg + static_cast<size_t>(u) * Cfg<HG>::kQBytes, b, (u - b * p.n_hg) * HG,
                        static_cast<int>(idx - static_cast<long long>(u) * kPieces));
    return;
  }
  constexpr int kSmemUnits = 4096;  // prefixes kept on chip for the per-CTA searches
  __shared__ int warp_sums[32];
  __shared__ int carry;
  __shared__ int pf_s[kSmemUnits + 1];
  const bool pf_on_chip = p.batch * p.n_hg < kSmemUnits;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nwarps = blockDim.x >> 5;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  for (int base = 0; base < p.batch; base += blockDim.x) {
    const int b = base + threadIdx.x;
    int tiles = 0;
    if (b < p.batch) {
      int len = p.seq_lens[b];
      if (len < 0 || len > p.max_blocks * kBlockTokens) {
        report(p.dev_err, QMLA_DEVERR_BAD_POSITION);
        len = 0;
      }
      tiles = (len + kTileTokens - 1) / kTileTokens;
    }
    const int v = tiles * p.n_hg;
    int x = v;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, off);
      if (lane >= off) x += y;
    }
    if (lane == 31) warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
      int sw = lane < nwarps ? warp_sums[lane] : 0;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, sw, off);
        if (lane >= off) sw += y;
      }
      warp_sums[lane] = sw;
    }
    __syncthreads();
    const int excl = carry + (warp > 0 ? warp_sums[warp - 1] : 0) + x - v;
    if (b < p.batch) {
      for (int hg = 0; hg < p.n_hg; ++hg) {
        p.prefix_w[b * p.n_hg + hg] = excl + hg * tiles;
        if (pf_on_chip) pf_s[b * p.n_hg + hg] = excl + hg * tiles;
      }
    }
    __syncthreads();
    if (threadIdx.x == blockDim.x - 1) carry = excl + v;
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    p.prefix_w[p.batch * p.n_hg] = carry;
    if (pf_on_chip) pf_s[p.batch * p.n_hg] = carry;
  }
  __syncthreads();
  // The unit holding the first tile of every decode CTA's range (the unit u
  // with prefix[u] <= t0 < prefix[u + 1]), so that no CTA has to search.
  const volatile int32_t* pf = pf_on_chip ? pf_s : p.prefix_w;
  const int units = p.batch * p.n_hg;
  const int T = pf[units];
  for (int c = threadIdx.x; c < p.grid; c += blockDim.x) {
    const int t0 = static_cast<int>(static_cast<long long>(c) * T / p.grid);
    int lo = 0, hi = units;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (pf[mid] <= t0) lo = mid; else hi = mid;
    }
    const int pu0 = pf[lo], pu1 = pf[lo + 1];
    p.cta_info[c] = make_int4(lo, pu0, pu1, T);
    // The first tile's block-table entries (clamped column, like row_ref) and length.
    const int b = lo / p.n_hg;
    const int j = t0 - pu0;
    const int32_t* trow = p.table + static_cast<size_t>(b) * p.max_blocks;
    const bool any = t0 < static_cast<int>(static_cast<long long>(c + 1) * T / p.grid);
    p.cta_first[c] = any ? make_int4(trow[min(2 * j, p.max_blocks - 1)], trow[min(2 * j + 1, p.max_blocks - 1)],
                                     p.seq_lens[b], j)
                         : make_int4(-1, -1, 0, 0);
    p.cta_t0[c] = t0;
  }
  if (threadIdx.x == 0) p.cta_t0[p.grid] = T;
  // prep reads nothing the cache writer before it writes, but the main kernel
  // waits only for prep: prep does not complete before the writer has.
  griddep_wait();
}

// The CTA whose range holds tile t (CTA c's range starts at c * T / grid).
__device__ __forceinline__ int cta_of(int t, int T, int grid) {
  return static_cast<int>((static_cast<long long>(t + 1) * grid - 1) / T);
}

// Merges the partials of split units with the App. C.5 rule, as a running
// merge: M = max m_j, l = sum 2^(m_j - M) l_j, O = sum 2^(m_j - M) o_j / l (the
// running form rescales by 2^(M_old - M_new) when M grows). One block per
// (unit, 4 heads), a warp per head, 16 channels per thread; the loads of the
// next partial do not depend on the previous one's arithmetic.
template <int HG>
__global__ void __launch_bounds__(128) combine_kernel(const Params p) {
  griddep_wait();  // the partials of the main kernel
  const int u = blockIdx.x;
  const int h = blockIdx.y * 4 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  const int units = p.batch * p.n_hg;
  const int b = u / p.n_hg;
  const int h0 = (u - b * p.n_hg) * HG;
  if (h >= HG || h0 + h >= p.heads) return;
  const int P0 = p.prefix[u], P1 = p.prefix[u + 1], T = p.prefix[units];
  float4* out = reinterpret_cast<float4*>(p.out + (static_cast<size_t>(b) * p.heads + h0 + h) * kDc) + lane * 4;
  if (P0 == P1) {
#pragma unroll
    for (int v = 0; v < 4; ++v) out[v] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (p.lse != nullptr && lane == 0) p.lse[static_cast<size_t>(b) * p.heads + h0 + h] = -INFINITY;
    return;
  }
  const int c0 = cta_of(P0, T, p.grid), c1 = cta_of(P1 - 1, T, p.grid);
  if (c0 == c1) return;  // one CTA covered the whole unit and wrote the result
  float M = -INFINITY, l = 0.0f;
  float4 acc[4];
#pragma unroll
  for (int v = 0; v < 4; ++v) acc[v] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 2
  for (int c = c0; c <= c1; ++c) {
    if (p.cta_t0[c] == p.cta_t0[c + 1]) continue;  // an empty range wrote no partial
    const size_t pi = (static_cast<size_t>(c) + u) * HG + h;
    const float2 ml = *reinterpret_cast<const float2*>(p.part_ml + pi * 2);
    const float4* o = reinterpret_cast<const float4*>(p.part_o + pi * kDc) + lane * 4;
    float4 ov[4];
#pragma unroll
    for (int v = 0; v < 4; ++v) ov[v] = o[v];
    const float Mn = fmaxf(M, ml.x);
    // A partial that saw no key for this head has m = -inf and l = o = 0.
    const float a = M == Mn ? 1.0f : exp2f(M - Mn), w = ml.x == Mn ? 1.0f : exp2f(ml.x - Mn);
    l = l * a + w * ml.y;
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      acc[v].x = acc[v].x * a + w * ov[v].x;
      acc[v].y = acc[v].y * a + w * ov[v].y;
      acc[v].z = acc[v].z * a + w * ov[v].z;
      acc[v].w = acc[v].w * a + w * ov[v].w;
    }
    M = Mn;
  }
  const float inv = l > 0.0f ? 1.0f / l : 0.0f;
#pragma unroll
  for (int v = 0; v < 4; ++v) out[v] = make_float4(acc[v].x * inv, acc[v].y * inv, acc[v].z * inv, acc[v].w * inv);
  if (lane == 0 && p.lse != nullptr) p.lse[static_cast<size_t>(b) * p.heads + h0 + h] = (M + log2f(l)) * kLn2;
}

// The same merge for launches with few units, each split over many CTAs (long
// contexts): one block per (unit, head) of kWideGroups x 128 threads. Thread i
// of the first pass holds piece c0 + i's (m, l); block reductions give M and l
// and the pieces' weights 2^(m_j - M) go to shared memory. Group g then sums
// pieces c0 + g, c0 + g + kWideGroups, ... for its float4 of every head row,
// with the loads of several pieces in flight, and the groups' sums are added.
constexpr int kWideGroups = 4;
constexpr int kWideThreads = kWideGroups * 128;

template <int HG>
__global__ void __launch_bounds__(kWideThreads) combine_wide_kernel(const Params p) {
  griddep_wait();  // the partials of the main kernel
  __shared__ float red[kWideThreads / 32];
  __shared__ float wts[kWideThreads];
  __shared__ float4 part[kWideGroups - 1][128];
  const int u = blockIdx.x;
  const int h = blockIdx.y;
  const int units = p.batch * p.n_hg;
  const int b = u / p.n_hg;
  const int h0 = (u - b * p.n_hg) * HG;
  if (h0 + h >= p.heads) return;
  const int P0 = p.prefix[u], P1 = p.prefix[u + 1], T = p.prefix[units];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int v = tid & 127, grp = tid >> 7;
  float4* out = reinterpret_cast<float4*>(p.out + (static_cast<size_t>(b) * p.heads + h0 + h) * kDc) + v;
  if (P0 == P1) {
    if (grp == 0) *out = make_float4(0.f, 0.f, 0.f, 0.f);
    if (p.lse != nullptr && tid == 0) p.lse[static_cast<size_t>(b) * p.heads + h0 + h] = -INFINITY;
    return;
  }
  const int c0 = cta_of(P0, T, p.grid), c1 = cta_of(P1 - 1, T, p.grid);
  if (c0 == c1) return;  // one CTA covered the whole unit and wrote the result
  // pieces c0..c1 <= grid <= kWideThreads: one per thread
  const int c = c0 + tid;
  float2 ml = make_float2(-INFINITY, 0.0f);
  if (c <= c1 && p.cta_t0[c] != p.cta_t0[c + 1])  // an empty range wrote no partial
    ml = __ldcg(reinterpret_cast<const float2*>(p.part_ml) + (static_cast<size_t>(c) + u) * HG + h);
  float x = ml.x;
#pragma unroll
  for (int s = 16; s >= 1; s >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, s));
  if (lane == 0) red[warp] = x;
  __syncthreads();
  float M = red[0];
#pragma unroll
  for (int i = 1; i < kWideThreads / 32; ++i) M = fmaxf(M, red[i]);
  const bool any = M != -INFINITY;  // some piece saw a key
  const float w = any && ml.x != -INFINITY ? exp2f(ml.x - M) : 0.0f;
  wts[tid] = w;
  float y = w * ml.y;
#pragma unroll
  for (int s = 16; s >= 1; s >>= 1) y += __shfl_xor_sync(0xffffffffu, y, s);
  __syncthreads();  // every thread has read red for M
  if (lane == 0) red[warp] = y;
  __syncthreads();
  float L = 0.0f;
#pragma unroll
  for (int i = 0; i < kWideThreads / 32; ++i) L += red[i];
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  const float4* ob = reinterpret_cast<const float4*>(p.part_o) + v;
#pragma unroll 4
  for (int cc = c0 + grp; cc <= c1; cc += kWideGroups) {
    const float wc = wts[cc - c0];
    const float4 o = __ldcg(ob + ((static_cast<size_t>(cc) + u) * HG + h) * (kDc / 4));
    if (wc != 0.0f) {  // a piece that wrote nothing is never multiplied in
      acc.x += wc * o.x;
      acc.y += wc * o.y;
      acc.z += wc * o.z;
      acc.w += wc * o.w;
    }
  }
  if (grp > 0) part[grp - 1][v] = acc;
  __syncthreads();
  if (grp == 0) {
#pragma unroll
    for (int g = 0; g < kWideGroups - 1; ++g) {
      const float4 q = part[g][v];
      acc.x += q.x;
      acc.y += q.y;
      acc.z += q.z;
      acc.w += q.w;
    }
    const float inv = L > 0.0f ? 1.0f / L : 0.0f;
    *out = make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
    if (tid == 0 && p.lse != nullptr)
      p.lse[static_cast<size_t>(b) * p.heads + h0 + h] = any ? (M + log2f(L)) * kLn2 : -INFINITY;
  }
}

// Test hook: the fp16 tile the decode kernel builds for tile j (tokens 128 j ..
// 128 j + 127) of sequence b, made by the same row loaders (packed rows
// dequantised, protected rows and BF16 rows converted) into the same swizzled
// chunks, then written out row-major in channel order: out [128][576] fp16,
// rows past the sequence end zero.
template <int CB, bool PROT>
__global__ void __launch_bounds__(kTileTokens) tile_dump_kernel(const Params p, int b, int j, uint16_t* out) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t chunks = smem_u32(smem);
  const int row = threadIdx.x;
  const int slot = row & 63;
  RowRef r;
  r.has = true;
  r.b = b;
  r.j = j;
  r.len = p.seq_lens[b];
  r.entry = p.table[static_cast<size_t>(b) * p.max_blocks + min(2 * j + (row >= 64 ? 1 : 0), p.max_blocks - 1)];
  bool valid = false;
  const uint8_t* ps = PROT ? prot_row(p, r, row) : nullptr;
  const uint8_t* blk = resolve_row<CB>(p, r, row, valid);
#pragma unroll 1
  for (int k = 0; k < kNumChunks; ++k) {
    const uint32_t cbase = chunks + k * kChunkBytes;
    if constexpr (CB == 16) {
      uint4 v[8];
#pragma unroll
      for (int i = 0; i < 8; ++i)
        v[i] = valid ? ldg_nc_v4(blk + slot * (kDqk * 2) + k * 128 + i * 16) : make_uint4(0, 0, 0, 0);
      store_row_bf16(cbase, row, v, valid);
    } else {
      const Fetch f = fetch_chunk<CB>(blk, valid && ps == nullptr, k, slot);
      dq_row<CB, PROT>(cbase, row, k, ps, f);
    }
  }
  __syncthreads();
#pragma unroll 1
  for (int k = 0; k < kNumChunks; ++k) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      uint32_t w[4];
      asm volatile("ld.shared.v4.b32 {%0,%1,%2,%3}, [%4];"
                   : "=r"(w[0]), "=r"(w[1]), "=r"(w[2]), "=r"(w[3])
                   : "r"(chunks + k * kChunkBytes + swz_off(row, i, 128)));
      const uint16_t* h = reinterpret_cast<const uint16_t*>(w);
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const int ch = CB == 16 ? e : (k == 8 ? Perm<4>::at(e) : Perm<CB>::at(e));
        out[static_cast<size_t>(row) * kDqk + k * 64 + i * 8 + ch] = h[e];
      }
    }
  }
}

template <int CB, bool PROT>
cudaError_t launch_tile_dump(const Params& prm, int b, int j, uint16_t* out, cudaStream_t stream) {
  constexpr int kSmem = 1024 + kNumChunks * kChunkBytes;
  cudaError_t e = cudaFuncSetAttribute(tile_dump_kernel<CB, PROT>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
  if (e != cudaSuccess) return e;
  tile_dump_kernel<CB, PROT><<<1, kTileTokens, kSmem, stream>>>(prm, b, j, out);
  return cudaGetLastError();
}

// Test hook: one warp waits, through the decode's own bounded wait, for a
// barrier phase that nothing completes; after limit_ns it reports
// QMLA_DEVERR_TIMEOUT and the wait site's bit in the error word and returns.
__global__ void __launch_bounds__(32) wait_timeout_kernel(uint32_t* dev_err, unsigned long long limit_ns) {
  __shared__ Ctrl ctl;
  if (threadIdx.x == 0) {
    mbar_init(&ctl.s_full, 1);  // never arrived on
    ctl.abort = 0u;
    fence_mbar_init();
  }
  __syncwarp();
  (void)wwait(&ctl.s_full, 0u, ctl, kSiteSmSFull, dev_err, limit_ns);
}

// Launches kern on stream; with pdl the launch may overlap the previous kernel
// in the stream (programmatic stream serialisation), which kern must wait for
// with griddep_wait before reading its results.
template <typename... Args>
cudaError_t launch_k(void (*kern)(Args...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream, bool pdl,
                     Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}


template <int CB, int HG, bool PROT>
cudaError_t launch_impl(const Params& prm, cudaStream_t stream, cudaEvent_t ev0, cudaEvent_t ev1) {
  static int configured_device = -1;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (configured_device != dev) {
    e = cudaFuncSetAttribute(decode_main<CB, HG, PROT>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<HG>::kSmem);
    if (e != cudaSuccess) return e;
    configured_device = dev;
  }
  // With measurement events around the main kernel every launch waits for the
  // previous one in full, so that the events bracket the main kernel alone.
  const bool pdl = ev0 == nullptr && ev1 == nullptr;
  const long long units = static_cast<long long>(prm.batch) * prm.n_hg;
  const long long pieces = units * kNumChunks * HG * 8;
  const unsigned prep_blocks = static_cast<unsigned>(1 + (pieces + kPrepThreads - 1) / kPrepThreads);
  if ((e = launch_k(prep_kernel<CB, HG>, dim3(prep_blocks), dim3(kPrepThreads), 0, stream, pdl, prm)) != cudaSuccess)
    return e;
  if (ev0 != nullptr && (e = cudaEventRecord(ev0, stream)) != cudaSuccess) return e;
  if ((e = launch_k(decode_main<CB, HG, PROT>, dim3(prm.grid), dim3(kThreads), Cfg<HG>::kSmem, stream, pdl, prm)) !=
      cudaSuccess)
    return e;
  if (ev1 != nullptr && (e = cudaEventRecord(ev1, stream)) != cudaSuccess) return e;
  // Few units split over many CTAs each (long contexts): spread each unit's
  // pieces over more threads; otherwise one warp per head.
  if (units * 4 < prm.grid && prm.grid <= kWideThreads) {
    return launch_k(combine_wide_kernel<HG>, dim3(static_cast<unsigned>(units), HG), dim3(kWideThreads), 0, stream,
                    pdl, prm);
  }
  return launch_k(combine_kernel<HG>, dim3(static_cast<unsigned>(units), (HG + 3) / 4), dim3(128), 0, stream, pdl,
                  prm);
}

template <int CB, bool PROT>
cudaError_t launch_hg(int hg, const Params& prm, cudaStream_t stream, cudaEvent_t ev0, cudaEvent_t ev1) {
  if (hg == 16) return launch_impl<CB, 16, PROT>(prm, stream, ev0, ev1);
  if (hg == 32) return launch_impl<CB, 32, PROT>(prm, stream, ev0, ev1);
  return launch_impl<CB, 64, PROT>(prm, stream, ev0, ev1);
}

}  // namespace

#ifdef QMLA_TRACE_BUILD
unsigned long long* g_trace_buf = nullptr;  // set by set_trace_buffer
#endif

int head_group_size(int heads) { return heads <= 16 ? 16 : (heads <= 32 ? 32 : 64); }

DecodeWorkspace decode_workspace_layout(int batch, int heads, int grid) {
  const int hg = head_group_size(heads);
  const size_t units = static_cast<size_t>(batch) * ((heads + hg - 1) / hg);
  auto up = [](size_t x) { return (x + 255) & ~static_cast<size_t>(255); };
  DecodeWorkspace w;
  w.prefix_off = 0;
  w.cta_off = up((units + 1) * sizeof(int32_t));
  w.part_o_off = w.cta_off + up(static_cast<size_t>(grid) * 2 * sizeof(int4) + (grid + 1) * sizeof(int32_t));
  const size_t nparts = static_cast<size_t>(grid) + units;
  w.part_ml_off = w.part_o_off + up(nparts * hg * kDc * sizeof(float));
  w.qimg_off = w.part_ml_off + up(nparts * hg * 2 * sizeof(float));
  w.total = w.qimg_off + up(units * kNumChunks * hg * 128);
  return w;
}

cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t stream) {
  const int hg = head_group_size(a.heads);
  const DecodeWorkspace w = decode_workspace_layout(a.batch, a.heads, a.grid);
  uint8_t* ws = static_cast<uint8_t*>(a.workspace);
  Params prm;
  prm.pool = static_cast<const uint8_t*>(a.pool);
  prm.prot = a.cache_kind == 16 ? nullptr : static_cast<const uint8_t*>(a.prot);
  prm.num_blocks = a.num_blocks;
  prm.q_lat = reinterpret_cast<const __nv_bfloat16*>(a.q_latent);
  prm.q_pe = reinterpret_cast<const __nv_bfloat16*>(a.q_pe);
  prm.batch = a.batch;
  prm.heads = a.heads;
  prm.n_hg = (a.heads + hg - 1) / hg;
  prm.q_tokens = a.q_tokens;
  prm.hpt = a.heads / a.q_tokens;
  prm.table = a.table;
  prm.max_blocks = a.max_blocks;
  prm.seq_lens = a.seq_lens;
  prm.scale_log2 = a.softmax_scale * 1.4426950408889634f;
  prm.out = a.out;
  prm.lse = a.lse;
  prm.prefix = reinterpret_cast<const int32_t*>(ws + w.prefix_off);
  prm.prefix_w = reinterpret_cast<int32_t*>(ws + w.prefix_off);
  prm.cta_info = reinterpret_cast<int4*>(ws + w.cta_off);
  prm.cta_first = prm.cta_info + a.grid;
  prm.cta_t0 = reinterpret_cast<int32_t*>(prm.cta_first + a.grid);
  prm.part_o = reinterpret_cast<float*>(ws + w.part_o_off);
  prm.part_ml = reinterpret_cast<float*>(ws + w.part_ml_off);
  prm.qimg = ws + w.qimg_off;
  prm.dev_err = a.dev_err;
  prm.grid = a.grid;
#ifdef QMLA_TRACE_BUILD
  prm.trace = g_trace_buf;
#else
  prm.trace = nullptr;
#endif
  const bool prot = prm.prot != nullptr;
  if (a.cache_kind == kC4R4)
    return prot ? launch_hg<kC4R4, true>(hg, prm, stream, a.ev_before_main, a.ev_after_main)
                : launch_hg<kC4R4, false>(hg, prm, stream, a.ev_before_main, a.ev_after_main);
  if (a.cache_kind == 4)
    return prot ? launch_hg<4, true>(hg, prm, stream, a.ev_before_main, a.ev_after_main)
                : launch_hg<4, false>(hg, prm, stream, a.ev_before_main, a.ev_after_main);
  if (a.cache_kind == 2)
    return prot ? launch_hg<2, true>(hg, prm, stream, a.ev_before_main, a.ev_after_main)
                : launch_hg<2, false>(hg, prm, stream, a.ev_before_main, a.ev_after_main);
  return launch_hg<16, false>(hg, prm, stream, a.ev_before_main, a.ev_after_main);
}

cudaError_t launch_tile_dump(const DecodeArgs& a, int b, int j, uint16_t* out, cudaStream_t stream) {
  Params prm{};
  prm.pool = static_cast<const uint8_t*>(a.pool);
  prm.prot = a.cache_kind == 16 ? nullptr : static_cast<const uint8_t*>(a.prot);
  prm.num_blocks = a.num_blocks;
  prm.batch = a.batch;
  prm.table = a.table;
  prm.max_blocks = a.max_blocks;
  prm.seq_lens = a.seq_lens;
  prm.dev_err = a.dev_err;
  const bool prot = prm.prot != nullptr;
  switch (a.cache_kind) {
    case 4: return prot ? launch_tile_dump<4, true>(prm, b, j, out, stream) : launch_tile_dump<4, false>(prm, b, j, out, stream);
    case 2: return prot ? launch_tile_dump<2, true>(prm, b, j, out, stream) : launch_tile_dump<2, false>(prm, b, j, out, stream);
    case kC4R4:
      return prot ? launch_tile_dump<kC4R4, true>(prm, b, j, out, stream)
                  : launch_tile_dump<kC4R4, false>(prm, b, j, out, stream);
    default: return launch_tile_dump<16, false>(prm, b, j, out, stream);
  }
}

cudaError_t launch_wait_timeout(uint32_t* dev_err, unsigned long long limit_ns, cudaStream_t stream) {
  wait_timeout_kernel<<<1, 32, 0, stream>>>(dev_err, limit_ns);
  return cudaGetLastError();
}

#ifdef QMLA_TRACE_BUILD
cudaError_t set_trace_buffer(void* buf) {
  g_trace_buf = static_cast<unsigned long long*>(buf);
  return cudaSuccess;
}
#endif

}  // namespace qmla
