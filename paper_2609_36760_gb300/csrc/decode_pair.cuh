// Cluster-pair decode for units of 128 query rows (heads) over the INT4 / INT2
// block (Eq. mla_compact; App. C.5 "cache update and tile reuse", "global
// attention normalization"). Included by decode.cu inside its anonymous
// namespace: it reuses that file's schedule, row loaders, dequantisation and
// prep / merge kernels.
//
// Two CTAs of a cluster walk the same tile range of the same units. CTA r
// (cluster rank) keeps one half of the channels:
//   content channels [256 r, 256 r + 256)  (four 64-channel chunks of the tile)
//   RoPE-key channels [32 r, 32 r + 32)    (one 32-channel half chunk)
// and TMEM holds, with the 128 heads on the 128 lanes (heads are the MMA M):
//   columns   0..255  O_r[h, c]  fp32, its 256 content channels
//   columns 256..383  S[h, t]    fp32 partial scores of the tile's 128 tokens,
//                                overwritten by P[h, t] fp16 (two per column)
//   columns 384..511  q[h, c]    fp16 query slice of its 256 content channels
// Per 128-token tile:
//   QK   S_r[h, t] = sum over its 288 channels of q[h, c] C_hat[t, c]:
//        16 MMAs with A = q from TMEM, B = the content chunks (K-major), and two
//        with A = the RoPE query half, B = the RoPE half chunk (both in shared
//        memory, 64-byte swizzle); M = 128 heads, N = 128 tokens.
//   Softmax, split by tokens: CTA r owns tokens [64 r, 64 r + 64) of the tile
//   for all 128 heads. Softmax warp (q, hh) (TMEM lane quarter q: heads
//   32 q .. 32 q + 31) owns the 32 tokens 64 r + 32 hh .. and sends this CTA's
//   partial scores of the peer's 32 tokens 64 (1 - r) + 32 hh .. to the peer's
//   warp (q, hh) (distributed shared memory), adds the peer's partial for its
//   own tokens, agrees the tile max with its partner warp and, through the P
//   message, with the peer, forms P = 2^(S scale log2e - m) in fp16 against the
//   per-head reference m (raised only when a score exceeds it by 2^8, as in
//   decode_main; P is sent optimistically against the current reference and
//   re-sent in the rare tile that raises it) and writes its own and the peer's
//   P over the scores in TMEM. Both CTAs sum the same fp16 weights in the same
//   order, so both hold the same row sums.
//   PV   O_r[h, c] += sum_t P[h, t] C_hat[t, c]: 8 MMAs with A = P from TMEM,
//        B = the same content chunks read MN-major, N = 256 channels.
// Dedicated warps dequantise the next tile into the second buffer while this
// one is in QK and softmax. Every wait is bounded; a wait that runs out
// records its site, stops both CTAs of the pair and they leave.
namespace pairk {

constexpr int kHeads = 128;                                     // query rows per unit (MMA M)
constexpr int kCChunks = 4;                                     // content chunks per CTA
constexpr int kRopeRow = 64;                                    // bytes per row of the RoPE half
constexpr int kBufBytes = kCChunks * kChunkBytes + kTileTokens * kRopeRow;  // 73728
constexpr int kQRopeBytes = kHeads * kRopeRow;                  // 8192
constexpr int kSWarps = 8;                                      // softmax warps (lane quarter x token half)
constexpr int kDqWarps = 4;                                     // dequantisation warps (a token row per thread)
constexpr int kPairMmaWarp = kSWarps + kDqWarps;                // one thread issues the MMAs
constexpr int kPairThreads = (kPairMmaWarp + 1) * 32;           // 416
constexpr int kSrecvBytes = kSWarps * 32 * 32 * 4;              // peer partial scores: [warp][8][lane][4 fp32]
constexpr int kPrecvBytes = kSWarps * 32 * 16 * 4;              // peer P: [warp][4][lane][8 fp16]
constexpr int kMrecvBytes = kSWarps * 32 * 4;                   // peer tile max: [warp][lane]
constexpr uint32_t kColO = 0, kColS = 256, kColQ = 384, kTmemCols = 512;
constexpr int kOffQRope = 2 * kBufBytes;
constexpr int kOffSrecv = kOffQRope + kQRopeBytes;
constexpr int kOffPrecv = kOffSrecv + kSrecvBytes;
constexpr int kOffMrecv = kOffPrecv + kPrecvBytes;
constexpr int kOffCtrl = kOffMrecv + kMrecvBytes;
static_assert(kBufBytes % 1024 == 0 && kOffQRope % 1024 == 0, "swizzle atom alignment");
static_assert((kCChunks * kChunkBytes) % 512 == 0, "64-byte swizzle alignment of the RoPE half");

struct __align__(16) Ctl {
  // full[b]: the tile in buffer b is dequantised (one arrive per dequantisation warp).
  // empty[b]: the PV that read buffer b has completed (MMA commit).
  uint64_t full[2], empty[2];
  uint64_t s_full, p_full, q_full, o_free, fin;
  // Arrived on by the peer's softmax warp w (every lane): its partial scores,
  // its P and tile max, its P again after a raised reference; done: the peer
  // no longer touches this CTA.
  uint64_t srecv[kSWarps], precv[kSWarps], precv2[kSWarps], done;
  uint64_t qbar[4];  // the two softmax warps of a TMEM lane quarter
  uint32_t tmem_base;
  uint32_t abort;
  alignas(16) float red[2][4][2][32];  // [use parity][lane quarter][token half][lane]
};
constexpr int kSmem = 1024 + kOffCtrl + static_cast<int>(sizeof(Ctl));
static_assert(kSmem <= 227 * 1024, "shared memory per CTA");

// Wait sites (bit 8 + site of the error word).
enum : uint32_t {
  kPsFull = 9, kPsEmpty, kPsS, kPsP, kPsQ, kPsO, kPsSrecv, kPsPrecv, kPsQbar, kPsFin, kPsDone
};

struct Peer {
  uint32_t rank, abort;  // cluster rank of the peer, its abort word
};

// Stops this CTA and the peer: every wait of either sees its abort word.
__device__ __forceinline__ void stop_pair(Ctl& c, const Peer& pr) {
  *reinterpret_cast<volatile uint32_t*>(&c.abort) = 1u;
  st_cluster_u32(pr.abort, 1u);
}
__device__ __forceinline__ bool chk(int r, uint32_t site, Ctl& c, const Peer& pr, uint32_t* dev_err) {
  if (r == 0) report(dev_err, QMLA_DEVERR_TIMEOUT | (0x100u << site));
  if (r != 1) stop_pair(c, pr);
  return r == 1;
}
// Warp-uniform bounded wait (every lane waits on the barrier itself).
__device__ __forceinline__ bool pwait(uint64_t* bar, uint32_t parity, Ctl& c, const Peer& pr, uint32_t site,
                                      uint32_t* dev_err, bool cluster_scope = false) {
  const int r = cluster_scope ? mbar_wait_cluster(bar, parity, kWaitNs, &c.abort)
                              : mbar_wait(bar, parity, kWaitNs, &c.abort);
  const bool all_ok = __all_sync(0xffffffffu, r == 1);
  if (r != 1) chk(r, site, c, pr, dev_err);
  return all_ok;
}
// Bounded wait of the single MMA thread.
__device__ __forceinline__ bool twait(uint64_t* bar, uint32_t parity, Ctl& c, const Peer& pr, uint32_t site,
                                      uint32_t* dev_err) {
  return chk(mbar_wait(bar, parity, kWaitNs, &c.abort), site, c, pr, dev_err);
}
// The two warps of lane quarter q meet (bounded); uses are counted per warp.
__device__ __forceinline__ bool quarter_sync(Ctl& c, int q, uint32_t& nq, const Peer& pr, uint32_t* dev_err,
                                             int lane) {
  __syncwarp();
  mbar_arrive_if(lane == 0 ? 1u : 0u, &c.qbar[q]);
  const bool ok = pwait(&c.qbar[q], nq & 1u, c, pr, kPsQbar, dev_err);
  ++nq;
  return ok;
}

// ------------------------------------------------------------ tile rows
// Packed rows of one token for this warp's chunks: content chunks th, th + 2
// of the CTA's half, and (th = 0) the CTA's half of the RoPE-key row.
struct Rows {
  Fetch c0, c1, pe;
};
template <int CB>
__device__ __forceinline__ void fetch_rows(Rows& f, const uint8_t* blk, bool valid, uint32_t rank, int th, int slot) {
  f.c0 = fetch_chunk<CB>(blk, valid, 4 * static_cast<int>(rank) + th, slot);
  f.c1 = fetch_chunk<CB>(blk, valid, 4 * static_cast<int>(rank) + th + 2, slot);
  if (th == 0) {
    f.pe.ok = valid;
    f.pe.a = make_uint4(0, 0, 0, 0);
    f.pe.b = f.pe.a;
    f.pe.sz = 0;
    f.pe.z = 0;
    if (valid) {
      using L = BlockLayout<CB>;
      f.pe.a = ldg_nc_v4(blk + L::code_off(8, slot) + 16 * rank);
      f.pe.sz = ldg_nc_u32(blk + L::sz_off(8, slot));
    }
  }
}
// 32 RoPE-key codes (16 bytes) of one row as RN_f16(s (q - z)) into the
// 64-byte-swizzled half chunk; the same within-piece order as the INT4 rows.
__device__ __forceinline__ void store_rope_half(uint32_t base, int row, const Fetch& f) {
  if (!f.ok) {
#pragma unroll
    for (int i = 0; i < 4; ++i) sts_v4(base + swz_off(row, i, kRopeRow), 0, 0, 0, 0);
    return;
  }
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
    sts_v4(base + swz_off(row, i, kRopeRow), dq2(__byte_perm(lo, K, 0x4140), zz, ss),
           dq2(__byte_perm(hi, K, 0x4140), zz, ss), dq2(__byte_perm(lo, K, 0x4342), zz, ss),
           dq2(__byte_perm(hi, K, 0x4342), zz, ss));
  }
}
template <int CB>
__device__ __forceinline__ void store_rows(const Rows& f, uint32_t buf, int row, int th) {
  store_row<CB>(buf + th * kChunkBytes, row, f.c0, CB == 4);
  store_row<CB>(buf + (th + 2) * kChunkBytes, row, f.c1, CB == 4);
  if (th == 0) store_rope_half(buf + kCChunks * kChunkBytes, row, f.pe);
}

// ------------------------------------------------------------- queries
// The query slice of head h of `unit` for this CTA: content channels
// [256 r + 128 th, +128) as fp16 pairs into TMEM columns 384 + 64 th .. +63
// (within-piece channel order of the tile rows), and the RoPE-query pieces
// 2 th, 2 th + 1 of channels [32 r, 32 r + 32) into the 64-byte-swizzled
// shared-memory tile. bf16 -> fp16 is exact for magnitudes in [2^-14, 65504].
template <int CB>
__device__ __forceinline__ void load_query(const Params& p, int unit, uint32_t t_q, uint32_t qrope, uint32_t rank,
                                           int h, int th) {
  const int b = unit / p.n_hg;
  const int v = (unit - b * p.n_hg) * kHeads + h;
  const size_t bh = static_cast<size_t>(b) * p.heads + v;
  const __nv_bfloat16* ql = p.q_lat + bh * kDc + 256 * rank + 128 * th;
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    uint32_t qk[32];
#pragma unroll
    for (int pc = 0; pc < 8; ++pc) {
      const uint4 raw = *reinterpret_cast<const uint4*>(ql + 64 * half + 8 * pc);
      const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
      float f[8];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        f[2 * e] = bf16_lo(w[e]);
        f[2 * e + 1] = bf16_hi(w[e]);
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) qk[4 * pc + e] = pack_h2(f[Perm<CB>::at(2 * e)], f[Perm<CB>::at(2 * e + 1)]);
    }
    tmem_st32(t_q + 64 * th + 32 * half, qk);
  }
  const __nv_bfloat16* qp = p.q_pe + bh * kDr + 32 * rank;
#pragma unroll
  for (int i = 2 * th; i < 2 * th + 2; ++i) {
    const uint4 raw = *reinterpret_cast<const uint4*>(qp + 8 * i);
    const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
    float f[8];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      f[2 * e] = bf16_lo(w[e]);
      f[2 * e + 1] = bf16_hi(w[e]);
    }
    uint32_t o[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) o[e] = pack_h2(f[Perm<4>::at(2 * e)], f[Perm<4>::at(2 * e + 1)]);
    sts_v4(qrope + swz_off(h, i, kRopeRow), o[0], o[1], o[2], o[3]);
  }
}

// O_r[h, cols 128 th .. +127] *= a (a rescale of the reference, rare).
__device__ __forceinline__ void scale_o(uint32_t t_o, float a) {
#pragma unroll 1
  for (int k = 0; k < 8; ++k) {
    uint32_t r[16];
    tmem_ld16(t_o + 16 * k, r);
    tmem_ld_wait();
#pragma unroll
    for (int e = 0; e < 16; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * a);
    tmem_st16(t_o + 16 * k, r);
  }
  tmem_st_wait();
}

// Adds 16 words of fp16 weight pairs to l in a fixed order (both CTAs sum
// the same values the same way, so both hold the same row sum).
__device__ __forceinline__ float add_weights(float l, const uint32_t (&w)[16]) {
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&w[k]));
    l += f.x;
    l += f.y;
  }
  return l;
}

// P of 32 scaled scores against the reference m: 2^(x - m) in fp16 pairs,
// 0 for the tokens at or past lim (masked or past the sequence end).
__device__ __forceinline__ void weights(uint32_t (&pk)[16], const float (&x)[32], float m, int lim) {
#pragma unroll
  for (int k = 0; k < 16; ++k)
    pk[k] = pack_h2(2 * k < lim ? ex2_approx(x[2 * k] - m) : 0.0f, 2 * k + 1 < lim ? ex2_approx(x[2 * k + 1] - m) : 0.0f);
}

// Segment end for the thread of head h (lane quarter q) and column half th:
// l = both token halves' row sums, then out = O / l over the CTA's channels
// (or the unnormalised partial), and LSE / (m, l) from `owner` (rank 0).
template <int CB>
__device__ bool epilogue(const Params& p, const SegEnd& e, Ctl& c, uint32_t t_row, uint32_t rank, bool owner,
                         int q, int th, int lane, float m_ref, float l_half, uint32_t& nq, const Peer& pr) {
  const uint32_t up = nq & 1u;
  c.red[up][q][th][lane] = l_half;
  if (!quarter_sync(c, q, nq, pr, p.dev_err, lane)) return false;
  const float l = c.red[up][q][0][lane] + c.red[up][q][1][lane];
  const float inv = l > 0.0f ? 1.0f / l : 0.0f;  // 0 for a head that saw no key
  const int h = 32 * q + lane;
  const int v = e.hg * kHeads + h;
  float* const orow = (e.whole ? p.out + (static_cast<size_t>(e.b) * p.heads + v) * kDc
                               : p.part_o + (e.pidx * kHeads + h) * kDc) +
                      256 * rank + 128 * th;
  const float f = e.whole ? inv : 1.0f;
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    uint32_t r[16];
    tmem_ld16(t_row + kColO + 128 * th + 16 * k, r);
    tmem_ld_wait();
#pragma unroll
    for (int pc = 0; pc < 2; ++pc) {
      float o8[8];
#pragma unroll
      for (int pos = 0; pos < 8; ++pos) o8[Perm<CB>::at(pos)] = __uint_as_float(r[8 * pc + pos]) * f;
      float4* dst = reinterpret_cast<float4*>(orow + 16 * k + 8 * pc);
      dst[0] = make_float4(o8[0], o8[1], o8[2], o8[3]);
      dst[1] = make_float4(o8[4], o8[5], o8[6], o8[7]);
    }
  }
  if (owner && th == 0) {
    if (e.whole) {
      if (p.lse != nullptr) p.lse[static_cast<size_t>(e.b) * p.heads + v] = (m_ref + log2f(l)) * kLn2;
    } else {
      p.part_ml[(e.pidx * kHeads + h) * 2 + 0] = m_ref;
      p.part_ml[(e.pidx * kHeads + h) * 2 + 1] = l;
    }
  }
  tc_fence_before();
  __syncwarp();
  mbar_arrive_if(lane == 0 ? 1u : 0u, &c.o_free);
  return true;
}

// ------------------------------------------------------- dequantisation
// Packed rows of one token for every chunk of this CTA's half: content chunks
// 0..3 and the RoPE-key half.
struct RowsAll {
  Fetch c[kCChunks];
  Fetch pe;
};
template <int CB>
__device__ __forceinline__ void fetch_all(RowsAll& f, const uint8_t* blk, bool valid, uint32_t rank, int slot) {
  Rows h;
#pragma unroll
  for (int th = 0; th < 2; ++th) {
    fetch_rows<CB>(h, blk, valid, rank, th, slot);
    f.c[th] = h.c0;
    f.c[th + 2] = h.c1;
    if (th == 0) f.pe = h.pe;
  }
}
template <int CB>
__device__ __forceinline__ void store_all(const RowsAll& f, uint32_t buf, int row) {
#pragma unroll
  for (int i = 0; i < kCChunks; ++i) store_row<CB>(buf + i * kChunkBytes, row, f.c[i], CB == 4);
  store_rope_half(buf + kCChunks * kChunkBytes, row, f.pe);
}

// Dequantisation warp d: token row 32 d + lane of every chunk. Tile `it` goes
// into buffer it & 1 once the PV of tile it - 2 has read that buffer; the
// packed rows of the next tile are loaded a tile ahead, its block-table
// entries a tile before that.
template <int CB>
__device__ void dequant_role(const Params& p, Sched sc, uint32_t sbase, Ctl& c, uint32_t rank, const Peer& pr,
                             int pair_id, int d, int lane) {
  const int row = 32 * d + lane, slot = row & 63;
  if (!sc.valid()) return;
  RowsAll f;
  {
    const int4 fr = p.cta_first[pair_id];  // tile 0's table entries, from the prep kernel
    RowRef r0;
    r0.has = true;
    r0.entry = row < 64 ? fr.x : fr.y;
    r0.len = fr.z;
    r0.j = fr.w;
    r0.b = sc.u / p.n_hg;
    bool v0 = false;
    const uint8_t* b0 = resolve_row<CB>(p, r0, row, v0);
    fetch_all<CB>(f, b0, v0, rank, slot);
  }
  Sched s1 = sc;  // the tile after the one being stored
  s1.next();
  RowRef r1 = row_ref(p, s1, row);
  uint32_t it = 0;
  for (; sc.valid(); sc.next()) {
    const uint32_t b = it & 1u;
    if (!pwait(&c.empty[b], ((it >> 1) & 1u) ^ 1u, c, pr, kPsEmpty, p.dev_err)) break;
    store_all<CB>(f, sbase + b * kBufBytes, row);
    bool v1 = false;
    const uint8_t* b1 = resolve_row<CB>(p, r1, row, v1);
    fetch_all<CB>(f, b1, v1, rank, slot);
    s1.next();
    r1 = row_ref(p, s1, row);
    fence_proxy_async_smem();
    __syncwarp();
    mbar_arrive_if(lane == 0 ? 1u : 0u, &c.full[b]);
    ++it;
  }
}

// ------------------------------------------------------------ softmax warps
// Trace builds: lane 0 of warps 0 and 2 records events 8.. and 16.. per tile.
#define PAIR_TRACE(k)                                                            \
  do {                                                                           \
    if (lane == 0 && (warp == 0 || warp == 2)) QMLA_TRACE(8 + 4 * warp + (k), it); \
  } while (0)

// Softmax warp w: TMEM lane quarter q = w & 3 (heads 32 q .. 32 q + 31), token
// half hh = w >> 2 of each CTA's 64 tokens. Token group g (tokens 32 g ..
// 32 g + 31 of the tile, K-steps 2 g and 2 g + 1 of the PV) is owned by warp
// (q, g & 1) of CTA g >> 1; this warp owns group 2 r + hh and relays group
// 2 (1 - r) + hh. It alone reads the scores of those two groups and writes
// their P (K-step k at columns 16 k .. 16 k + 7 of the score block), so P
// never overwrites scores another warp still has to read.
template <int CB>
__device__ void softmax_role(const Params& p, Sched sc, uint32_t sbase, Ctl& c, uint32_t tmem, uint32_t rank,
                             const Peer& pr, int pair_id, int warp, int lane) {
  const int q = warp & 3, hh = warp >> 2;
  const int h = 32 * q + lane;
  const int g_own = 2 * static_cast<int>(rank) + hh, g_rel = 2 * (1 - static_cast<int>(rank)) + hh;
  const uint32_t t_row = tmem + (static_cast<uint32_t>(32 * q) << 16);
  const uint32_t sr_loc = sbase + kOffSrecv + warp * 4096 + lane * 16;  // + 512 per 4 tokens
  const uint32_t pr_loc = sbase + kOffPrecv + warp * 2048 + lane * 16;  // + 512 per 8 tokens
  const uint32_t m_loc = sbase + kOffMrecv + (warp * 32 + lane) * 4;
  const uint32_t sr_peer = cluster_map(sr_loc, pr.rank);
  const uint32_t pr_peer = cluster_map(pr_loc, pr.rank);
  const uint32_t m_peer = cluster_map(m_loc, pr.rank);
  const uint32_t srb_peer = cluster_map(smem_u32(&c.srecv[warp]), pr.rank);
  const uint32_t prb_peer = cluster_map(smem_u32(&c.precv[warp]), pr.rank);
  const uint32_t pr2b_peer = cluster_map(smem_u32(&c.precv2[warp]), pr.rank);
  const uint32_t qrope = sbase + kOffQRope;
  const float sl2 = p.scale_log2;
  uint32_t it = 0, nq = 0, n2 = 0;
  float m_ref = -INFINITY, l_half = 0.0f;
  int seg_j0 = 0;
  bool ok = true;
  if (!sc.valid()) return;
  load_query<CB>(p, sc.u, t_row + kColQ, qrope, rank, h, hh);
  tmem_st_wait();
  fence_proxy_async_smem();
  tc_fence_before();
  __syncwarp();
  mbar_arrive_if(lane == 0 ? 1u : 0u, &c.q_full);

  for (; ok && sc.valid(); sc.next()) {
    const TileFlags tf = tile_flags(sc);
    if (tf.first) seg_j0 = sc.t - sc.pu0;
    PAIR_TRACE(0);
    if (!(ok = pwait(&c.s_full, it & 1u, c, pr, kPsS, p.dev_err))) break;
    tc_fence_after();
    PAIR_TRACE(3);
    const TileInfo ti = tile_info(sc, p);
    uint32_t s[32];
    // this CTA's partial scores of the relayed group to the peer's warp (q, hh)
    tmem_ld32(t_row + kColS + 32 * g_rel, s);
    tmem_ld_wait();
#pragma unroll
    for (int tg = 0; tg < 8; ++tg) st_cluster_v4(sr_peer + tg * 512, s[4 * tg], s[4 * tg + 1], s[4 * tg + 2], s[4 * tg + 3]);
    mbar_arrive_cluster(srb_peer);
    tmem_ld32(t_row + kColS + 32 * g_own, s);
    // Visible tokens of the own group: positions up to the head's query token
    // (Eq. mla_compact's causal mask; every cached position for one token).
    const int tq = (ti.hg * kHeads + h) / p.hpt;
    const int lim = min(max(ti.len - p.q_tokens + tq - kTileTokens * ti.j - 32 * g_own + 1, 0), 32);
    tmem_ld_wait();
    PAIR_TRACE(4);
    if (!(ok = pwait(&c.srecv[warp], it & 1u, c, pr, kPsSrecv, p.dev_err, true))) break;
    float x[32];
    float mx = -INFINITY;
#pragma unroll
    for (int tg = 0; tg < 8; ++tg) {
      const uint4 o = lds_v4(sr_loc + tg * 512);
      const uint32_t ov[4] = {o.x, o.y, o.z, o.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int i = 4 * tg + e;
        x[i] = (__uint_as_float(s[i]) + __uint_as_float(ov[e])) * sl2;
        if (i < lim) mx = fmaxf(mx, x[i]);
      }
    }
    // tile max of this CTA's 64 tokens (the partner warp holds the other 32)
    const uint32_t up = nq & 1u;
    c.red[up][q][hh][lane] = mx;
    if (!(ok = quarter_sync(c, q, nq, pr, p.dev_err, lane))) break;
    const float m_loc_max = fmaxf(c.red[up][q][0][lane], c.red[up][q][1][lane]);
    PAIR_TRACE(5);
    // P against the current reference (discarded if the tile raises it), with
    // the local tile max, to the peer's warp (q, hh)
    uint32_t pk[16];
    if (ti.first) {
#pragma unroll
      for (int k = 0; k < 16; ++k) pk[k] = 0u;
    } else {
      weights(pk, x, m_ref, lim);
    }
#pragma unroll
    for (int tg = 0; tg < 4; ++tg) st_cluster_v4(pr_peer + tg * 512, pk[4 * tg], pk[4 * tg + 1], pk[4 * tg + 2], pk[4 * tg + 3]);
    st_cluster_u32(m_peer, __float_as_uint(m_loc_max));
    mbar_arrive_cluster(prb_peer);
    PAIR_TRACE(6);
    if (!(ok = pwait(&c.precv[warp], it & 1u, c, pr, kPsPrecv, p.dev_err, true))) break;
    // The tile max over both CTAs; both compute the same reference.
    const float M = fmaxf(m_loc_max, lds_f32(m_loc));
    const bool resc = ti.first || M > m_ref + kRescaleLog2;
    float alpha = 1.0f;
    if (__any_sync(0xffffffffu, resc)) {
      // A new segment, or a score above the reference by more than 2^8 for
      // some head of this warp: its lanes move the reference (alpha =
      // 2^(m_old - m_new); 0 when no key was seen yet), recompute P and send
      // it again; the peer's warp takes the same branch for the same heads.
      if (resc) {
        if (!ti.first) alpha = exp2f(m_ref - M);
        m_ref = M;
      }
      weights(pk, x, m_ref, lim);
#pragma unroll
      for (int tg = 0; tg < 4; ++tg) st_cluster_v4(pr_peer + tg * 512, pk[4 * tg], pk[4 * tg + 1], pk[4 * tg + 2], pk[4 * tg + 3]);
      mbar_arrive_cluster(pr2b_peer);
      // O_r holds the sum through the previous tile (its PV completed before
      // this tile's QK started) and is scaled to the new reference.
      if (!ti.first && __any_sync(0xffffffffu, alpha != 1.0f)) scale_o(t_row + kColO + 128 * hh, alpha);
      if (!(ok = pwait(&c.precv2[warp], n2 & 1u, c, pr, kPsPrecv, p.dev_err, true))) break;
      ++n2;
    }
    uint32_t pp[16];  // the peer's P of the relayed group
#pragma unroll
    for (int tg = 0; tg < 4; ++tg) {
      const uint4 o = lds_v4(pr_loc + tg * 512);
      pp[4 * tg] = o.x;
      pp[4 * tg + 1] = o.y;
      pp[4 * tg + 2] = o.z;
      pp[4 * tg + 3] = o.w;
    }
    // Row sums in group order (group hh, then 2 + hh): the peer's warp (q, hh)
    // adds the same words in the same order.
    l_half = ti.first ? 0.0f : l_half * alpha;
    l_half = add_weights(l_half, rank == 0 ? pk : pp);
    l_half = add_weights(l_half, rank == 0 ? pp : pk);
    tmem_st8(t_row + kColS + 32 * g_own, *reinterpret_cast<const uint32_t(*)[8]>(&pk[0]));
    tmem_st8(t_row + kColS + 32 * g_own + 16, *reinterpret_cast<const uint32_t(*)[8]>(&pk[8]));
    tmem_st8(t_row + kColS + 32 * g_rel, *reinterpret_cast<const uint32_t(*)[8]>(&pp[0]));
    tmem_st8(t_row + kColS + 32 * g_rel + 16, *reinterpret_cast<const uint32_t(*)[8]>(&pp[8]));
    tmem_st_wait();
    tc_fence_before();
    __syncwarp();
    mbar_arrive_if(lane == 0 ? 1u : 0u, &c.p_full);
    PAIR_TRACE(7);

    if (ti.last) {
      // The next unit's queries first (this tile's QK, the last reader of the
      // query slice, has completed), so that its QK can overlap the results.
      Sched nx = sc;
      nx.next();
      if (nx.valid()) {
        load_query<CB>(p, nx.u, t_row + kColQ, qrope, rank, h, hh);
        tmem_st_wait();
        fence_proxy_async_smem();
        tc_fence_before();
        __syncwarp();
        mbar_arrive_if(lane == 0 ? 1u : 0u, &c.q_full);
      }
      SegEnd e;
      e.b = ti.b;
      e.hg = ti.hg;
      e.whole = (seg_j0 == 0) && (sc.t + 1 == sc.pu1);
      e.pidx = static_cast<size_t>(pair_id) + sc.u;
      if (!(ok = pwait(&c.empty[it & 1u], (it >> 1) & 1u, c, pr, kPsEmpty, p.dev_err))) break;
      tc_fence_after();
      if (!(ok = epilogue<CB>(p, e, c, t_row, rank, rank == 0, q, hh, lane, m_ref, l_half, nq, pr))) break;
    }
    ++it;
  }
  if (!ok && lane == 0) stop_pair(c, pr);
}

// ------------------------------------------------------------ MMA thread
template <int CB>
__device__ void mma_role(const Params& p, Sched sc, uint32_t sbase, Ctl& c, uint32_t tmem, const Peer& pr) {
  constexpr uint32_t kIdQK = idesc_f16_f32(128, 128, false, false);
  constexpr uint32_t kIdPV = idesc_f16_f32(128, 256, false, true);
  const uint32_t t_o = tmem + kColO, t_s = tmem + kColS, t_q = tmem + kColQ;
  const uint64_t qk_b0 = smem_desc(sbase, 16, 1024, SWZ_128B);
  const uint64_t pe_b0 = smem_desc(sbase + kCChunks * kChunkBytes, 16, 8 * kRopeRow, SWZ_64B);
  const uint64_t pe_a0 = smem_desc(sbase + kOffQRope, 16, 8 * kRopeRow, SWZ_64B);
  const uint64_t pv_b0 = smem_desc(sbase, kChunkBytes, 1024, SWZ_128B);
  uint32_t it = 0, seg = 0;
  bool ok = true;
  for (; ok && sc.valid(); sc.next()) {
    const TileFlags tf = tile_flags(sc);
    const uint32_t b = it & 1u;
    const uint64_t boff = static_cast<uint64_t>((b * kBufBytes) >> 4);
    QMLA_TRACE(0, it);
    if (tf.first && !(ok = twait(&c.q_full, seg & 1u, c, pr, kPsQ, p.dev_err))) break;
    if (!(ok = twait(&c.full[b], (it >> 1) & 1u, c, pr, kPsFull, p.dev_err))) break;
    // S and P share TMEM columns: the previous tile's PV must have read its P.
    if (it > 0 && !(ok = twait(&c.empty[b ^ 1u], ((it - 1) >> 1) & 1u, c, pr, kPsEmpty, p.dev_err))) break;
    tc_fence_after();
#pragma unroll
    for (int ks = 0; ks < 16; ++ks)
      umma_f16_ts(t_s, t_q + 8 * ks,
                  qk_b0 + boff + static_cast<uint64_t>(((ks >> 2) * kChunkBytes + (ks & 3) * 32) >> 4), kIdQK,
                  ks > 0 ? 1u : 0u);
#pragma unroll
    for (int ks = 0; ks < 2; ++ks)
      umma_f16_ss(t_s, pe_a0 + static_cast<uint64_t>((ks * 32) >> 4),
                  pe_b0 + boff + static_cast<uint64_t>((ks * 32) >> 4), kIdQK, 1u);
    QMLA_TRACE(4, it);
    umma_commit(&c.s_full);
    QMLA_TRACE(1, it);
    if (!(ok = twait(&c.p_full, it & 1u, c, pr, kPsP, p.dev_err))) break;
    QMLA_TRACE(2, it);
    if (tf.first && seg > 0 && !(ok = twait(&c.o_free, (seg - 1) & 1u, c, pr, kPsO, p.dev_err))) break;
    tc_fence_after();
    const uint32_t acc0 = tf.first ? 0u : 1u;
#pragma unroll
    for (int ks = 0; ks < 8; ++ks)
      umma_f16_ts(t_o, t_s + 16 * ks, pv_b0 + boff + static_cast<uint64_t>((ks * 2048) >> 4),
                  kIdPV, ks > 0 ? 1u : acc0);
    umma_commit(&c.empty[b]);
    QMLA_TRACE(3, it);
    ++it;
    if (tf.last) ++seg;
  }
  if (!ok) stop_pair(c, pr);
  // Every MMA must have landed before TMEM and shared memory are released;
  // this wait ignores the abort word.
  umma_commit(&c.fin);
  if (mbar_wait(&c.fin, 0, kWaitNs, nullptr) != 1) report(p.dev_err, QMLA_DEVERR_TIMEOUT | (0x100u << kPsFin));
}

template <int CB>
__global__ void __launch_bounds__(kPairThreads, 1) decode_pair(const Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  Ctl& c = *reinterpret_cast<Ctl*>(smem + kOffCtrl);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int pair_id = static_cast<int>(blockIdx.x >> 1);
  if (threadIdx.x == 0) {
    QMLA_TRACE_CTA(0, globaltimer_ns());
    uint32_t smid;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(smid));
    QMLA_TRACE_CTA(2, smid);
  }
  if (threadIdx.x == 0) {
    for (int b = 0; b < 2; ++b) {
      mbar_init(&c.full[b], kDqWarps);
      mbar_init(&c.empty[b], 1);
    }
    mbar_init(&c.s_full, 1);
    mbar_init(&c.p_full, kSWarps);
    mbar_init(&c.q_full, kSWarps);
    mbar_init(&c.o_free, kSWarps);
    mbar_init(&c.fin, 1);
    for (int w = 0; w < kSWarps; ++w) {  // the peer's softmax warp w, every lane
      mbar_init(&c.srecv[w], 32);
      mbar_init(&c.precv[w], 32);
      mbar_init(&c.precv2[w], 32);
    }
    mbar_init(&c.done, 1);
    for (int i = 0; i < 4; ++i) mbar_init(&c.qbar[i], 2);
    c.abort = 0u;
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(&c.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // the peer's barriers are initialised before any remote arrive
  tc_fence_after();
  const uint32_t tmem = c.tmem_base;
  Peer pr;
  pr.rank = rank ^ 1u;
  pr.abort = cluster_map(smem_u32(&c.abort), pr.rank);
  if (warp == kPairMmaWarp && lane != 0) return;  // the MMA role is a single thread
  griddep_wait();  // prep (and the cache writer before it)

  Sched sc;
  sc.init(p.prefix, p.cta_info[pair_id], p.batch * p.n_hg, pair_id, p.grid);
  if (warp < kSWarps) {
    softmax_role<CB>(p, sc, sbase, c, tmem, rank, pr, pair_id, warp, lane);
  } else if (warp < kPairMmaWarp) {
    dequant_role<CB>(p, sc, sbase, c, rank, pr, pair_id, warp - kSWarps, lane);
  } else {
    mma_role<CB>(p, sc, sbase, c, tmem, pr);
  }
  griddep_launch_dependents();
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0) {
    // This CTA no longer touches the peer's shared memory; it leaves once the
    // peer has said the same about this one.
    mbar_arrive_cluster(cluster_map(smem_u32(&c.done), pr.rank));
    if (mbar_wait_cluster(&c.done, 0u, kWaitNs, nullptr) != 1)
      report(p.dev_err, QMLA_DEVERR_TIMEOUT | (0x100u << kPsDone));
  }
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  if (threadIdx.x == 0) {
    QMLA_TRACE_CTA(1, globaltimer_ns());
    QMLA_TRACE_CTA(3, static_cast<unsigned long long>(sc.t1 - sc.t0));
  }
}

#undef PAIR_TRACE
}  // namespace pairk

// Launches kern with clusters of two CTAs (and programmatic stream
// serialisation when pdl is set).
template <typename... Args>
cudaError_t launch_pairs(void (*kern)(Args...), unsigned clusters, size_t smem, cudaStream_t stream, bool pdl,
                         Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * clusters);
  cfg.blockDim = dim3(pairk::kPairThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

// prep (block 0 only: no query image) -> decode_pair -> merge. prm.grid is set
// to the number of CTA pairs that can be resident at once (at most sms / 2).
template <int CB>
cudaError_t launch_pair_impl(Params prm, int sms, cudaStream_t stream, cudaEvent_t ev0, cudaEvent_t ev1) {
  static int configured_device = -1;
  static int clusters = 0;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (configured_device != dev) {
    e = cudaFuncSetAttribute(pairk::decode_pair<CB>, cudaFuncAttributeMaxDynamicSharedMemorySize, pairk::kSmem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * (sms / 2));
    cfg.blockDim = dim3(pairk::kPairThreads);
    cfg.dynamicSmemBytes = pairk::kSmem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    e = cudaOccupancyMaxActiveClusters(&n, pairk::decode_pair<CB>, &cfg);
    if (e != cudaSuccess) return e;
    if (n < 1) return cudaErrorInvalidConfiguration;
    clusters = n < sms / 2 ? n : sms / 2;
    configured_device = dev;
  }
  prm.grid = clusters;
  prm.n_hg = prm.heads / pairk::kHeads;
  const bool pdl = ev0 == nullptr && ev1 == nullptr;
  if ((e = launch_k(prep_kernel<CB, pairk::kHeads>, dim3(1), dim3(kPrepThreads), 0, stream, pdl, prm)) != cudaSuccess)
    return e;
  if (ev0 != nullptr && (e = cudaEventRecord(ev0, stream)) != cudaSuccess) return e;
  if ((e = launch_pairs(pairk::decode_pair<CB>, static_cast<unsigned>(clusters), pairk::kSmem, stream, pdl, prm)) !=
      cudaSuccess)
    return e;
  if (ev1 != nullptr && (e = cudaEventRecord(ev1, stream)) != cudaSuccess) return e;
  const long long units = static_cast<long long>(prm.batch) * prm.n_hg;
  if (units * 4 < prm.grid && prm.grid <= kWideThreads) {
    return launch_k(combine_wide_kernel<pairk::kHeads>, dim3(static_cast<unsigned>(units), pairk::kHeads),
                    dim3(kWideThreads), 0, stream, pdl, prm);
  }
  return launch_k(combine_kernel<pairk::kHeads>, dim3(static_cast<unsigned>(units), pairk::kHeads / 4), dim3(128), 0,
                  stream, pdl, prm);
}
