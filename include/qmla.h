/*
 * qmla — low-bit MLA decode attention on one GB300 (sm_103a).
 *
 * C ABI of the library libqmla.so. It implements the decode hot path of
 * QuantMLA (arXiv 2609.36760): Multi-head Latent Attention read directly from a
 * jointly low-bit paged cache, with unpacking and dequantisation fused into the
 * attention (Sec. 3.3; App. C.5).
 *
 *   qmla_quant_append   quantise + pack new tokens into the paged cache
 *                       (App. C.4 quantiser; App. C.5 "cache update": content- and
 *                       RoPE-cache quantisation, integer packing, slot-mapped
 *                       page insertion)
 *   qmla_mla_decode     split-KV decode attention over the packed cache, plus the
 *                       split-result combination (Eq. mla_compact; App. C.5
 *                       "global attention normalization")
 *   *_protected         the same with sink4/local128 BF16 protection (App. C.5)
 *   *_c4r4              the same over the paper's own 20,480-byte INT4 page
 *   qmla_mla_decode_multi  several query tokens per sequence under the causal mask
 *   qmla_mla_decode_ex  every decode variant from one descriptor, with optional
 *                       per-call events around the main kernel
 *
 * Conventions for every call
 * --------------------------
 * - Pointers named *_dev are device pointers owned by the caller; the library
 *   never allocates, frees or keeps them. Host pointers are marked _host.
 * - Every call that launches work is asynchronous on `stream` (a cudaStream_t;
 *   NULL = legacy default stream) and returns a status code immediately.
 *   Arguments are validated on the host before anything is launched; an invalid
 *   argument launches nothing.
 * - Problems only visible on the device (a bad block id, a position beyond the
 *   block table, a pipeline wait that ran out) are OR-ed into the caller's
 *   32-bit error word `dev_err_dev` (QMLA_DEVERR_*). The offending access is
 *   skipped; no call traps or aborts. Read the word with qmla_read_dev_err.
 * - bf16 / fp16 tensors are passed as uint16_t bit patterns.
 *
 * Cache format (this library's own 64-token block, little-endian)
 * ----------------------------------------------------------------
 * Each token is quantised in 9 groups of 64 coordinates: groups 0..7 are the
 * content latent c_KV channels [64g, 64g+64) at c_bits (4 or 2), group 8 is the
 * decoupled RoPE key k_pe (d_r = 64) at 4 bits. Per group, per token
 * (App. C.4, with the fp16 staging fixed by this library):
 *     d = RN_f32(x_max - x_min);  s = RN_f16(RN_f32(max(d, 1e-8) / m)), m = 2^b - 1
 *     (s = 2^-24 if that underflows to 0, 65504 if it overflows)
 *     z = clip(rne(-x_min / s), 0, m);  q = clip(rne(x / s + z), 0, m)
 * Codes are packed low bits first: INT4 byte j = q[2j] | q[2j+1] << 4, INT2
 * byte j = q[4j] | q[4j+1] << 2 | q[4j+2] << 4 | q[4j+3] << 6.
 * A block of 64 token slots, cb = 64 * c_bits / 8:
 *     [0, 8*64*cb)                 content codes   [group 8][slot 64][cb bytes]
 *     [8*64*cb, +2048)             RoPE-key codes  [slot 64][32 bytes]
 *     [8*64*cb + 2048, +2304)      scale/zero      [group 9][slot 64][fp16 s, fp16 z]
 * INT4 content: 20736 bytes per block; INT2 content: 12544 bytes per block.
 * Token at position p of sequence b lives in block block_table[b*max_blocks + p/64],
 * slot p % 64.
 *
 * The BF16 comparison cache (qmla_bf16_append / qmla_mla_decode_bf16cache)
 * stores each token as 576 bf16 (latent then k_pe): blocks of 64 x 1152 bytes,
 * the paper's BF16 page (App. C.5, storage layout).
 */
#ifndef QMLA_H_
#define QMLA_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* qmla_stream_t; /* same type as cudaStream_t */

/* Status codes returned by every call. */
enum qmla_status {
  QMLA_OK = 0,
  QMLA_ERR_INVALID_ARG = 1,          /* null pointer, bad size, bad bit width, misalignment */
  QMLA_ERR_UNSUPPORTED = 2,          /* no sm_103a device, or a shape outside the supported range */
  QMLA_ERR_WORKSPACE_TOO_SMALL = 3,  /* decode workspace smaller than qmla_decode_workspace_bytes */
  QMLA_ERR_CUDA = 4                  /* a CUDA runtime call failed; see qmla_last_cuda_error */
};

/* Bits of the device error word. */
enum qmla_device_error {
  QMLA_DEVERR_BAD_BLOCK = 1u,     /* a block-table entry outside [0, num_blocks) was needed */
  QMLA_DEVERR_BAD_POSITION = 2u,  /* a position or sequence length < 0 or beyond max_blocks*64 */
  QMLA_DEVERR_BAD_SEQ = 4u,       /* an append sequence id outside [0, num_seqs) */
  QMLA_DEVERR_TIMEOUT = 8u        /* an on-chip pipeline wait ran out; that kernel left early */
};

/* Most query tokens per sequence qmla_mla_decode_multi accepts. */
#define QMLA_MAX_Q_TOKENS 8

/* Bytes of one 64-token block for content bit width c_bits (4 -> 20736,
 * 2 -> 12544); 0 if c_bits is not supported. */
size_t qmla_block_bytes(int c_bits);

/* Bytes of one 64-token BF16 comparison block (73728). */
size_t qmla_bf16_block_bytes(void);

/*
 * Quantise n new tokens and insert them into the packed cache
 * (App. C.4 quantiser; App. C.5 fused writer without the BF16 protection
 * buffers).
 *
 *   pool_dev        [num_blocks * qmla_block_bytes(c_bits)] bytes, 32-byte aligned
 *                   (every call that takes a pool requires this: the decode
 *                   reads a token's 32-byte code row in one request);
 *                   only the slots of the given tokens are written
 *   c_bits          content bit width, 4 or 2 (the RoPE key is always 4-bit)
 *   latent_dev      [n, 512] bf16, row-major, 4-byte aligned: content latent c_KV
 *   k_pe_dev        [n, 64]  bf16, row-major, 4-byte aligned: decoupled RoPE key
 *   seq_ids_dev     [n] int32 sequence of each token, or NULL meaning token i
 *                   belongs to sequence i
 *   positions_dev   [n] int32 zero-based position of each token in its sequence
 *   block_table_dev [num_seqs, max_blocks] int32 physical block ids
 *   dev_err_dev     device error word (see above)
 * Two tokens with the same (sequence, position) in one call race; the result
 * is one of them. n == 0 is a no-op.
 */
int qmla_quant_append(void* pool_dev, int c_bits, int num_blocks, const uint16_t* latent_dev,
                      const uint16_t* k_pe_dev, const int32_t* seq_ids_dev,
                      const int32_t* positions_dev, int n, const int32_t* block_table_dev,
                      int num_seqs, int max_blocks, uint32_t* dev_err_dev, qmla_stream_t stream);

/* Same insertion into the BF16 comparison cache (blocks of qmla_bf16_block_bytes()):
 * the 576 bf16 values of each token are copied unchanged. */
int qmla_bf16_append(void* pool_dev, int num_blocks, const uint16_t* latent_dev,
                     const uint16_t* k_pe_dev, const int32_t* seq_ids_dev,
                     const int32_t* positions_dev, int n, const int32_t* block_table_dev,
                     int num_seqs, int max_blocks, uint32_t* dev_err_dev, qmla_stream_t stream);

/*
 * Sink4/local128 BF16 protection (App. C.5, "BF16 protection and cache
 * lifecycle"). For a request of L cached tokens the protected positions are
 *     P_L = {0, ..., min(4, L) - 1}  U  {max(0, L - 128), ..., L - 1};
 * attention reads their pre-quantisation bf16 content and RoPE-key values and
 * reads every other position from the packed cache, all under one softmax. A
 * packed copy is written for every token, protected or not, so a token leaving
 * the recent window switches to its packed copy with no further work.
 *
 * Protection buffer (caller-owned, one per request): [num_seqs][132][576] bf16,
 * qmla_protect_bytes_per_seq() = 132 * 576 * 2 = 152064 bytes per request (the
 * paper's figure), 16-byte aligned. A row holds a token's 512 latent values
 * then its 64 RoPE-key values; rows 0..3 hold sink positions 0..3, row
 * 4 + (p mod 128) holds recent position p. The buffer needs no initialisation:
 * a row is only read once the writer has filled it.
 */
size_t qmla_protect_bytes_per_seq(void);

/* qmla_quant_append plus the protection rows: token i (request s = seq_ids[i],
 * position p) is also copied into row p when p < 4 and into row 4 + (p mod 128)
 * when p >= seq_lens_dev[s] - 128, where seq_lens_dev [num_seqs] int32 holds the
 * requests' lengths after this call. So one call may carry a whole prefill:
 * positions older than the recent window never reach the ring, and no two
 * positions of one call share a row. latent_dev, k_pe_dev and prot_dev must be
 * 16-byte aligned; the other arguments and errors are those of qmla_quant_append. */
int qmla_quant_append_protected(void* pool_dev, int c_bits, int num_blocks, const uint16_t* latent_dev,
                                const uint16_t* k_pe_dev, const int32_t* seq_ids_dev,
                                const int32_t* positions_dev, int n, const int32_t* block_table_dev,
                                int num_seqs, int max_blocks, const int32_t* seq_lens_dev, void* prot_dev,
                                uint32_t* dev_err_dev, qmla_stream_t stream);

/* Workspace bytes qmla_mla_decode needs for this batch and head count on the
 * current device (split plan + split partials). For qmla_mla_decode_multi pass
 * heads = q_tokens x heads (up to 128 x QMLA_MAX_Q_TOKENS); 0 for bad arguments. */
size_t qmla_decode_workspace_bytes(int batch, int heads);

/*
 * Decode attention of one query token per sequence over the packed cache
 * (Eq. mla_compact with the dequantised cache s (q - z), App. C.4):
 *     S[b,h,t] = softmax_scale * (q_latent[b,h,:] . C_hat[b,t,:] + q_pe[b,h,:] . K_hat[b,t,:])
 *     out[b,h,:] = sum_t softmax_t(S[b,h,:]) C_hat[b,t,:]      (t < seq_lens[b])
 *     lse[b,h]   = log sum_t exp(S[b,h,t])
 * The caller applies the value/output up-projection. Sequences are split
 * across the GPU's SMs and the split results merged with the App. C.5 rule.
 *
 *   pool_dev        packed cache written by qmla_quant_append with the same c_bits,
 *                   32-byte aligned
 *   q_latent_dev    [batch, heads, 512] bf16 absorbed content query, 16-byte aligned
 *   q_pe_dev        [batch, heads, 64]  bf16 RoPE query, 16-byte aligned
 *   heads           1..128
 *   block_table_dev [batch, max_blocks] int32
 *   seq_lens_dev    [batch] int32 tokens to attend to (including any just appended)
 *   softmax_scale   tau, e.g. 1/sqrt(192)
 *   out_dev         [batch, heads, 512] float32
 *   lse_dev         [batch, heads] float32 natural-log LSE, or NULL
 *   workspace_dev   >= qmla_decode_workspace_bytes(batch, heads) bytes, 256-byte aligned;
 *                   contents need no initialisation and are scratch after the call
 * A sequence with seq_lens == 0 gets out = 0 and lse = -inf.
 */
int qmla_mla_decode(const void* pool_dev, int c_bits, int num_blocks, const uint16_t* q_latent_dev,
                    const uint16_t* q_pe_dev, int batch, int heads, const int32_t* block_table_dev,
                    int max_blocks, const int32_t* seq_lens_dev, float softmax_scale,
                    float* out_dev, float* lse_dev, void* workspace_dev, size_t workspace_bytes,
                    uint32_t* dev_err_dev, qmla_stream_t stream);

/* qmla_mla_decode under sink4/local128 protection: for request b with
 * L = seq_lens_dev[b], positions in P_L read row p (p < 4) or row 4 + (p mod 128)
 * of prot_dev[b] (rounded to fp16 like the BF16 cache path), every other
 * position the packed cache; one global softmax over all L positions. The
 * buffer must hold every protected position (qmla_quant_append_protected with
 * the same lengths leaves it so). prot_dev 16-byte aligned, non-null; outputs,
 * workspace and errors as qmla_mla_decode. */
int qmla_mla_decode_protected(const void* pool_dev, int c_bits, int num_blocks, const uint16_t* q_latent_dev,
                              const uint16_t* q_pe_dev, int batch, int heads, const int32_t* block_table_dev,
                              int max_blocks, const int32_t* seq_lens_dev, const void* prot_dev,
                              float softmax_scale, float* out_dev, float* lse_dev, void* workspace_dev,
                              size_t workspace_bytes, uint32_t* dev_err_dev, qmla_stream_t stream);

/* Decode with q_tokens query tokens per sequence (multi-token prediction,
 * speculative verification): Eq. mla_compact with its additive causal mask.
 * For sequence b with L = seq_lens_dev[b] cached tokens (the q_tokens new ones
 * included, written by the append beforehand), query token t sits at position
 * L - q_tokens + t and attends to positions [0, L - q_tokens + t]:
 *     S[b,t,h,p] = softmax_scale * (q_latent[b,t,h,:] . C_hat[b,p,:] + q_pe[b,t,h,:] . K_hat[b,p,:]),
 *                  p <= L - q_tokens + t
 *     out[b,t,h,:] = sum_p softmax_p(S[b,t,h,:]) C_hat[b,p,:];  lse[b,t,h] = log sum_p exp(S[b,t,h,p])
 * A query token with no admissible position (L - q_tokens + t < 0) gets out = 0,
 * lse = -inf. One pass over each sequence's cache serves all its query tokens:
 * the kernel treats the q_tokens x heads (token, head) pairs as heads.
 *
 *   q_latent_dev    [batch, q_tokens, heads, 512] bf16, 16-byte aligned
 *   q_pe_dev        [batch, q_tokens, heads, 64]  bf16, 16-byte aligned
 *   q_tokens        1 .. QMLA_MAX_Q_TOKENS; heads 1..128 per token
 *   prot_dev        NULL, or the sink4/local128 protection buffer (as
 *                   qmla_mla_decode_protected; P_L from the full length L)
 *   out_dev         [batch, q_tokens, heads, 512] float32
 *   lse_dev         [batch, q_tokens, heads] float32, or NULL
 *   workspace_dev   >= qmla_decode_workspace_bytes(batch, q_tokens * heads)
 * Other arguments, ownership and errors as qmla_mla_decode; q_tokens = 1 is
 * qmla_mla_decode. */
int qmla_mla_decode_multi(const void* pool_dev, int c_bits, int num_blocks, const uint16_t* q_latent_dev,
                          const uint16_t* q_pe_dev, int batch, int q_tokens, int heads,
                          const int32_t* block_table_dev, int max_blocks, const int32_t* seq_lens_dev,
                          const void* prot_dev, float softmax_scale, float* out_dev, float* lse_dev,
                          void* workspace_dev, size_t workspace_bytes, uint32_t* dev_err_dev,
                          qmla_stream_t stream);

/* The same decode over the BF16 comparison cache (same kernel, no dequantisation;
 * the paper's BF16 baseline, App. F.1). */
int qmla_mla_decode_bf16cache(const void* pool_dev, int num_blocks, const uint16_t* q_latent_dev,
                              const uint16_t* q_pe_dev, int batch, int heads,
                              const int32_t* block_table_dev, int max_blocks,
                              const int32_t* seq_lens_dev, float softmax_scale, float* out_dev,
                              float* lse_dev, void* workspace_dev, size_t workspace_bytes,
                              uint32_t* dev_err_dev, qmla_stream_t stream);

/*
 * The paper's own INT4 page ("C4R4": 4-bit content, 4-bit RoPE key; App. C.5,
 * storage layout; App. C.4, scale precisions). Same codes, groups and packing as
 * the c_bits = 4 block above; the metadata differ: per token and group a bf16
 * scale for content groups, an fp32 scale for the RoPE group, and a uint8 zero
 * point. Staging (App. C.4 with m = 15; d = RN_f32(x_max - x_min)):
 *     content  s = RN_bf16(RN_f32(max(d, 1e-8) / 15))
 *     RoPE     s = RN_f32(max(d, 1e-8) / 15)
 *     z = clip(rne(RN_f32(-x_min / s)), 0, 15);  q = clip(rne(RN_f32(RN_f32(x / s) + z)), 0, 15)
 * (for content groups the fp32 quotients give the exact-arithmetic codes, since
 * a bf16 x over a bf16 s is never within fp32 rounding of a half-integer).
 * A page of 64 token slots, 20480 bytes (320 per token):
 *     [0, 16384)       content codes   [group 8][slot 64][32 bytes]
 *     [16384, 18432)   RoPE-key codes  [slot 64][32 bytes]
 *     [18432, 19456)   content scales  [group 8][slot 64] bf16
 *     [19456, 19712)   RoPE scales     [slot 64] fp32
 *     [19712, 20288)   zero points     [group 9][slot 64] uint8 (group 8: RoPE key)
 *     [20288, 20480)   padding, never written or read
 * The decode's fp16 tile value of a code is RN_f16(s (q - z)) for content and
 * RN_f16(RN_f32(s (q - z))) for the RoPE key.
 */
size_t qmla_c4r4_page_bytes(void);

/* qmla_quant_append into pages of the paper's format (qmla_c4r4_page_bytes()
 * bytes each). prot_dev is optional: NULL writes the packed pages only; non-NULL
 * also writes the sink4/local128 protection rows as qmla_quant_append_protected
 * does, and then seq_lens_dev (lengths after this call) must be non-NULL and
 * latent_dev, k_pe_dev, prot_dev 16-byte aligned. Errors as qmla_quant_append. */
int qmla_quant_append_c4r4(void* pool_dev, int num_blocks, const uint16_t* latent_dev, const uint16_t* k_pe_dev,
                           const int32_t* seq_ids_dev, const int32_t* positions_dev, int n,
                           const int32_t* block_table_dev, int num_seqs, int max_blocks,
                           const int32_t* seq_lens_dev, void* prot_dev, uint32_t* dev_err_dev,
                           qmla_stream_t stream);

/* qmla_mla_decode over pages of the paper's format. prot_dev NULL attends over
 * the packed pages only; non-NULL (16-byte aligned) applies sink4/local128
 * protection as qmla_mla_decode_protected does. Outputs, workspace
 * (qmla_decode_workspace_bytes) and errors as qmla_mla_decode. */
int qmla_mla_decode_c4r4(const void* pool_dev, int num_blocks, const uint16_t* q_latent_dev,
                         const uint16_t* q_pe_dev, int batch, int heads, const int32_t* block_table_dev,
                         int max_blocks, const int32_t* seq_lens_dev, const void* prot_dev, float softmax_scale,
                         float* out_dev, float* lse_dev, void* workspace_dev, size_t workspace_bytes,
                         uint32_t* dev_err_dev, qmla_stream_t stream);

/*
 * Every decode variant above from one descriptor (Eq. mla_compact; App. C.5):
 * qmla_mla_decode, _protected, _c4r4, _multi and _bf16cache are this call with
 * some fields fixed. Fields:
 *   cache_kind      4 or 2 (this library's block at that content width),
 *                   QMLA_CACHE_C4R4 (the paper's page) or QMLA_CACHE_BF16
 *   pool, num_blocks, q_latent, q_pe, block_table, max_blocks, seq_lens,
 *   softmax_scale, out, lse, workspace, workspace_bytes, dev_err
 *                   as in qmla_mla_decode (q_latent / q_pe / out / lse shaped
 *                   [batch, q_tokens, heads, ...] when q_tokens > 1)
 *   batch, q_tokens, heads
 *                   q_tokens 1..QMLA_MAX_Q_TOKENS query tokens per sequence,
 *                   heads 1..128 per token (as qmla_mla_decode_multi)
 *   prot            sink4/local128 protection buffer or NULL (not with BF16)
 *   ev_before_main, ev_after_main
 *                   optional cudaEvent_t (NULL = none): recorded on `stream`
 *                   immediately before and after the main decode kernel of
 *                   this call only, so that a caller can time that kernel
 *                   with cudaEventElapsedTime. With either set, the call's
 *                   launches wait for one another in full instead of
 *                   overlapping their start-up, so that the events bracket
 *                   the main kernel alone. The library keeps no reference to
 *                   them after the call returns.
 * Returns QMLA_ERR_INVALID_ARG for a NULL descriptor or a bad field, else as
 * qmla_mla_decode. The descriptor is read during the call only.
 */
typedef struct qmla_decode_desc {
  const void* pool;
  int cache_kind;
  int num_blocks;
  const uint16_t* q_latent;
  const uint16_t* q_pe;
  int batch;
  int q_tokens;
  int heads;
  const int32_t* block_table;
  int max_blocks;
  const int32_t* seq_lens;
  const void* prot;
  float softmax_scale;
  float* out;
  float* lse;
  void* workspace;
  size_t workspace_bytes;
  uint32_t* dev_err;
  void* ev_before_main;
  void* ev_after_main;
} qmla_decode_desc;
int qmla_mla_decode_ex(const qmla_decode_desc* desc, qmla_stream_t stream);

/* Bytes of the fixed device scratch array qmla_mla_decode_static uses
 * (32 MiB). */
size_t qmla_static_scratch_bytes(void);

/*
 * qmla_mla_decode without a workspace argument, for callers that cannot
 * allocate device memory where they call it (for example code running inside
 * an allocator-free region of a serving loop, or a host library that is
 * handed finished buffers and must not call cudaMalloc, whose implicit
 * synchronisation and memory growth it does not control). The paper has no
 * counterpart; this is a deployment convenience.
 *
 * Inputs, outputs and results are exactly those of qmla_mla_decode. The
 * scratch the decode needs lives in one file-scope device array of
 * qmla_static_scratch_bytes() bytes that every GPU loading this library holds
 * until the process exits. Nothing is allocated or freed by this call.
 * - The first call on a device looks up that array's device address
 *   (cudaGetSymbolAddress) with the device current; make that first call
 *   before capturing any stream.
 * - Accepts batch x heads whose workspace fits the array:
 *   qmla_decode_workspace_bytes(batch, heads) <= qmla_static_scratch_bytes().
 *   Larger ones return QMLA_ERR_WORKSPACE_TOO_SMALL before any launch. The
 *   workspace grows with the SM count; on a 152-SM GB300 32 sequences at 128
 *   heads fit, 64 sequences at 128 heads do not.
 * - Every call shares the array, which keeps the last call's contents;
 *   nothing in it needs to start at zero (each call rewrites or clears
 *   everything it reads). Calls whose work overlaps on the GPU (different
 *   streams, or different host threads on one device) race on it: serialise
 *   them.
 * - The looked-up address is kept for the life of the process: after a
 *   cudaDeviceReset of a device this entry point has run on, the address is
 *   stale, so do not call it on that device again in the same process.
 * - It is qmla_mla_decode_ex with the array as the workspace: argument checks
 *   and errors are those of qmla_mla_decode.
 */
int qmla_mla_decode_static(const void* pool_dev, int c_bits, int num_blocks, const uint16_t* q_latent_dev,
                           const uint16_t* q_pe_dev, int batch, int heads, const int32_t* block_table_dev,
                           int max_blocks, const int32_t* seq_lens_dev, float softmax_scale, float* out_dev,
                           float* lse_dev, uint32_t* dev_err_dev, qmla_stream_t stream);

/*
 * Test hook (no counterpart in the paper): the fp16 tile the decode kernel builds
 * from the cache for tile j (positions 128 j .. 128 j + 127) of sequence b, made
 * by the decode's own row loaders into its swizzled shared-memory chunks and
 * written out row-major in channel order.
 *   cache_kind   4 or 2: this library's block with that content width;
 *                QMLA_CACHE_C4R4: the paper's page; QMLA_CACHE_BF16: the BF16 cache
 *   prot_dev     NULL, or the sink4/local128 protection buffer (packed kinds):
 *                rows in P_L come from it as in qmla_mla_decode_protected
 *   tile_dev     [128][576] fp16 (uint16 bits), 16-byte aligned; row r holds the
 *                512 latent then 64 RoPE-key values of position 128 j + r, zero for
 *                rows at or past seq_lens_dev[b]
 * Table, lengths and errors as qmla_mla_decode; 0 <= b < batch, 0 <= j. One CTA
 * of 128 threads; not a fast path.
 */
#define QMLA_CACHE_C4R4 5
#define QMLA_CACHE_BF16 16
int qmla_debug_tile(const void* pool_dev, int cache_kind, int num_blocks, const int32_t* block_table_dev,
                    int max_blocks, const int32_t* seq_lens_dev, int batch, int b, int j, const void* prot_dev,
                    uint16_t* tile_dev, uint32_t* dev_err_dev, qmla_stream_t stream);

/* Test hook (no counterpart in the paper): one warp waits, through the decode
 * kernel's bounded wait, for a barrier phase that nothing completes. After
 * limit_us microseconds (1 .. 1000000) the wait gives up and ORs
 * QMLA_DEVERR_TIMEOUT | QMLA_DEVERR_SITE_SOFTMAX into *dev_err_dev, and the
 * kernel returns; the context stays usable. The decode's own waits give up after
 * 2 s the same way (one site bit per wait, bits 8 and up). */
#define QMLA_DEVERR_SITE_SOFTMAX (0x100u << 5)
int qmla_debug_wait_timeout(uint32_t limit_us, uint32_t* dev_err_dev, qmla_stream_t stream);

/* Copies the device error word to *host_out after synchronising `stream`. */
int qmla_read_dev_err(const uint32_t* dev_err_dev, uint32_t* host_out, qmla_stream_t stream);

/* The cudaError_t of the last failed CUDA call in this thread (0 if none). */
int qmla_last_cuda_error(void);

/* Static text for a status code. */
const char* qmla_status_string(int status);

/* Number of SMs of the current device (the decode grid size), or -1. */
int qmla_num_sms(void);

#ifdef __cplusplus
}
#endif

#endif /* QMLA_H_ */
