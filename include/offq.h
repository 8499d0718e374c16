/*
 * offq.h -- C ABI of the OffQ W4A4 linear hot path on GB300 (sm_103a).
 *
 * OffQ (arxiv 2606.07116) makes 4-bit weight/activation/KV quantization work
 * by rotating each activation row with a Hadamard matrix whose first row is all
 * ones, so the concentrated outlier channel turns into a constant offset shared
 * by a whole block of channels (Sec. 3.2, Eq. 4-5), and quantizing what is left
 * on a uniform 4-bit grid (Sec. 3, Eq. 1). This library runs the online part of
 * that method:
 *
 *   offq_quantize_act   token rows -> block Hadamard -> offsets -> 4-bit codes
 *   offq_w4a4_linear    4-bit x 4-bit GEMM + dequant + offset epilogue
 *   offq_kv4_quantize   per-(token, head) version of the quantizer (KV cache)
 *   offq_prepare_weight offline: rotated, per-channel 4-bit weights + tables
 *
 * and the paper's evaluated per-group asymmetric variant of the first two:
 *
 *   offq_quantize_act_group  rotation -> groups of 128 with zero-points -> codes
 *   offq_weight_group_sums   offline: weight row sums per activation group
 *   offq_w4a4_linear_group   GEMM with per-group scales and zero-points
 *
 * and, for keys with bias-induced outliers, the dense per-head rotation
 * M = U3 P3 H3 in place of H3:
 *
 *   offq_kv4_quantize_rotated  key cache: rotate by M, then offset / scale / codes
 *   offq_rotate_heads          queries: rotate by the same M
 *   offq_prepare_key_rotation  offline: M in three bf16 parts, tensor-core order
 *   offq_kv4_quantize_prepared, offq_rotate_heads_prepared
 *                              the two above from the prepared parts (bf16)
 *   offq_prepare_key_reflection  offline (host): M = U3 P3 H3 from U3's
 *                              direction and P3, in structured form
 *   offq_kv4_quantize_reflected, offq_rotate_heads_reflected
 *                              key cache / queries with the structured M (bf16)
 *
 * and the offline transform builder (top-1 tokens, top-1 PCA direction,
 * reflection, sorted grouping, fusion into the weights).
 *
 * Conventions shared by every call
 *   - Pointers named as device buffers are device pointers allocated and owned
 *     by the caller. The library never allocates, frees, or synchronizes the
 *     stream (offq_get_device_status is the one call that synchronizes).
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *   - Arguments are checked on the host before anything is launched. A bad
 *     shape or flag returns OFFQ_ERR_INVALID_ARG or OFFQ_ERR_UNSUPPORTED; a
 *     pointer or leading dimension that breaks the alignment rule of the call
 *     returns OFFQ_ERR_MISALIGNED; a failed launch returns OFFQ_ERR_CUDA.
 *     Nothing is written when a call returns an error.
 *   - Errors that only the device can see (a bounded wait that ran out inside
 *     a kernel) are recorded in a device status word; offq_get_device_status
 *     reads and clears it.
 *   - NaN or Inf inputs: results are unspecified (no checks on the hot path).
 *   - Calls are thread-safe. The only state is set on first use per device
 *     (kernel attributes, the SM count, the status word's address) and the
 *     device status word itself.
 *
 * Block size g. The online rotation is block-diagonal with g x g Sylvester
 * Hadamard blocks (group-wise offsetting, Sec. 3.2); each block of g channels
 * of a row gets one offset. g is a power of two in [32, 8192] and divides K.
 * The scale is one per token row across all blocks.
 *
 * Code formats (the paper fixes the 4-bit uniform grid, not a bit layout):
 *   Activation codes: Eq. 1's unsigned form with zero-point 8. A residual
 *     quantized to q in [-7, 7] is stored as the nibble u = q + 8 (1..15). Two
 *     nibbles per byte, the even channel in the low nibble, so row t is a
 *     string of K/2 bytes.
 *   Weight codes: per-output-channel signed q in [-7, 7], sign-magnitude,
 *     interleaved per group of 8 channels c0..c7 held in 4 bytes B0..B3:
 *       Bj bits 0-2 = |q(c_2j)|, bit 7 = sign(q(c_2j)),
 *       Bj bits 4-6 = |q(c_2j+1)|, bit 3 = sign(q(c_(2j-1) mod 8)).
 *     (This lets the GEMM widen 8 codes to fp8 tensor-core operands with one
 *     rotate and two masks.) Row n is a string of K/2 bytes.
 *   Tiled operand layout (activation and weight codes): rows are grouped by
 *     32 and split into 16-byte chunks of 32 codes; byte j of row r is stored
 *     at ((r / 32) * (K / 32) + j / 16) * 512 + (r % 32) * 16 + j % 16. A
 *     buffer of R rows therefore holds ceil(R/32)*32 rows (offq_act_codes_bytes,
 *     offq_weight_codes_bytes). The GEMM's warps then load 32 rows x 16 bytes
 *     as 512 contiguous bytes. KV-cache codes stay row-major.
 */
#ifndef OFFQ_H
#define OFFQ_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define OFFQ_ABI_VERSION 1

/* Bytes of one head's prepared rotation (offq_prepare_key_rotation). */
#define OFFQ_KEY_ROTATION_BYTES 98304
/* Bytes of one head's prepared structured rotation (offq_prepare_key_reflection). */
#define OFFQ_KEY_REFLECTION_BYTES 37376

typedef enum {
  OFFQ_OK = 0,
  OFFQ_ERR_INVALID_ARG = -1,  /* shape, flag or NULL pointer not allowed   */
  OFFQ_ERR_UNSUPPORTED = -2,  /* valid request the library does not handle */
  OFFQ_ERR_MISALIGNED = -3,   /* pointer / leading dimension alignment     */
  OFFQ_ERR_CUDA = -4,         /* a CUDA runtime call failed                */
  OFFQ_ERR_TIMEOUT = -5       /* a device-side bounded wait ran out        */
} offq_status;

/* Element types of floating-point buffers. */
enum { OFFQ_F32 = 0, OFFQ_BF16 = 1, OFFQ_F16 = 2 };

/* Flags of the quantizers. */
enum {
  OFFQ_ROTATE = 1, /* apply the online block Hadamard H/sqrt(g) (Eq. 4)       */
  OFFQ_OFFSET = 2  /* subtract each block's mean as its offset (Eq. 5)        */
};

/*
 * offq_quantize_act -- online activation quantizer (paper Sec. 3.2 Eq. 4-5,
 * Sec. 3 Eq. 1; the online rotation H4 of Sec. 3.3 Step 2 (4)).
 *
 * For each token row x (K channels) and each block b of g channels:
 *   y = x_b H_g / sqrt(g)          if OFFQ_ROTATE (else y = x_b)
 *   o[b] = mean(y)                 if OFFQ_OFFSET (else 0); with the rotation
 *                                  this equals x_b[0] / sqrt(g)
 *   r = y - o[b]
 * then over the whole row: s = max|r| / 7 (0 for an all-zero residual),
 * q = clamp(round_half_even(r / s), -7, 7), stored as u = q + 8.
 *
 *   x       device, [T][ldx] elements of x_dtype (OFFQ_F32/BF16/F16), row-major;
 *           16-byte aligned, ldx * sizeof(elem) a multiple of 16, ldx >= K.
 *   T       token rows, >= 0 (T = 0 launches nothing).
 *   K       channels, a multiple of g and of 32, K <= 32768.
 *   g       block size, power of two in [32, 8192].
 *   flags   OR of OFFQ_ROTATE, OFFQ_OFFSET.
 *   codes   device, offq_act_codes_bytes(T, K) bytes, activation code format in
 *           the tiled operand layout, 16-byte aligned (rows beyond T in the
 *           last 32-row group are left as they are).
 *   scale   device, [T] float32.
 *   offset  device, [T][K/g] float32; required with OFFQ_OFFSET; when given
 *           without OFFQ_OFFSET it is filled with zeros; may be NULL otherwise.
 *
 * Arithmetic: fp32 throughout; the rounding decisions are taken in fp32. The
 * rotation is a radix-2 tree of fp32 additions, except for bf16 rows with
 * g = 1024 and OFFQ_ROTATE when ceil(T / floor(65536 / K)) (tiles of up to
 * 64 blocks of whole tokens) is at least the SM count: those take the tensor cores
 * for a 128-point factor of the Hadamard (exact bf16 x +-1 products summed in
 * the MMA's fp32 accumulator), with the remaining three factors in fp32. The
 * two forms agree within their fp32 error bounds, not bit for bit, so a code
 * near a rounding tie may differ between them.
 */
int offq_quantize_act(const void* x, int x_dtype, int64_t T, int64_t K, int64_t ldx,
                      int32_t g, int32_t flags,
                      uint8_t* codes, float* scale, float* offset, void* stream);

/*
 * offq_w4a4_linear -- W4A4 GEMM with fused dequant and offset epilogue
 * ("all matrix multiplications in uniform 4-bit execution", Sec. 1; the
 * offset leaves a block as a constant, Eq. 5, so it meets the weight block
 * row sums).
 *
 *   y[t][n] = s_a[t] * s_w[n] * sum_k q_a[t][k] q_w[n][k]
 *           + s_w[n] * sum_b o[t][b] * R[b][n]
 *
 * accumulated exactly in integers (the tensor cores see both codes as exact
 * fp8 values; at T <= 4 the CUDA cores use dp4a; every partial sum is an
 * integer below 2^24), dequantized in fp32
 * and rounded once to the output type.
 *
 *   a_codes   device, tiled activation codes of T rows (offq_quantize_act), 16-B aligned.
 *             The buffer holds ceil(T/32)*32 rows. Rows T .. ceil(T/32)*32-1 may
 *             hold anything: they are read as operands (every nibble is a
 *             finite fp8 value), but the output rows they feed are never
 *             written, nor do they reach acc_debug.
 *   a_scale   device, [T] float32.
 *   a_offset  device, [T][K/g] float32, or NULL for all-zero offsets.
 *   T, N, K   tokens, output channels, input channels; T >= 0, N >= 1,
 *             K a multiple of g and of 32, K <= 65536.
 *   g         block size used when the codes were made (power of two, 32..8192).
 *   w_codes   device, tiled weight codes of N rows (offq_prepare_weight), 16-B aligned.
 *   w_scale   device, [N] float32.
 *   w_offsum  device, [K/g][N] float32: R[b][n] = sum_{k in block b} q_w[n][k],
 *             the integer block row sums of the weight codes (exact in fp32).
 *   out       device, [T][ldo] of out_dtype (OFFQ_F32/BF16/F16), ldo >= N,
 *             16-byte aligned with ldo * sizeof(out) a multiple of 16.
 *   acc_debug device, [T][N] int32 or NULL. When given, also receives the
 *             integer the tensor cores accumulate, sum_k (q_a + 8) * q_w
 *             (equal to the true dot product plus 8 * sum_k q_w[n][k]).
 * Forms: T > 64 the pair-tile tensor-core kernel; 5 <= T <= 64 the decode
 * kernel (weights on the MMA's M side); T <= 4 (with T' * K <= 96 KB, T'
 * the token count rounded up to 1, 2 or 4) the CUDA-core form. All give the
 * same accumulator and apply the same epilogue.
 * Ordering: the T <= 4 form starts reading w_codes before the kernel ahead of
 * it in the stream has finished (programmatic dependent launch), so the
 * weight codes must not be written by a kernel that releases its dependents
 * early (ordinary kernels never do; no kernel of this library that writes
 * weight codes does).
 */
int offq_w4a4_linear(const uint8_t* a_codes, const float* a_scale, const float* a_offset,
                     int64_t T, int64_t N, int64_t K, int32_t g,
                     const uint8_t* w_codes, const float* w_scale, const float* w_offsum,
                     void* out, int out_dtype, int64_t ldo, int32_t* acc_debug, void* stream);

/*
 * offq_kv4_quantize -- KV-cache quantizer: offq_quantize_act applied to every
 * (token, head) vector with g = head_dim, i.e. the per-head online Hadamard H3
 * of the keys (Sec. 3.3 Step 2 (3)) with one offset and one scale per head
 * (the KV quantization group equals the head dimension, Sec. 4.2).
 *
 *   kv        device, element (t, h, d) at kv[t*ld_token + h*head_dim + d];
 *             16-byte aligned, ld_token * sizeof(elem) a multiple of 16,
 *             ld_token >= H * head_dim.
 *   T, H      tokens (>= 0) and heads (>= 1).
 *   head_dim  power of two in [32, 8192].
 *   flags     OR of OFFQ_ROTATE, OFFQ_OFFSET (V vectors, rotated offline by
 *             R2, may pass OFFQ_OFFSET alone).
 *   codes     device, [T][H][head_dim/2] activation code format, 16-B aligned.
 *   scale     device, [T][H] float32.
 *   offset    device, [T][H] float32 (same rules as offq_quantize_act).
 */
int offq_kv4_quantize(const void* kv, int dtype, int64_t T, int32_t H, int32_t head_dim,
                      int64_t ld_token, int32_t flags,
                      uint8_t* codes, float* scale, float* offset, void* stream);

/*
 * offq_prepare_weight -- offline weight preparation (not on the timed path).
 * The inverse of the online rotation is fused into the weight (Sec. 3.3
 * Step 2 (4): W x = (W H)(H x) for the symmetric orthonormal block Hadamard),
 * then each output channel is quantized symmetrically (per-channel symmetric
 * weights, Sec. 4 "Implementation and Settings"; round-to-nearest stands in
 * for GPTQ, which needs calibration data):
 *   W_eff = W blockdiag(H_g)/sqrt(g) if rotate else W
 *   s_w[n] = max|W_eff[n]| / 7,  q_w = clamp(rne(W_eff / s_w), -7, 7)
 *   R[b][n] = sum_{k in block b} q_w[n][k]   (integers, stored as float32)
 *
 *   w         device, [N][K] of dtype, row-major, 16-byte aligned.
 *   N, K, g   as in offq_w4a4_linear.
 *   rotate    nonzero to fuse the block Hadamard.
 *   w_codes   device, offq_weight_codes_bytes(N, K) bytes, weight code format in
 *             the tiled operand layout (padding rows set to zero), 16-B aligned.
 *   w_scale   device, [N] float32.
 *   w_offsum  device, [K/g][N] float32.
 */
int offq_prepare_weight(const void* w, int dtype, int64_t N, int64_t K, int32_t g, int32_t rotate,
                        uint8_t* w_codes, float* w_scale, float* w_offsum, void* stream);

/*
 * Per-group asymmetric path -- the paper's evaluated activation setting
 * (Sec. 4 "Implementation and Settings": activations quantized per group of
 * 128 channels, asymmetrically; Sec. 3 Eq. 1 with its zero-point z). After
 * the Hadamard rotation the outlier is a constant offset over a block
 * (Eq. 5), which each group's zero-point absorbs (Sec. 3.2 footnote: the grid
 * need not hold 0), so this path stores no explicit offset.
 *
 * offq_quantize_act_group -- for each token row x (K channels):
 *   y = x_b H_g / sqrt(g) per block b of g channels   if OFFQ_ROTATE (else y = x)
 * then for each group j of `group` channels of y:
 *   s[j] = (max - min) / 15,  z[j] = -round_half_even(min / s[j])  (any integer),
 *   u = clamp(round_half_even(y / s[j]) + z[j], 0, 15);
 * a constant group gets s = z = u = 0. y ~ s (u - z). The ratios y / s and
 * min / s are taken as 15 y / (max - min) and 15 min / (max - min) in fp32 (s
 * is not rounded first), so exact half-integer ratios round half to even.
 *
 *   x       device, [T][ldx] elements of x_dtype, row-major; 16-byte aligned,
 *           ldx * sizeof(elem) a multiple of 16, ldx >= K.
 *   T       token rows, >= 0 (T = 0 launches nothing).
 *   K       channels, a multiple of `group` (and of g with the rotation),
 *           K <= 65536.
 *   g       rotation block, power of two in [32, 8192]; ignored without
 *           OFFQ_ROTATE.
 *   group   channels per quantization group; this library supports 128
 *           (OFFQ_ERR_UNSUPPORTED for other positive values).
 *   flags   0 or OFFQ_ROTATE.
 *   codes   device, offq_act_codes_bytes(T, K) bytes: u as the nibble, two per
 *           byte (even channel low), in the tiled operand layout, 16-B aligned
 *           (rows beyond T in the last 32-row group are left as they are).
 *   scale   device, [T][K/group] float32.
 *   zero    device, [T][K/group] float32 (integer-valued).
 */
int offq_quantize_act_group(const void* x, int x_dtype, int64_t T, int64_t K, int64_t ldx,
                            int32_t g, int32_t group, int32_t flags,
                            uint8_t* codes, float* scale, float* zero, void* stream);

/*
 * offq_weight_group_sums -- offline: R[j][n] = sum_{k in group j} q_w[n][k],
 * the integer row sums of prepared weight codes (offq_prepare_weight) over
 * each activation group, stored as float32. They carry the zero-point term
 * of the per-group GEMM.
 *
 *   w_codes     device, tiled weight codes of N rows (offq_prepare_weight), 16-B aligned.
 *   N, K        output and input channels (K a multiple of 32 and of group).
 *   group       power of two >= 32 dividing K.
 *   w_groupsum  device, [K/group][N] float32.
 */
int offq_weight_group_sums(const uint8_t* w_codes, int64_t N, int64_t K, int32_t group,
                           float* w_groupsum, void* stream);

/*
 * offq_w4a4_linear_group -- W4A4 GEMM of the per-group path:
 *   y[t][n] = s_w[n] * sum_j s[t][j] * (P_j[t][n] - z[t][j] * R[j][n]),
 *   P_j[t][n] = sum_{k in group j} u[t][k] * q_w[n][k]   (exact integers),
 * i.e. y = X_hat W_hat^T with X_hat = s (u - z) and W_hat = s_w q_w. Each
 * group's product is exact on the tensor cores; the per-group scaling and the
 * zero-point term are fp32 multiply-adds in group order, rounded once to the
 * output type.
 *
 *   a_codes, a_scale, a_zero  from offq_quantize_act_group (T rows, K channels).
 *   T, N, K     T >= 0, N >= 1, K a multiple of group, K <= 65536.
 *   group       128 in this library (OFFQ_ERR_UNSUPPORTED otherwise).
 *   w_codes, w_scale          from offq_prepare_weight (any rotation block).
 *   w_groupsum  from offq_weight_group_sums with the same group.
 *   out         device, [T][ldo] of out_dtype, ldo >= N, 16-byte aligned with
 *               ldo * sizeof(out) a multiple of 16.
 */
int offq_w4a4_linear_group(const uint8_t* a_codes, const float* a_scale, const float* a_zero,
                           int64_t T, int64_t N, int64_t K, int32_t group,
                           const uint8_t* w_codes, const float* w_scale, const float* w_groupsum,
                           void* out, int out_dtype, int64_t ldo, void* stream);

/*
 * Key cache under a dense per-head rotation -- paper Sec. 3.3 Step 2 (3):
 * with bias-induced outliers in the keys, the per-head online Hadamard H3 is
 * replaced by M = U3 P3 H3 (a per-head top-1 PCA rotation, a permutation and
 * H3), applied to the RoPE-encoded outputs of W_Q and W_K, so Q K^T is
 * unchanged for orthonormal M.
 *
 * offq_kv4_quantize_rotated -- for every (token, head) vector x of head_dim:
 *   y = x M[h]  with fp32 accumulation (bf16 keys: on the tensor cores with M
 *               split into three bf16 parts, M = M1 + M2 + M3 to 24 bits; fp32
 *               and fp16 keys: fp32 FMAs in input-channel order),
 *   o = mean(y) with OFFQ_OFFSET (else 0), r = y - o, s = max|r| / 7,
 *   q = clamp(round_half_even(r / s), -7, 7), stored as u = q + 8;
 * the outputs of offq_kv4_quantize with M[h] in place of H3 / sqrt(head_dim).
 *
 *   kv        device, element (t, h, d) at kv[t*ld_token + h*head_dim + d];
 *             16-byte aligned, ld_token * sizeof(elem) a multiple of 16,
 *             ld_token >= H * head_dim.
 *   T, H      tokens (>= 0) and heads (1..65535).
 *   head_dim  128 in this library (OFFQ_ERR_UNSUPPORTED otherwise).
 *   rot       device, [H][head_dim][head_dim] float32, row-major (y_j =
 *             sum_i x_i rot[h][i][j]), 16-byte aligned. It is orthonormal
 *             in the method; the call does not check that.
 *   flags     0 or OFFQ_OFFSET.
 *   codes     device, [T][H][head_dim/2] activation code format, 16-B aligned.
 *   scale     device, [T][H] float32.
 *   offset    device, [T][H] float32; required with OFFQ_OFFSET, else may be NULL.
 */
int offq_kv4_quantize_rotated(const void* kv, int dtype, int64_t T, int32_t H, int32_t head_dim,
                              int64_t ld_token, const float* rot, int32_t flags,
                              uint8_t* codes, float* scale, float* offset, void* stream);

/*
 * offq_rotate_heads -- the same y = x M[h] without quantization (the query
 * side of the rotation), rounded once to out_dtype.
 *
 *   x, T, H, head_dim, ld_token, rot   as in offq_kv4_quantize_rotated.
 *   out       device, element (t, h, d) at out[t*ld_out + h*head_dim + d] of
 *             out_dtype; 16-byte aligned, ld_out * sizeof(out) a multiple of
 *             16, ld_out >= H * head_dim.
 */
int offq_rotate_heads(const void* x, int dtype, int64_t T, int32_t H, int32_t head_dim, int64_t ld_token,
                      const float* rot, void* out, int out_dtype, int64_t ld_out, void* stream);

/*
 * offq_prepare_key_rotation -- offline, once per model: each M[h] split into
 * three bf16 parts, M = M1 + M2 + M3 (M1 = bf16(M), M2 = bf16(M - M1),
 * M3 = bf16(M - M1 - M2), differences exact in float32: the parts carry M's
 * 24-bit significand), written in the operand order of the tensor-core
 * kernel, which then copies a head's parts into shared memory as they are
 * instead of splitting M in every CTA.
 *
 *   rot       device, as in offq_kv4_quantize_rotated.
 *   H         heads (1..65535).   head_dim  128 in this library.
 *   prepared  device, H * OFFQ_KEY_ROTATION_BYTES bytes, 16-byte aligned,
 *             written. An opaque image: head h's bytes start at
 *             h * OFFQ_KEY_ROTATION_BYTES; part s (0..2) of it is 128 rows
 *             n of 128 bf16 M_s[k][n] (k-major), 16-byte chunks swizzled
 *             within 128-byte rows.
 */
int offq_prepare_key_rotation(const float* rot, int32_t H, int32_t head_dim, void* prepared, void* stream);

/*
 * offq_kv4_quantize_prepared / offq_rotate_heads_prepared --
 * offq_kv4_quantize_rotated and offq_rotate_heads for bf16 inputs, with M
 * given as offq_prepare_key_rotation's image. Same arithmetic and results
 * (the tensor-core path with M in three bf16 parts).
 *
 *   dtype     OFFQ_BF16 (OFFQ_ERR_UNSUPPORTED otherwise).
 *   prepared  device, offq_prepare_key_rotation's output for the same H.
 *   other arguments as in offq_kv4_quantize_rotated / offq_rotate_heads.
 */
int offq_kv4_quantize_prepared(const void* kv, int dtype, int64_t T, int32_t H, int32_t head_dim,
                               int64_t ld_token, const void* prepared, int32_t flags,
                               uint8_t* codes, float* scale, float* offset, void* stream);
int offq_rotate_heads_prepared(const void* x, int dtype, int64_t T, int32_t H, int32_t head_dim,
                               int64_t ld_token, const void* prepared, void* out, int out_dtype,
                               int64_t ld_out, void* stream);

/*
 * The structured form of M = U3 P3 H3 -- paper Sec. 3.3 Step 2 (3) with Step 1
 * (2)'s top-1 PCA rotation taken as the reflection U3 = I - 2 w w^T that maps
 * channel 0 to the head's top-1 direction v (w = (v/|v| - e_0) normalised;
 * U3 = I when v/|v| = e_0), P3 the channel permutation ((x P3)_c = x_perm[c])
 * and H3 = H / sqrt(128) the normalised Sylvester Hadamard. Then
 *   y = x M = u - 2 (x . w) w'',  u = x P3 H3,  w'' = (P3 H3)^T w,
 * and x P3 H3 has +-1 coefficients (exact in bf16): one tensor-core product
 * of N = 144 per tile gives u * sqrt(128) and x . w (w in three bf16 parts),
 * instead of the three-part product with a general M.
 *
 * offq_prepare_key_reflection -- HOST function, offline: the per-head image.
 *   v         host, [H][head_dim] float32, head h's top-1 direction (any
 *             nonzero length; OFFQ_ERR_INVALID_ARG for a zero or non-finite v).
 *   perm      host, [H][head_dim] int32, each row a permutation of
 *             0..head_dim-1 (OFFQ_ERR_INVALID_ARG otherwise). The method keeps
 *             perm[h][0] = 0 (the concentrated channel stays first); the call
 *             does not require it.
 *   H, head_dim  heads (1..65535), 128.
 *   prepared  host, H * OFFQ_KEY_REFLECTION_BYTES bytes, written: for each
 *             head, 144 rows n x 128 bf16 (k-major, 16-byte chunks swizzled
 *             within 128-byte rows, the 64-channel halves 18432 bytes apart):
 *             rows n < 128 are sqrt(128) (P3 H3)[k][n] = +-1, rows 128..130
 *             the bf16 parts of fp32(w), rows 131..143 zero; then w'' as 128
 *             float32 (computed in float64, rounded once). Copy it to the
 *             device as is.
 *
 * offq_kv4_quantize_reflected / offq_rotate_heads_reflected --
 * offq_kv4_quantize_rotated and offq_rotate_heads for bf16 inputs with M in
 * this form: y_j = fma(acc_j, fp32(1/sqrt(128)), fl(-2 d w''_j)), where acc =
 * sqrt(128) x P3 H3 and d = x . w are fp32 tensor-core sums of exact products.
 *   dtype     OFFQ_BF16 (OFFQ_ERR_UNSUPPORTED otherwise).
 *   prepared  device, 16-byte aligned, offq_prepare_key_reflection's image.
 *   other arguments as in offq_kv4_quantize_rotated / offq_rotate_heads.
 */
int offq_prepare_key_reflection(const float* v, const int32_t* perm, int32_t H, int32_t head_dim,
                                void* prepared);
int offq_kv4_quantize_reflected(const void* kv, int dtype, int64_t T, int32_t H, int32_t head_dim,
                                int64_t ld_token, const void* prepared, int32_t flags,
                                uint8_t* codes, float* scale, float* offset, void* stream);
int offq_rotate_heads_reflected(const void* x, int dtype, int64_t T, int32_t H, int32_t head_dim,
                                int64_t ld_token, const void* prepared, void* out, int out_dtype,
                                int64_t ld_out, void* stream);

/*
 * Offline transform builder -- paper Sec. 3.1 (top-1 PCA), Sec. 3.2 (sorted
 * grouping for group-wise offsetting), Sec. 3.3 Steps 1-2 (fusion). Run once
 * per model on calibration activations; not on the inference path.
 *
 * offq_top1_tokens -- for each sequence s of x (L tokens of D channels), the
 * token of largest L-infinity norm max_d |x| (Sec. 3.1 "top-1"; the first on
 * ties): index[s], and that token as float32 in rows[s][0 .. D).
 *   x         device, element (s, l, d) at x[s*ld_seq + l*ld_token + d] of dtype,
 *             aligned to its element size; ld_token >= D, ld_seq >= L*ld_token.
 *   S, L, D   sequences (>= 0), tokens (>= 1), channels (>= 1).
 *   index     device, [S] int32.   rows  device, [S][D] float32.
 */
int offq_top1_tokens(const void* x, int dtype, int64_t S, int64_t L, int64_t D, int64_t ld_token,
                     int64_t ld_seq, int32_t* index, float* rows, void* stream);

/*
 * offq_top1_direction -- the leading eigenvector of C = X^T X / N (Eq. 6) by
 * `iters` steps of power iteration from v0: v <- X^T (X v), normalised. The
 * result's largest-magnitude entry is positive; proj[n] = X[n] . v for the
 * returned v (the tokens' top-1 scores). v and proj carry the iteration.
 *   X     device, [N][D] float32 row-major.   v0  device, [D] float32 start vector.
 *   v     device, [D] float32 (output).        proj device, [N] float32 (output).
 */
int offq_top1_direction(const float* X, int64_t N, int64_t D, int32_t iters, const float* v0, float* v,
                        float* proj, void* stream);

/*
 * offq_reflect_rows -- out[r] = A[r] U1 with U1 = I - 2 w w^T / |w|^2,
 * w = v/|v| - e_1: the symmetric reflection with U1 e_1 = v/|v|, so x U1
 * carries x . v/|v| in channel 0 (the concentrated outlier channel).
 *   A, out  device, [R][D] float32 (may not overlap).  v  device, [D] float32.
 *   D <= 16384 in this library.
 */
int offq_reflect_rows(const float* A, int64_t R, int64_t D, const float* v, float* out, void* stream);

/* offq_column_absmax -- mag[d] = max_r |A[r][d]| for A device [R][D] float32,
 * mag device [D] float32. */
int offq_column_absmax(const float* A, int64_t R, int64_t D, float* mag, void* stream);

/*
 * offq_sorted_grouping -- the sorted-grouping permutation of D channels into G
 * groups of D/G (Sec. 3.2; Sec. 4 "Sorted versus Zigzag Grouping"): the G
 * channels of largest |mag| lead the groups (largest first), the others fill
 * the groups in ascending order of |mag|; equal magnitudes keep channel order.
 * New channel c takes old channel perm[c]. HOST pointers (mag [D] float32,
 * perm [D] int32); synchronous, no stream.
 */
int offq_sorted_grouping(const float* mag, int64_t D, int32_t G, int32_t* perm);

/*
 * offq_fuse_rotation -- out = W U1 P1 blockdiag(H_g)/sqrt(g): the weight that
 * meets activations rotated as x U1 P1 H1 (Sec. 3.3 Step 2 (1)), so that
 * W x = out (x U1 P1 H1)^T. U1 as in offq_reflect_rows; P1 from perm (new
 * column c = old column perm[c]); H_g Sylvester.
 *   W, out  device, [N][D] float32 (may not overlap).  v device [D] float32.
 *   perm    device, [D] int32 permutation.   g  power of two dividing D.
 *   D <= 16384 in this library.
 */
int offq_fuse_rotation(const float* W, int64_t N, int64_t D, const float* v, const int32_t* perm, int32_t g,
                       float* out, void* stream);

/*
 * MXFP4 residuals with the offset as zero-point (paper Sec. 3.4 "Generality
 * on Data Formats": micro-scaling formats extended with a zero-point per block
 * absorb the outlier offset; the paper leaves the extension to future work).
 *
 * offq_quantize_act_mx -- for each token row x (K channels):
 *   y = x_b H_g / sqrt(g) per block b of g channels   if OFFQ_ROTATE (else y = x)
 *   o[b] = mean(y_b) if OFFQ_OFFSET (else 0),  r = y - o
 * then per 32 channels j of r (MXFP4's shared exponent and E2M1 elements):
 *   X_j = floor(log2(max |r_j|)) - 2, raised to at least Xmax - 6 (Xmax the
 *         row's largest; an all-zero block takes Xmax - 6),
 *   e = E2M1 code of r / 2^X_j: nearest of the magnitudes 0, 0.5, 1, 1.5, 2, 3,
 *       4, 6 (codes 0..7), ties to the even code, saturating at 6; sign in bit 3.
 * r ~ value(e) * 2^X_j, so x ~ value(e) * 2^X_j + o.
 *
 *   x, T, K, ldx  as offq_quantize_act; K a multiple of g and of 128, K <= 32768.
 *   g         block of the rotation and of the offsets, power of two in [32, 8192].
 *   codes     device, offq_act_codes_bytes(T, K) bytes: e as nibbles, two per byte
 *             (even channel low), in the tiled operand layout, 16-B aligned.
 *   shifts    device, offq_mx_shift_bytes(T, K) bytes, 4-B aligned: sh_j = X_j -
 *             (Xmax - 6) in 0..6, byte ((r/32 * K/128 + j/4) * 32 + r%32) * 4 + j%4
 *             for row r and block j (the four shifts of a row's 128-code k-tile
 *             are one 32-bit word).
 *   row_scale device, [T] float32: 2^(Xmax - 6).
 *   offset    device, [T][K/g] float32; required with OFFQ_OFFSET.
 * Rows of the last 32-row group beyond T are left as they are.
 */
int offq_quantize_act_mx(const void* x, int x_dtype, int64_t T, int64_t K, int64_t ldx, int32_t g, int32_t flags,
                         uint8_t* codes, uint8_t* shifts, float* row_scale, float* offset, void* stream);

/*
 * offq_prepare_weight_mx -- offline: MXFP4 weights W [N][K] (row-major, dtype
 * OFFQ_F32/BF16/F16), per output row as offq_quantize_act_mx without offsets,
 * after the rotation fused into W when `rotate` (W_eff = W blockdiag(H_g)/sqrt(g)).
 *   w_codes, w_shifts, w_scale  as codes, shifts, row_scale above (N rows); the
 *             padding rows of the last 32-row group are zero codes and shifts.
 *   w_offsum  device, [K/g][N] float32: R[b][n] = sum over block b of
 *             value(e) * 2^sh (the operand values; exact, multiples of 1/2).
 */
int offq_prepare_weight_mx(const void* w, int dtype, int64_t N, int64_t K, int32_t g, int32_t rotate,
                           uint8_t* w_codes, uint8_t* w_shifts, float* w_scale, float* w_offsum, void* stream);

/*
 * offq_mx_linear -- the W4A4 linear of MXFP4 operands:
 *   y[t][n] = s_w[n] * ( s_a[t] * sum_k A[t][k] W[n][k] + sum_b o[t][b] R[b][n] ),
 * A = value(e_a) * 2^sh_a and W = value(e_w) * 2^sh_w, each an exact E4M3 value,
 * multiplied on the tensor cores (kind::f8f6f4) with fp32 accumulation,
 * s_a / s_w the row scales. Arguments as offq_w4a4_linear (no acc_debug), plus
 * the shift buffers; K a multiple of 128 and of g.
 */
int offq_mx_linear(const uint8_t* a_codes, const uint8_t* a_shifts, const float* a_scale, const float* a_offset,
                   int64_t T, int64_t N, int64_t K, int32_t g, const uint8_t* w_codes, const uint8_t* w_shifts,
                   const float* w_scale, const float* w_offsum, void* out, int out_dtype, int64_t ldo, void* stream);

/* Bytes of a tiled MXFP4 shift buffer for R rows of K channels (-1 unless K is
 * a positive multiple of 128 and R >= 0): ceil(R/32) * 32 * K / 32. */
int64_t offq_mx_shift_bytes(int64_t R, int64_t K);

/* Bytes of a tiled activation-code buffer for T rows of K codes (-1 if K is
 * not a positive multiple of 32 or T < 0): ceil(T/32) * 32 * K / 2. */
int64_t offq_act_codes_bytes(int64_t T, int64_t K);

/* Bytes of a tiled weight-code buffer for N rows of K codes (-1 on bad sizes). */
int64_t offq_weight_codes_bytes(int64_t N, int64_t K);

/*
 * offq_get_device_status -- synchronizes `stream`, returns the device status
 * word of the current device (OFFQ_OK, or OFFQ_ERR_TIMEOUT when a kernel's
 * bounded wait ran out since the last call) and clears it. Returns
 * OFFQ_ERR_CUDA if the synchronization itself fails.
 */
int offq_get_device_status(void* stream);

/*
 * offq_set_wait_cycles -- test hook for the failure path (no counterpart in
 * the paper). Sets, for the calls that follow in this process, the budget in
 * SM clock cycles of the bounded waits with which the persistent row
 * quantizers (offq_quantize_act and offq_kv4_quantize on inputs with more row
 * groups than SMs, and the shared-memory ring kernel of rotation-free
 * single-block rows) wait for the rows they stage by bulk copies, and with
 * which the tensor-core form of offq_quantize_act (bf16, g = 1024) waits for
 * each tile's MMAs. A budget shorter than the default makes those waits
 * behave as waits for a flag that nothing sets: they do not look at their
 * barrier and give up after about that many cycles. The kernel then lets
 * every copy and MMA already in flight complete (waiting for it with the full
 * budget), releases its tensor memory, returns without writing the rest of
 * its outputs, and records OFFQ_ERR_TIMEOUT for offq_get_device_status.
 * 0 restores the default (about 2 s), and with it the normal waits. Returns
 * OFFQ_ERR_INVALID_ARG for a negative value. The setting is process-wide and
 * is read when a call launches; meant for tests only.
 */
int offq_set_wait_cycles(int64_t cycles);

/* Human-readable name of a status code (static string, never NULL). */
const char* offq_status_string(int status);

/* OFFQ_ABI_VERSION of the loaded library. */
int offq_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* OFFQ_H */
