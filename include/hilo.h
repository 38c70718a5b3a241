/*
 * hilo.h -- C ABI of libhilo, the GB300 (sm_103a) hot path of HiLo-Token
 * (input-adaptive high/low-frequency token compression around a diffusion
 * transformer block; paper Sec. 2.3 "HiLo-Token Selection").
 *
 * The path, per batch of B images of H x W latent tokens with d channels and
 * T text tokens each:
 *
 *   hilo_score          per-token high-frequency energy
 *   hilo_split          keep / pool decision, packed offsets
 *   hilo_pack           packed variable-length image sequence
 *   hilo_block_forward  MMDiT block (joint attention + MLP) on the packed rows
 *   hilo_unpack         back to the full token grid
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - All data pointers are DEVICE pointers owned by the caller; the library
 *   allocates no device memory in any call. Scratch space is the
 *   caller-provided workspace, sized by the *_workspace_bytes queries.
 * - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *   Every call is asynchronous on that stream; no call synchronises with the
 *   host, so a sequence of calls can be captured in a CUDA graph.
 * - Argument and shape errors are detected on the host before any launch and
 *   returned synchronously (HILO_ERR_ARG / HILO_ERR_SHAPE); a launch failure
 *   returns HILO_ERR_CUDA. Device-side failures (a bounded wait that ran out)
 *   are latched in a device word that hilo_sync_status() reads and clears.
 *   hilo_last_error() gives a human-readable detail of the last error of the
 *   calling thread.
 * - bf16 tensors are passed as void* (IEEE bfloat16, 2 bytes per element).
 * - Token index i of image b is p*W + q for grid position (p, q) (raster
 *   order); latents are [B, H, W, d] row-major with d contiguous.
 * - Packed rows ("row space"): the block works on R = B*T + cap rows of d
 *   channels. Rows [0, B*T) are the text tokens (image b owns rows
 *   b*T .. b*T+T-1); rows [B*T, B*T + cu_img[B]) are the packed image rows
 *   (image b owns B*T + cu_img[b] .. B*T + cu_img[b+1] - 1). cap >= cu_img[B]
 *   is the capacity the caller allocated (hilo_row_capacity always suffices:
 *   B*H*W without the low-frequency set), so no host read-back of the
 *   data-dependent row counts is ever needed.
 */
#ifndef HILO_H
#define HILO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes. */
enum {
  HILO_OK = 0,
  HILO_ERR_ARG = -1,         /* null pointer or bad scalar argument */
  HILO_ERR_SHAPE = -2,       /* shape outside the supported set (see hilo_shape) */
  HILO_ERR_CUDA = -3,        /* a CUDA runtime/driver call failed */
  HILO_ERR_WORKSPACE = -4,   /* workspace missing or smaller than required */
  HILO_ERR_TIMEOUT = -5,     /* a device-side bounded wait ran out (see hilo_sync_status) */
  HILO_ERR_UNSUPPORTED = -6, /* no sm_103a device, or a feature not built */
  HILO_ERR_CHECK = -7        /* a device-side index check failed (checks build only) */
};

/* Per-token labels written by hilo_split (HILO_LF: a non-kept token of the
 * separate low-frequency mode, shape.lf > 0). */
enum { HILO_KEEP = 0, HILO_POOL2 = 1, HILO_POOL4 = 2, HILO_LF = 3 };

/* Input dtypes of hilo_block_forward (HILO_F16: hilo_quantize_rows_e4m3). */
enum { HILO_BF16 = 0, HILO_F32 = 1, HILO_F16 = 2 };

/*
 * Problem shape.
 *   B       images in the batch (>= 1)
 *   H, W    latent token grid (even; multiples of 4 when levels == 2)
 *   d       channels (multiple of 128, <= 4096)
 *   T       text tokens per image (>= 0)
 *   heads   attention heads; head_dim = d / heads must be 64 or 128
 *   mlp     1: attention + 4x GELU MLP (a full MMDiT block); 0: attention only
 *   levels  1: every non-kept token is pooled 2x2; 2: 2x2 and 4x4 pooling
 *   lf      0: the in-grid pooling above; 2, 4 or 8: the separate
 *           low-frequency token set (paper Sec. 2.3: the kept tokens are
 *           concatenated with every token of a downsampled image; here the
 *           grid average-pooled lf-fold per side, all members included).
 *           Needs levels == 1 and H, W multiples of lf.
 * Also H*W <= 32768, and B * (H*W (+ H*W/lf^2) + T) < 2^31 (row indices are
 * int32). Any other combination returns HILO_ERR_SHAPE.
 */
typedef struct {
  int32_t B, H, W, d, T, heads, mlp, levels, lf;
} hilo_shape;

/*
 * The most packed image rows a split of this shape can produce over the
 * batch: B*N, or B*(N + N/lf^2) with the separate low-frequency set (every
 * token kept and every window added). Size row_src, the packed rows, the
 * block's image rows (cap) and the unpack inputs to at least this; 0 for an
 * invalid shape.
 */
size_t hilo_row_capacity(const hilo_shape* shape);

/*
 * Outputs of hilo_split (device pointers, caller-allocated), N = H*W:
 *   labels   uint8 [B*N]  HILO_KEEP / HILO_POOL2 / HILO_POOL4 per token
 *   row_src  int32 [hilo_row_capacity]  for packed image row r
 *                         (0 <= r < cu_img[B]): the
 *                         token id of a kept row, else the window id of a
 *                         pooled row (2x2 window id (p/2)*(W/2) + q/2, 4x4
 *                         window id (p/4)*(W/4) + q/4)
 *   counts   int32 [B*3]  per image: kept tokens, 2x2 windows, 4x4 windows
 *   cu_img   int32 [B+1]  packed image-row offsets, cu_img[0] = 0
 *   tok_row  int32 [B*N]  the packed image row (0-based, without the B*T text
 *                         offset) each grid token reads its output from
 * Per image the packed rows are: kept tokens in raster order, then 2x2
 * windows in window-raster order, then 4x4 windows in window-raster order.
 * With shape.lf > 0: kept tokens, then every lf x lf window of the grid in
 * window-raster order (counts = kept, windows, 0; row_src of window rows =
 * the window id (p/lf)*(W/lf) + q/lf; tok_row of an HILO_LF token = its
 * window's row).
 */
typedef struct {
  uint8_t* labels;
  int32_t* row_src;
  int32_t* counts;
  int32_t* cu_img;
  int32_t* tok_row;
} hilo_split_out;

/*
 * Weights of one stream (text or image) of the MMDiT block: device pointers
 * in PyTorch nn.Linear layout, W[out, in] row-major, bias[out]. Attention
 * weights and all biases are bf16; the MLP matrices w_1 and w_2 are IEEE fp16
 * (convert a bf16 checkpoint once with hilo_convert_bf16_to_f16: exact for
 * every bf16 value in the fp16 normal range). The MLP runs with fp16
 * tensor-core operands (11-bit mantissa) because its two activation roundings
 * (LayerNorm output, GELU output) dominate the block's error budget; the
 * tensor-core rate is the same as for bf16.
 *   w_qkv [3d, d]  bf16; output columns: q (d) | k (d) | v (d); head h owns
 *                  columns h*head_dim .. (h+1)*head_dim - 1 of each part
 *   w_o   [d, d]   bf16
 *   w_1   [4d, d], w_2 [d, 4d]   fp16 (ignored when shape.mlp == 0)
 */
typedef struct {
  const void *w_qkv, *b_qkv, *w_o, *b_o, *w_1, *b_1, *w_2, *b_2;
} hilo_stream_weights;

typedef struct {
  hilo_stream_weights txt, img;
} hilo_block_weights;

/*
 * FP8 weights of one stream for hilo_block_forward_fp8: each matrix W[out, in]
 * as e4m3 codes with one fp32 dequantisation scale per output channel (row),
 * e.g. from hilo_quantize_rows_e4m3 of the bf16 matrix; biases bf16.
 *   w_*  uint8 e4m3 [out, in], 16-byte aligned
 *   s_*  fp32 [out], 16-byte aligned: W[o, i] ~ e4m3(w[o, i]) * s[o]
 */
typedef struct {
  const void *w_qkv, *w_o, *w_1, *w_2;
  const float *s_qkv, *s_o, *s_1, *s_2;
  const void *b_qkv, *b_o, *b_1, *b_2;
} hilo_stream_weights_fp8;

typedef struct {
  hilo_stream_weights_fp8 txt, img;
} hilo_block_weights_fp8;

/* Readable name of a status code. */
const char* hilo_status_string(int status);

/* Detail of the last error returned to the calling thread ("" if none). */
const char* hilo_last_error(void);

/*
 * Synchronises `stream`, then reads and clears the device error words.
 * Returns HILO_OK, HILO_ERR_TIMEOUT if a device-side bounded wait ran out
 * since the last call, HILO_ERR_CHECK if (in the checks build of the
 * library, compiled with -DHILO_DEVICE_CHECKS) a kernel found an index read
 * from device data out of range and skipped that access, or HILO_ERR_CUDA
 * if the stream reported an error.
 */
int hilo_sync_status(void* stream);

/*
 * hilo_debug_wait_timeout -- test hook for the device-side failure path.
 * Launches one CTA whose thread 0 waits, with the same bounded mbarrier wait
 * the tcgen05 kernels use (1 s limit on %globaltimer), on an mbarrier that
 * nothing arrives at. The wait runs out, latches its code in the probe's
 * device word and the kernel returns: nothing faults, traps or hangs. The
 * next hilo_sync_status(stream) returns HILO_ERR_TIMEOUT ("probe=3" in
 * hilo_last_error) and clears the word; the context stays usable.
 * Returns HILO_OK once launched, HILO_ERR_CUDA if the launch failed.
 */
int hilo_debug_wait_timeout(void* stream);

/* Number of SMs of the current device and whether it is sm_103 (1/0). */
int hilo_device_info(int* num_sms, int* is_sm103);

/*
 * hilo_score -- per-token high-frequency energy (paper Sec. 2.3: the
 * frequency map that decides which tokens keep full resolution; here the
 * token-space form, the energy of a token minus its 2x2 average-pooled then
 * nearest-upsampled value).
 *   x      bf16 [B, H, W, d]
 *   score  fp32 [B, H*W]   s_i = sum_c (x_ic - m_c)^2, m the mean of the
 *                          aligned 2x2 window holding token i
 * Arithmetic is fp32 in one fixed order: m = ((a + b) + (c + e)) * 0.25 over
 * the window members in raster order; channels are summed in groups of 8
 * consecutive channels, group g folded into partial g mod 128 (groups and
 * channels ascending), partials combined by the halving tree p[j] += p[j + h]
 * for h = 64, 32, 16, 8, 4, 2, 1; no fused multiply-add. The result is therefore
 * bit-reproducible by any IEEE fp32 implementation of the same order.
 */
int hilo_score(const hilo_shape* shape, const void* x, float* score, void* stream);

/* Workspace bytes hilo_split needs (currently 0: NULL is accepted). */
size_t hilo_split_workspace_bytes(const hilo_shape* shape);

/*
 * hilo_split -- deterministic keep / pool split (paper Sec. 2.3: tokens
 * inside the edit mask are always retained, high-frequency tokens are
 * selected, the low-frequency rest is represented by pooled tokens).
 *   score   fp32 [B, N]   from hilo_score (finite, >= 0)
 *   mask    uint8 [B, N]  nonzero = edit-mask token (always kept)
 *   k_keep  int32 [B]     device; top-k budget per image, 0 <= k <= N
 *   k_mid   int32 [B]     device; levels == 2 only (else may be NULL):
 *                         the next k_mid tokens are pooled 2x2, the rest 4x4
 * Ranking is (score descending, token index ascending), so ties break by
 * index and the result is unique. kept = top-k_keep ∪ mask.
 * Values of k outside [0, N] are clamped on the device.
 */
int hilo_split(const hilo_shape* shape, const float* score, const uint8_t* mask,
               const int32_t* k_keep, const int32_t* k_mid, const hilo_split_out* out,
               void* ws, size_t ws_bytes, void* stream);

/*
 * hilo_split_regions -- the window-granular (regionalised) split: the token-
 * space reading of the coherent, region-level selection of paper Sec. 2.3.
 * Arguments, outputs and ranking are those of hilo_split; the labels then
 * give every pooling window the finest class of any of its members:
 *   - an aligned 2x2 window holding a token of top-k_keep ∪ mask is kept
 *     whole (all four members HILO_KEEP);
 *   - levels == 2: the remaining tokens are ranked as in hilo_split and the
 *     first k_mid are "above the cut"; an aligned 4x4 block is pooled 4x4
 *     only when all 16 members are below the cut, otherwise its non-kept
 *     members are pooled 2x2.
 * Every pooled window is therefore full (4 or 16 members), and kept regions
 * are whole 2x2 windows. Errors as hilo_split.
 */
int hilo_split_regions(const hilo_shape* shape, const float* score, const uint8_t* mask,
                       const int32_t* k_keep, const int32_t* k_mid, const hilo_split_out* out,
                       void* ws, size_t ws_bytes, void* stream);

/* Workspace bytes hilo_sobel_select needs (token maxima and one maximum per
 * 32 x 64-pixel tile). */
size_t hilo_sobel_workspace_bytes(const hilo_shape* shape);

/*
 * hilo_sobel_select -- the paper's own token selector (Sec. 2.3 "HiLo-Token
 * Selection"): a Sobel spatial-frequency map of the input image, normalised
 * by its per-image maximum, thresholded and regionalised onto the token grid,
 * united with the user mask dilated by `radius` tokens. The keep map it
 * writes goes to hilo_split as the mask, with k_keep = 0, for an
 * input-adaptive number of kept tokens.
 *   img        fp32 [B, H*patch, W*patch, channels], channels last, device;
 *              channels in [1, 4]
 *   patch      pixels per token side: 16 (the paper's 16x pooling) or 8
 *   mask       uint8 [B, H*W] device, nonzero = inside the edit mask
 *   radius     mask dilation in tokens (square window), in [0, 64]
 *   threshold  on the normalised map, finite; a token is selected when the
 *              largest normalised magnitude of its pixels is > threshold
 *   keep       uint8 [B, H*W] device output, 1 = kept
 *   ws         device workspace of hilo_sobel_workspace_bytes bytes, 16-byte
 *              aligned; overwritten
 * Per pixel and channel gx = ((P(y-1,x+1) + 2P(y,x+1)) + P(y+1,x+1)) -
 * ((P(y-1,x-1) + 2P(y,x-1)) + P(y+1,x-1)) and gy likewise over rows, with
 * replicate borders; g = sqrt(sum over channels ascending of (gx*gx +
 * gy*gy)); every step a correctly rounded fp32 operation, so the keep map is
 * reproducible bit for bit. The normalised value of a token is one correctly
 * rounded division tokmax / imgmax; an image with no gradient selects
 * nothing. Errors: HILO_ERR_ARG (NULL pointer, bad channels, patch, radius or
 * threshold), HILO_ERR_SHAPE, HILO_ERR_WORKSPACE, HILO_ERR_CUDA.
 */
int hilo_sobel_select(const hilo_shape* shape, const float* img, int channels, int patch,
                      const uint8_t* mask, int radius, float threshold, uint8_t* keep, void* ws,
                      size_t ws_bytes, void* stream);

/*
 * hilo_pack -- the packed image sequence (paper Sec. 2.3: selected tokens and
 * low-frequency tokens concatenated along the token axis).
 *   x       bf16 [B, H, W, d]
 *   split   the outputs of hilo_split for the same x
 *   packed  bf16 [cap, d]; rows [0, cu_img[B]) are written. A kept row is a
 *           copy of its token; a pooled row is the mean of the window's
 *           members of that class: fp32 sum in raster member order, one
 *           correctly rounded division by the member count, bf16 round to
 *           nearest even.
 */
int hilo_pack(const hilo_shape* shape, const void* x, const hilo_split_out* split,
              void* packed, int32_t cap, void* stream);

/* Workspace bytes hilo_block_forward needs for `cap` image-row capacity. */
size_t hilo_block_workspace_bytes(const hilo_shape* shape, int32_t cap);

/*
 * hilo_block_forward -- one MMDiT block on the row space (the DiT the
 * selected tokens feed, paper Sec. 2.1/2.3): for each stream s in {text,
 * image} with its own weights
 *     u += Attn(LN(u) W_qkv^s + b_qkv^s) W_o^s + b_o^s
 *     u += GELU_tanh(LN(u) W_1^s + b_1^s) W_2^s + b_2^s        (mlp == 1)
 * where LN has no affine parameters (eps 1e-6, biased variance) and the
 * attention of image b is non-causal softmax attention over the joint
 * sequence [its T text rows ; its packed image rows], scale 1/sqrt(head_dim).
 *   in_txt   [B*T, d] text rows,  dtype in_dtype (HILO_BF16 or HILO_F32)
 *   in_img   [cap, d] packed image rows, dtype in_dtype
 *   cu_img   int32 [B+1] device, from hilo_split (any non-decreasing
 *            offsets: rows past cap are not part of the block).
 *   out      fp32 [B*T + cap, d]: the residual stream after the block, text
 *            rows first (row space). With in_dtype == HILO_F32, in-place use
 *            (in_txt == out, in_img == out + B*T*d) is allowed.
 * in_txt, in_img and out must be 16-byte aligned (HILO_ERR_ARG otherwise).
 * QKV / out-projection GEMM operands and attention inputs are bf16, the MLP
 * GEMM operands fp16 (saturating conversion), all with fp32 accumulation; the
 * residual stream stays fp32.
 */
int hilo_block_forward(const hilo_shape* shape, const hilo_block_weights* weights,
                       const int32_t* cu_img, int32_t cap, const void* in_txt,
                       const void* in_img, int in_dtype, float* out, void* ws,
                       size_t ws_bytes, void* stream);

/*
 * hilo_row_sizes -- the number of grid tokens each packed image row stands
 * for: 1 for a kept token, the number of its class members for a pooled
 * window. These are the weights of proportional attention.
 *   split  outputs of hilo_split or hilo_split_regions
 *   n_img  fp32 [cap] device; rows [0, cu_img[B]) are written
 */
int hilo_row_sizes(const hilo_shape* shape, const hilo_split_out* split, float* n_img, int32_t cap,
                   void* stream);

/*
 * hilo_block_forward_prop -- hilo_block_forward with proportional attention
 * for pooled tokens: as a key, packed image row r adds ln(n_img[r]) to its
 * logits (text keys add 0), so a row standing for n grid tokens draws the
 * attention of n identical copies of itself:
 *     softmax_j(s_ij + ln n_j) = n_j e^(s_ij) / sum_k n_k e^(s_ik).
 * The paper does not say how pooled tokens attend; this weighting keeps the
 * attention mass of the uncompressed sequence. The kernel multiplies each
 * probability by n_j before the row sum and the bf16 rounding of P.
 *   n_img  fp32 [cap] device, 4-byte aligned, positive; e.g. hilo_row_sizes
 * Other arguments, layouts and errors as hilo_block_forward (HILO_ERR_ARG
 * for a NULL or unaligned n_img).
 */
int hilo_block_forward_prop(const hilo_shape* shape, const hilo_block_weights* weights,
                            const int32_t* cu_img, int32_t cap, const void* in_txt,
                            const void* in_img, int in_dtype, const float* n_img, float* out,
                            void* ws, size_t ws_bytes, void* stream);

/*
 * hilo_unpack -- back to the full grid (nearest broadcast): every token reads
 * the block output of its kept row or of its window's row.
 *   out_img  fp32 [cap, d]  image rows of the block output (out + B*T*d)
 *   y        fp32 [B, H, W, d]   y[b, i] = out_img[tok_row[b, i]]
 */
int hilo_unpack(const hilo_shape* shape, const float* out_img, const hilo_split_out* split,
                float* y, void* stream);

/*
 * hilo_unpack_delta -- back to the full grid with the delta unpool: a kept
 * token takes its own output row; a pooled member keeps its own value and
 * receives its window's update,
 *     y[b, i] = x[b, i] + (out_img[r] - packed[r]),   r = tok_row[b, i],
 * one fp32 subtract then one fp32 add, x and packed widened from bf16.
 *   out_img  fp32 [cap, d]  image rows of the block output
 *   packed   bf16 [cap, d]  the block's input rows, as hilo_pack wrote them
 *   x        bf16 [B, H, W, d]  the tokens hilo_pack read
 *   y        fp32 [B, H, W, d]
 * All four pointers 16-byte aligned (HILO_ERR_ARG otherwise).
 */
int hilo_unpack_delta(const hilo_shape* shape, const float* out_img, const void* packed, const void* x,
                      const hilo_split_out* split, float* y, void* stream);

/*
 * hilo_unpack_update -- unpack fused with the denoising-loop update
 *   x[b, i] <- bf16(x[b, i] - alpha * out_img[tok_row[b, i]])
 * computed as an fp32 multiply, then an fp32 subtract (no fused
 * multiply-add), then bf16 round to nearest even. x is bf16 [B, H, W, d],
 * updated in place.
 */
int hilo_unpack_update(const hilo_shape* shape, const float* out_img,
                       const hilo_split_out* split, void* x, float alpha, void* stream);

/*
 * hilo_quantize_rows_e4m3 -- per-row e4m3 quantisation: for each row, amax =
 * the largest magnitude, inv = 448 / amax and scale = amax / 448 (correctly
 * rounded fp32 divisions; 1 and 1 for an all-zero row), dst = e4m3(src * inv)
 * with the product rounded to fp32, then round to nearest even and saturate
 * at +-448. Used for the weights of hilo_block_forward_fp8 (once, at load)
 * and, inside it, for the attention output and the MLP hidden rows.
 *   src    [rows, cols] device, HILO_BF16, HILO_F16 or HILO_F32, 16-byte aligned
 *   dst    uint8 e4m3 [rows, cols] device, 16-byte aligned; cols a multiple of 8
 *   scale  fp32 [rows] device
 */
int hilo_quantize_rows_e4m3(const void* src, int src_dtype, int64_t rows, int32_t cols, uint8_t* dst,
                            float* scale, void* stream);

/* Workspace bytes hilo_block_forward_fp8 needs for `cap` image-row capacity. */
size_t hilo_block_fp8_workspace_bytes(const hilo_shape* shape, int32_t cap);

/*
 * hilo_block_forward_fp8 -- the block of hilo_block_forward with e4m3 GEMM
 * operands and fp32 accumulation (paper Sec. 3.3 reports FP8 on top of
 * HiLo-Token; this scaling scheme is the library's): every GEMM input row is
 * quantised per row (the LayerNorm outputs inside the LayerNorm kernel, the
 * attention output and the MLP hidden rows by a row pass), the weights per
 * output channel; each output is acc * row scale * column scale + bias. The
 * q|k|v rows, the attention and the residual stream are as in
 * hilo_block_forward (bf16 / fp32); the MLP hidden rows are fp16 before
 * their quantisation. Needs d a multiple of 256 and at least 1024 (else
 * HILO_ERR_SHAPE). Other arguments, layouts, in-place use and errors as
 * hilo_block_forward, with hilo_block_fp8_workspace_bytes of workspace.
 */
int hilo_block_forward_fp8(const hilo_shape* shape, const hilo_block_weights_fp8* weights,
                           const int32_t* cu_img, int32_t cap, const void* in_txt, const void* in_img,
                           int in_dtype, float* out, void* ws, size_t ws_bytes, void* stream);

/*
 * hilo_block_forward_fp8_prop -- hilo_block_forward_fp8 with the proportional
 * attention of hilo_block_forward_prop: as a key, packed image row r adds
 * ln(n_img[r]) to its logits (text keys add 0), the kernel multiplying each
 * probability by n_img[r] before the row sum and the bf16 rounding of P.
 * The paper gives neither FP8 scheme nor pooled-token attention (Sec. 3.3,
 * Sec. 2.3); both are this library's readings. n_img: fp32 [cap] device,
 * 4-byte aligned, from hilo_row_sizes. Other arguments, layouts and errors
 * as hilo_block_forward_fp8.
 */
int hilo_block_forward_fp8_prop(const hilo_shape* shape, const hilo_block_weights_fp8* weights,
                                const int32_t* cu_img, int32_t cap, const void* in_txt, const void* in_img,
                                int in_dtype, const float* n_img, float* out, void* ws, size_t ws_bytes,
                                void* stream);

/*
 * hilo_block_forward_static_ws -- hilo_block_forward without a workspace
 * argument, for callers that cannot allocate device memory at call time (code
 * inside a host framework whose allocator the call site cannot reach, or a
 * service that fixes its device-memory footprint at start-up). The paper has
 * no counterpart; this is a deployment convenience.
 *
 * The scratch is one fixed array of HILO_STATIC_SCRATCH_BYTES in the
 * library's own device memory; every GPU that loads the library holds it until
 * the process exits. The call allocates nothing. Arguments, layouts and
 * results are those of hilo_block_forward. Limits and caveats:
 *   - shapes whose hilo_block_workspace_bytes(shape, cap) exceeds
 *     HILO_STATIC_SCRATCH_BYTES are rejected with HILO_ERR_WORKSPACE (the
 *     detail in hilo_last_error()); e.g. d=512, T=64, 1024 image rows fits,
 *     the d=3072 blocks do not;
 *   - every call looks up the array's device address in the current device's
 *     context (nothing is cached across calls, so a device reset or another
 *     context is safe); the first call on a device also loads the library's
 *     device code, so make it before any stream capture;
 *   - an invalid shape returns HILO_ERR_SHAPE before any size check;
 *   - all calls share the one array: calls that overlap on the GPU (other
 *     streams, other host threads) race and must be serialised by the caller.
 *     No part of the array needs to start at zero.
 */
#define HILO_STATIC_SCRATCH_BYTES (16u << 20)
int hilo_block_forward_static_ws(const hilo_shape* shape, const hilo_block_weights* weights,
                                 const int32_t* cu_img, int32_t cap, const void* in_txt,
                                 const void* in_img, int in_dtype, float* out, void* stream);

/*
 * hilo_convert_bf16_to_f16 -- dst[i] = fp16(src[i]) for n elements (n a
 * multiple of 8, both pointers 16-byte aligned, device memory), round to
 * nearest even, saturating at +-65504. For preparing the fp16 MLP weights
 * once at load time (no counterpart in the paper).
 */
int hilo_convert_bf16_to_f16(const void* src, void* dst, size_t n, void* stream);

/*
 * Instrumentation (no counterpart in the paper; used by the benchmark).
 *
 * hilo_set_stage_events -- register up to 16 CUDA events (cudaEvent_t as
 * void*) for the calling thread. While registered, hilo_block_forward records
 * events[k] on its stream at the stage boundaries k = 0..7: before the first
 * LayerNorm, after it, after the QKV GEMM, after attention, after the
 * out-projection GEMM, after the second LayerNorm, after the MLP1 GEMM and
 * after the MLP2 GEMM (k = 5..7 only when mlp == 1). The caller owns the
 * events; n = 0 unregisters them. Returns HILO_ERR_ARG for n outside [0, 16].
 *
 * hilo_launch_count -- number of kernels libhilo has launched in this process.
 */
int hilo_set_stage_events(void* const* events, int n);
unsigned long long hilo_launch_count(void);

#ifdef __cplusplus
}
#endif

#endif /* HILO_H */
