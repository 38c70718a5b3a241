// Internal launch interface between the C ABI (api.cu) and the kernel files.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/hilo.h"

#define HILO_LABEL_KEEP 0
#define HILO_LABEL_POOL2 1
#define HILO_LABEL_POOL4 2
#define HILO_LABEL_LF 3

namespace hilo {

// ---- bandwidth kernels (bw_kernels.cu)
cudaError_t launch_score(const void* x, float* s, int B, int H, int W, int d, int num_sms,
                         cudaStream_t st);
size_t split_select_smem(int N);
size_t split_compact_smem(int N);
cudaError_t launch_split(const float* score, const uint8_t* mask, const int32_t* k_keep,
                         const int32_t* k_mid, uint8_t* labels, int32_t* row_src, int32_t* counts,
                         int32_t* cu_img, int32_t* tok_row, int B, int H, int W, int levels,
                         int granular, int lf, cudaStream_t st);
cudaError_t launch_pack(const void* x, const uint8_t* labels, const int32_t* row_src,
                        const int32_t* counts, const int32_t* cu_img, void* packed, int B, int H,
                        int W, int d, int cap, int lf, int num_sms, cudaStream_t st);
// rows_max: rows of out_img (the row capacity); a token row at or past it
// is an error of the checks build
cudaError_t launch_unpack(const float* out_img, const int32_t* tok_row, float* y, long long ntok,
                          int d, long long rows_max, int num_sms, cudaStream_t st);
cudaError_t launch_row_sizes(const uint8_t* labels, const int32_t* row_src, const int32_t* counts,
                             const int32_t* cu_img, float* n_img, int B, int H, int W, int cap, int lf,
                             int num_sms, cudaStream_t st);
cudaError_t launch_unpack_delta(const float* out_img, const void* packed, const void* x,
                                const uint8_t* labels, const int32_t* tok_row, float* y, long long ntok,
                                int d, long long rows_max, int num_sms, cudaStream_t st);
cudaError_t launch_unpack_update(const float* out_img, const int32_t* tok_row, void* x,
                                 long long ntok, int d, float alpha, long long rows_max, int num_sms,
                                 cudaStream_t st);
cudaError_t launch_layernorm(const void* in_txt, const void* in_img, int in_f32, float* resid,
                             void* ln, int ln_mode, float* ln_scale, const int32_t* cu_img, int B, int n_txt,
                             int cap, int d, int num_sms, cudaStream_t st);
cudaError_t launch_quant_rows(const void* src, int type, int cols, int rows_static, const int32_t* cu_img,
                              int B, int n_txt, int cap, uint8_t* dst, float* scale, int num_sms,
                              cudaStream_t st);
cudaError_t launch_bf16_to_f16(const void* src, void* dst, long long n, int num_sms,
                               cudaStream_t st);

// ---- the paper's Sobel selector (select.cu)
size_t sobel_workspace_bytes(int B, int H, int W);
cudaError_t launch_sobel_select(const float* img, int B, int H, int W, int C, int patch,
                                const uint8_t* mask, int radius, float threshold, uint8_t* keep, void* ws,
                                int num_sms, cudaStream_t st);

// ---- tcgen05 grouped GEMM (gemm_tc.cu)
enum GemmEpilogue : int {
  EPI_BIAS_BF16 = 0,      // out_bf16 = acc + bias
  EPI_BIAS_GELU_F16 = 1,  // out_f16 = gelu_tanh(acc + bias)   (saturating)
  EPI_BIAS_RESID_F32 = 2, // out_f32 += acc + bias
  EPI_BIAS_RESIDIN_F32 = 3,  // out_f32 = resid_src + acc + bias (resid_src bf16 or fp32, per group)
};

// Two row groups of the row space share the A operand (one tensor map over
// all R rows) but use their own weights / bias. Group g covers rows
// [row_base_g, row_base_g + rows_g); rows_g is rows_static_g, or, when
// rows_dev_g is not null, read on the device from *rows_dev_g.
struct GemmGroupArgs {
  int row_base;
  int rows_static;
  const int32_t* rows_dev;
  const void* weight;  // bf16 [N, K] (e4m3 with GemmArgs::fp8)
  const void* bias;    // bf16 [N]
  int rows_cap;        // upper bound of rows (grid sizing)
  const float* w_scale = nullptr;  // fp8: dequantisation scale per output column
};

struct GemmArgs {
  const void* A;  // [R, K] row space, bf16 (op_f16 = 0) or fp16 (op_f16 = 1); W_g the same type
  int R, N, K;
  int op_f16;
  int fp8 = 0;                     // A and W_g e4m3 (kind::f8f6f4), pair kernel only
  const float* a_scale = nullptr;  // fp8: dequantisation scale per row of A
  GemmGroupArgs g[2];
  int epilogue;
  void* out;  // bf16 or f32 [R, N]
  // EPI_BIAS_RESIDIN_F32: the residual rows of group g start at resid_src[g]
  // (row stride N elements), fp32 when resid_f32 else bf16
  const void* resid_src[2] = {nullptr, nullptr};
  int resid_f32 = 0;
};

cudaError_t launch_gemm(const GemmArgs& a, int num_sms, cudaStream_t st);
int gemm_take_device_error();

// ---- tcgen05 grouped GEMM on CTA pairs, 256x256 tiles (gemm2_tc.cu)
bool gemm_pair_supported(const GemmArgs& a);
cudaError_t launch_gemm_pair(const GemmArgs& a, int num_sms, cudaStream_t st);
int gemm2_take_device_error();

// ---- tcgen05 joint varlen attention (attn_tc.cu)
struct AttnArgs {
  const void* qkv;  // bf16 [R, 3d]
  void* out;        // bf16 [R, d]
  const int32_t* cu_img;
  const float* n_img = nullptr;  // proportional attention: weight per packed image row
  int B, T, heads, head_dim, d, R;
};
cudaError_t launch_attention(const AttnArgs& a, int num_sms, cudaStream_t st);
int attn_take_device_error();
// The wait-timeout probe: one bounded mbarrier wait that runs out; its code
// is read (and cleared) like the kernels' device error words.
cudaError_t launch_wait_probe(cudaStream_t st);
int probe_take_device_error();
// The check word of the bandwidth kernels (checks build; 0 otherwise).
int dcheck_take_bw();

// ---- error text of the calling thread (api.cu)
int set_error(int status, const char* msg);
// The shape check of hilo_block_forward (HILO_OK, or the status it returns
// with the calling thread's error text set).
int check_block_shape(const hilo_shape* shape);

// ---- tensor maps (api.cu): 2-D, row-major, 128-byte swizzled boxes
enum TmapType : int { TMAP_BF16 = 0, TMAP_F16 = 1, TMAP_F32 = 2, TMAP_U8 = 3 };
bool encode_tmap_2d(CUtensorMap* map, TmapType type, const void* base, uint64_t inner, uint64_t outer,
                    uint64_t row_stride_elems, uint32_t box_inner, uint32_t box_outer);
bool encode_tmap_bf16_2d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
                         uint64_t row_stride_elems, uint32_t box_inner, uint32_t box_outer);

}  // namespace hilo
