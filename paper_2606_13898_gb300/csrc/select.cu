// The paper's token selector (Sec. 2.3 "HiLo-Token Selection"): a Sobel
// frequency map of the input image, normalised by its per-image maximum,
// thresholded and regionalised onto the token grid (each token covers P x P
// pixels), united with the user mask dilated by R tokens.
//
// Two kernels:
//   sobel_tokmax_kernel  one CTA per 32 x 64 pixel tile (plus a one-pixel
//                        halo, replicate borders) in shared memory; each
//                        pixel's gradient magnitude in the fixed fp32 order
//                        below; the largest magnitude of each token by
//                        shared-memory atomics on the float bits (magnitudes
//                        are >= +0, so their bit patterns order like the
//                        values), then one global atomic per token for the
//                        image maximum.
//   sobel_keep_kernel    per token: tokmax / imgmax (one correctly rounded
//                        division) > threshold, or any mask token within R
//                        tokens (square window).
// Order of the magnitude, per channel c (P the replicate-padded pixels):
//   gx = ((P(y-1,x+1) + 2 P(y,x+1)) + P(y+1,x+1)) - ((P(y-1,x-1) + 2 P(y,x-1)) + P(y+1,x-1))
//   gy = ((P(y+1,x-1) + 2 P(y+1,x)) + P(y+1,x+1)) - ((P(y-1,x-1) + 2 P(y-1,x)) + P(y-1,x+1))
//   acc = acc + (gx gx + gy gy) over c ascending from 0;  g = sqrt(acc)
// with every operation an explicitly rounded fp32 add, mul or sqrt, so the
// keep map equals a CPU evaluation of the same definition bit for bit.
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"
#include "internal.h"

namespace hilo {

namespace {

constexpr int TILE_Y = 32;
constexpr int TILE_X = 64;
constexpr int SOBEL_THREADS = 256;
constexpr int MAX_CH = 4;

template <int P>
__global__ void __launch_bounds__(SOBEL_THREADS) sobel_tokmax_kernel(const float* __restrict__ img,
                                                                     float* __restrict__ tokmax,
                                                                     uint32_t* __restrict__ imgmax, int H,
                                                                     int W, int C) {
  pdl_trigger();
  pdl_wait();
  constexpr int TOK_Y = TILE_Y / P, TOK_X = TILE_X / P;
  __shared__ float tile[MAX_CH][TILE_Y + 2][TILE_X + 2];
  __shared__ uint32_t tmax[TOK_Y * TOK_X];
  const int Hp = H * P, Wp = W * P;
  const int b = blockIdx.z;
  const int y0 = blockIdx.y * TILE_Y, x0 = blockIdx.x * TILE_X;
  const float* base = img + static_cast<long long>(b) * Hp * Wp * C;
  for (int i = threadIdx.x; i < (TILE_Y + 2) * (TILE_X + 2) * C; i += SOBEL_THREADS) {
    const int c = i % C;
    const int xx = (i / C) % (TILE_X + 2);
    const int yy = i / (C * (TILE_X + 2));
    const int gy = min(max(y0 + yy - 1, 0), Hp - 1);
    const int gx = min(max(x0 + xx - 1, 0), Wp - 1);
    tile[c][yy][xx] = __ldg(base + (static_cast<long long>(gy) * Wp + gx) * C + c);
  }
  if (threadIdx.x < TOK_Y * TOK_X) tmax[threadIdx.x] = 0u;
  __syncthreads();
  for (int i = threadIdx.x; i < TILE_Y * TILE_X; i += SOBEL_THREADS) {
    const int ty = i / TILE_X, tx = i % TILE_X;
    if (y0 + ty >= Hp || x0 + tx >= Wp) continue;
    const int r = ty + 1, q = tx + 1;  // position in the padded tile
    float acc = 0.0f;
    for (int c = 0; c < C; ++c) {
      const float(*t)[TILE_X + 2] = tile[c];
      const float right = __fadd_rn(__fadd_rn(t[r - 1][q + 1], __fmul_rn(2.0f, t[r][q + 1])), t[r + 1][q + 1]);
      const float left = __fadd_rn(__fadd_rn(t[r - 1][q - 1], __fmul_rn(2.0f, t[r][q - 1])), t[r + 1][q - 1]);
      const float bottom = __fadd_rn(__fadd_rn(t[r + 1][q - 1], __fmul_rn(2.0f, t[r + 1][q])), t[r + 1][q + 1]);
      const float top = __fadd_rn(__fadd_rn(t[r - 1][q - 1], __fmul_rn(2.0f, t[r - 1][q])), t[r - 1][q + 1]);
      const float gx = __fsub_rn(right, left);
      const float gy = __fsub_rn(bottom, top);
      acc = __fadd_rn(acc, __fadd_rn(__fmul_rn(gx, gx), __fmul_rn(gy, gy)));
    }
    const float g = __fsqrt_rn(acc);
    atomicMax(&tmax[(ty / P) * TOK_X + tx / P], __float_as_uint(g));
  }
  __syncthreads();
  if (threadIdx.x < TOK_Y * TOK_X) {
    const int ti = blockIdx.y * TOK_Y + threadIdx.x / TOK_X;
    const int tj = blockIdx.x * TOK_X + threadIdx.x % TOK_X;
    if (ti < H && tj < W) {
      const uint32_t v = tmax[threadIdx.x];
      tokmax[(static_cast<long long>(b) * H + ti) * W + tj] = __uint_as_float(v);
      atomicMax(imgmax + b, v);
    }
  }
}

__global__ void __launch_bounds__(256) sobel_keep_kernel(const float* __restrict__ tokmax,
                                                         const uint32_t* __restrict__ imgmax,
                                                         const uint8_t* __restrict__ mask,
                                                         uint8_t* __restrict__ keep, int B, int H, int W,
                                                         int radius, float threshold) {
  pdl_trigger();
  pdl_wait();
  const long long n = static_cast<long long>(B) * H * W;
  for (long long t = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; t < n;
       t += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int b = static_cast<int>(t / (static_cast<long long>(H) * W));
    const int i = static_cast<int>((t / W) % H), j = static_cast<int>(t % W);
    // 0 / 0 (an image without any gradient) is NaN and selects nothing
    const float f = __fdiv_rn(tokmax[t], __uint_as_float(imgmax[b]));
    bool k = f > threshold;
    const uint8_t* mb = mask + static_cast<long long>(b) * H * W;
    for (int ii = max(0, i - radius); ii <= min(H - 1, i + radius) && !k; ++ii)
      for (int jj = max(0, j - radius); jj <= min(W - 1, j + radius); ++jj)
        if (mb[ii * W + jj]) {
          k = true;
          break;
        }
    keep[t] = k ? 1 : 0;
  }
}

}  // namespace

size_t sobel_workspace_bytes(int B, int H, int W) {
  return static_cast<size_t>(B) * H * W * sizeof(float) + 256 + static_cast<size_t>(B) * sizeof(uint32_t);
}

cudaError_t launch_sobel_select(const float* img, int B, int H, int W, int C, int patch,
                                const uint8_t* mask, int radius, float threshold, uint8_t* keep, void* ws,
                                int num_sms, cudaStream_t st) {
  float* tokmax = static_cast<float*>(ws);
  uint32_t* imgmax = reinterpret_cast<uint32_t*>(
      (reinterpret_cast<uintptr_t>(tokmax + static_cast<size_t>(B) * H * W) + 255) & ~static_cast<uintptr_t>(255));
  cudaError_t e = cudaMemsetAsync(imgmax, 0, static_cast<size_t>(B) * sizeof(uint32_t), st);
  if (e != cudaSuccess) return e;
  const dim3 grid((W * patch + TILE_X - 1) / TILE_X, (H * patch + TILE_Y - 1) / TILE_Y, B);
  if (patch == 16)
    e = launch_pdl(sobel_tokmax_kernel<16>, grid, dim3(SOBEL_THREADS), 0, st, img, tokmax, imgmax, H, W, C);
  else if (patch == 8)
    e = launch_pdl(sobel_tokmax_kernel<8>, grid, dim3(SOBEL_THREADS), 0, st, img, tokmax, imgmax, H, W, C);
  else
    return cudaErrorInvalidValue;
  if (e != cudaSuccess) return e;
  const long long n = static_cast<long long>(B) * H * W;
  long long g = (n + 255) / 256;
  if (g > static_cast<long long>(num_sms) * 8) g = static_cast<long long>(num_sms) * 8;
  return launch_pdl(sobel_keep_kernel, dim3(static_cast<int>(g)), dim3(256), 0, st,
                    static_cast<const float*>(tokmax), static_cast<const uint32_t*>(imgmax), mask, keep, B, H, W,
                    radius, threshold);
}

}  // namespace hilo
