// The paper's token selector (Sec. 2.3 "HiLo-Token Selection"): a Sobel
// frequency map of the input image, normalised by its per-image maximum,
// thresholded and regionalised onto the token grid (each token covers P x P
// pixels), united with the user mask dilated by R tokens.
//
// Two kernels:
//   sobel_tokmax_kernel  one CTA per 32 x 64 pixel tile (plus a one-pixel
//                        halo, replicate borders) in shared memory; each
//                        pixel's gradient magnitude in the fixed fp32 order
//                        below; the largest magnitude of each token from
//                        per-thread maxima, a warp reduction over the lanes
//                        of one token and one shared atomic per token and
//                        warp, on the float bits (magnitudes are >= +0, so
//                        their bit patterns order like the values); then one
//                        global atomic per token for the image maximum.
//   sobel_keep_kernel    one CTA per 16 x 16 tokens, the mask tile and a halo
//                        of R tokens in shared memory; per token: tokmax /
//                        imgmax (one correctly rounded division) > threshold,
//                        or any mask token within R tokens (square window).
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

template <int P, int C>
__global__ void __launch_bounds__(SOBEL_THREADS) sobel_tokmax_kernel(const float* __restrict__ img,
                                                                     float* __restrict__ tokmax,
                                                                     uint32_t* __restrict__ imgmax, int H,
                                                                     int W) {
  pdl_trigger();
  pdl_wait();
  constexpr int TOK_Y = TILE_Y / P, TOK_X = TILE_X / P;
  __shared__ float tile[C][TILE_Y + 2][TILE_X + 2];
  __shared__ uint32_t tmax[TOK_Y * TOK_X];
  const int Hp = H * P, Wp = W * P;
  const int b = blockIdx.z;
  const int y0 = blockIdx.y * TILE_Y, x0 = blockIdx.x * TILE_X;
  const float* base = img + static_cast<long long>(b) * Hp * Wp * C;
  // the tile and its halo: each row is one contiguous run of (TILE_X + 2) * C
  // floats (clamped at the image edges); every load of the thread is issued
  // before the first store, so the whole tile is in flight at once
  constexpr int ROW = (TILE_X + 2) * C;
  constexpr int TOTAL = (TILE_Y + 2) * ROW;
  constexpr int PER = (TOTAL + SOBEL_THREADS - 1) / SOBEL_THREADS;
  float v[PER];
#pragma unroll
  for (int k = 0; k < PER; ++k) {
    const int e = threadIdx.x + k * SOBEL_THREADS;
    if (e < TOTAL) {
      const int yy = e / ROW, w = e - yy * ROW;
      const int xx = w / C, c = w - xx * C;
      const int gy = min(max(y0 + yy - 1, 0), Hp - 1);
      const int gx = min(max(x0 + xx - 1, 0), Wp - 1);
      v[k] = __ldg(base + (static_cast<long long>(gy) * Wp + gx) * C + c);
    }
  }
#pragma unroll
  for (int k = 0; k < PER; ++k) {
    const int e = threadIdx.x + k * SOBEL_THREADS;
    if (e < TOTAL) {
      const int yy = e / ROW, w = e - yy * ROW;
      const int xx = w / C, c = w - xx * C;
      tile[c][yy][xx] = v[k];
    }
  }
  if (threadIdx.x < TOK_Y * TOK_X) tmax[threadIdx.x] = 0u;
  __syncthreads();
  // Thread t takes pixel column tx = t % 64 of rows ty0, ty0 + 4, ..., so a
  // warp covers 32 consecutive columns (32 / P tokens) of one row at a time;
  // each thread keeps one maximum per token row it visits, the lanes of one
  // token combine them with a warp reduction, and one lane per token issues
  // the shared atomic.
  constexpr int RSTEP = SOBEL_THREADS / TILE_X;  // rows between a thread's pixels
  static_assert(SOBEL_THREADS % TILE_X == 0 && 32 % P == 0 && P % RSTEP == 0, "tile mapping");
  const int tx = threadIdx.x % TILE_X, ty0 = threadIdx.x / TILE_X;
  uint32_t mx[TOK_Y];
#pragma unroll
  for (int k = 0; k < TOK_Y; ++k) mx[k] = 0u;
#pragma unroll
  for (int j = 0; j < TILE_Y / RSTEP; ++j) {
    const int ty = ty0 + RSTEP * j;
    if (y0 + ty >= Hp || x0 + tx >= Wp) continue;
    const int r = ty + 1, q = tx + 1;  // position in the padded tile
    float acc = 0.0f;
#pragma unroll
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
    const uint32_t g = __float_as_uint(__fsqrt_rn(acc));
    // ty0 < RSTEP and RSTEP divides P, so the token row is (RSTEP j) / P
    mx[(RSTEP * j) / P] = max(mx[(RSTEP * j) / P], g);
  }
  const int lane = threadIdx.x & 31;
  const uint32_t seg = (P >= 32 ? 0xffffffffu : ((1u << P) - 1u)) << (lane & ~(P - 1));
#pragma unroll
  for (int k = 0; k < TOK_Y; ++k) {
    const uint32_t m = __reduce_max_sync(seg, mx[k]);
    if ((lane & (P - 1)) == 0) atomicMax(&tmax[k * TOK_X + tx / P], m);
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

// One CTA per 16 x 16 tokens: the mask tile with a halo of `radius` tokens
// in shared memory, then each token's normalised maximum and its dilation
// window (radius <= MAX_RADIUS).
constexpr int KEEP_T = 16;
constexpr int MAX_RADIUS = 64;

__global__ void __launch_bounds__(KEEP_T * KEEP_T) sobel_keep_kernel(const float* __restrict__ tokmax,
                                                                   const uint32_t* __restrict__ imgmax,
                                                                   const uint8_t* __restrict__ mask,
                                                                   uint8_t* __restrict__ keep, int H, int W,
                                                                   int radius, float threshold) {
  pdl_trigger();
  pdl_wait();
  __shared__ uint8_t mt[KEEP_T + 2 * MAX_RADIUS][KEEP_T + 2 * MAX_RADIUS];
  const int b = blockIdx.z;
  const int i0 = blockIdx.y * KEEP_T - radius, j0 = blockIdx.x * KEEP_T - radius;
  const int S = KEEP_T + 2 * radius;
  const uint8_t* mb = mask + static_cast<long long>(b) * H * W;
  for (int e = threadIdx.x; e < S * S; e += blockDim.x) {
    const int ii = i0 + e / S, jj = j0 + e % S;
    mt[e / S][e % S] = (ii >= 0 && ii < H && jj >= 0 && jj < W) ? mb[ii * W + jj] : 0;
  }
  __syncthreads();
  const int ti = threadIdx.x / KEEP_T, tj = threadIdx.x % KEEP_T;
  const int i = blockIdx.y * KEEP_T + ti, j = blockIdx.x * KEEP_T + tj;
  if (i >= H || j >= W) return;
  const long long t = (static_cast<long long>(b) * H + i) * W + j;
  // 0 / 0 (an image without any gradient) is NaN and selects nothing
  const float f = __fdiv_rn(tokmax[t], __uint_as_float(imgmax[b]));
  bool k = f > threshold;
  for (int di = 0; di <= 2 * radius && !k; ++di)
    for (int dj = 0; dj <= 2 * radius; ++dj)
      if (mt[ti + di][tj + dj]) {
        k = true;
        break;
      }
  keep[t] = k ? 1 : 0;
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
#define HILO_SOBEL_CASE(PP, CC)                                                                        \
  if (patch == PP && C == CC)                                                                          \
    e = launch_pdl(sobel_tokmax_kernel<PP, CC>, grid, dim3(SOBEL_THREADS), 0, st, img, tokmax, imgmax, H, W);
  e = cudaErrorInvalidValue;
  HILO_SOBEL_CASE(16, 1) HILO_SOBEL_CASE(16, 2) HILO_SOBEL_CASE(16, 3) HILO_SOBEL_CASE(16, 4)
  HILO_SOBEL_CASE(8, 1) HILO_SOBEL_CASE(8, 2) HILO_SOBEL_CASE(8, 3) HILO_SOBEL_CASE(8, 4)
#undef HILO_SOBEL_CASE
  if (e != cudaSuccess) return e;
  if (radius > MAX_RADIUS) return cudaErrorInvalidValue;
  const dim3 kgrid((W + KEEP_T - 1) / KEEP_T, (H + KEEP_T - 1) / KEEP_T, B);
  return launch_pdl(sobel_keep_kernel, kgrid, dim3(KEEP_T * KEEP_T), 0, st, static_cast<const float*>(tokmax),
                    static_cast<const uint32_t*>(imgmax), mask, keep, H, W, radius, threshold);
}

}  // namespace hilo
