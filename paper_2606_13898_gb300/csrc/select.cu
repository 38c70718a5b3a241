// The paper's token selector (Sec. 2.3 "HiLo-Token Selection"): a Sobel
// frequency map of the input image, normalised by its per-image maximum,
// thresholded and regionalised onto the token grid (each token covers P x P
// pixels), united with the user mask dilated by R tokens.
//
// Two kernels:
//   sobel_tokmax_kernel  one CTA per 32 x 64 pixel tile (plus a one-pixel
//                        halo, replicate borders) in shared memory, channel
//                        planes; full-width tiles load their interior as
//                        16-byte vectors. Each thread walks 8 consecutive
//                        pixel rows of one column, so the horizontal sums of
//                        a row serve as the bottom term of one pixel and the
//                        top term of the pixel two rows below (the same
//                        value, not a re-association). The largest magnitude
//                        of each token comes from per-thread maxima, a warp
//                        reduction over the lanes of one token and one shared
//                        atomic per token and warp, on the float bits
//                        (magnitudes are >= +0, so their bit patterns order
//                        like the values); the tile's maximum goes to its own
//                        slot (no global atomics, nothing to clear).
//   sobel_keep_kernel    one CTA per 16 x 16 tokens: the image maximum from
//                        the tile slots, the mask tile and a halo of R
//                        tokens in shared memory; per token: tokmax / imgmax
//                        (one correctly rounded division) > threshold, or
//                        any mask token within R tokens (square window).
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
constexpr int ROWS = TILE_Y / (SOBEL_THREADS / TILE_X);  // consecutive pixel rows per thread

// (a + 2 b) + c, each step rounded to fp32
__device__ __forceinline__ float sobel_sum3(float a, float b, float c) {
  return __fadd_rn(__fadd_rn(a, __fmul_rn(2.0f, b)), c);
}

// Tiles of the tokmax grid for an H x W-token image at `patch` pixels per
// token: one maximum slot each.
inline int sobel_tiles(int H, int W, int patch) {
  return ((W * patch + TILE_X - 1) / TILE_X) * ((H * patch + TILE_Y - 1) / TILE_Y);
}

template <int P, int C>
__global__ void __launch_bounds__(SOBEL_THREADS) sobel_tokmax_kernel(const float* __restrict__ img,
                                                                     float* __restrict__ tokmax,
                                                                     uint32_t* __restrict__ tilemax, int H,
                                                                     int W, int vec_ok) {
  pdl_trigger();
  pdl_wait();
  constexpr int TOK_Y = TILE_Y / P, TOK_X = TILE_X / P;
  static_assert(TOK_Y * TOK_X <= 32, "token maxima of a tile fit one warp");
  __shared__ float tile[C][TILE_Y + 2][TILE_X + 2];
  __shared__ uint32_t tmax[TOK_Y * TOK_X];
  const int Hp = H * P, Wp = W * P;
  const int b = blockIdx.z;
  const int y0 = blockIdx.y * TILE_Y, x0 = blockIdx.x * TILE_X;
  const float* base = img + static_cast<long long>(b) * Hp * Wp * C;
  if (threadIdx.x < TOK_Y * TOK_X) tmax[threadIdx.x] = 0u;
  if (vec_ok && x0 + TILE_X <= Wp) {
    // Interior columns x0 .. x0 + 63 of each (row-clamped) tile row are
    // 64 C contiguous floats starting at a multiple of 4 floats (x0 is a
    // multiple of 64, Wp of 8, the image 16-byte aligned): 16 C vectors. The
    // two halo columns are single floats. Every load is issued before the
    // first shared store, so the whole tile is in flight at once.
    constexpr int V = TILE_X * C / 4;
    constexpr int NV = (TILE_Y + 2) * V;
    constexpr int PERV = (NV + SOBEL_THREADS - 1) / SOBEL_THREADS;
    constexpr int NH = (TILE_Y + 2) * 2 * C;
    constexpr int PERH = (NH + SOBEL_THREADS - 1) / SOBEL_THREADS;
    float4 v[PERV];
    float h[PERH];
#pragma unroll
    for (int k = 0; k < PERV; ++k) {
      const int e = threadIdx.x + k * SOBEL_THREADS;
      if (e < NV) {
        const int yy = e / V, m = e - yy * V;
        const int gy = min(max(y0 + yy - 1, 0), Hp - 1);
        v[k] = __ldg(reinterpret_cast<const float4*>(base + (static_cast<long long>(gy) * Wp + x0) * C) + m);
      }
    }
#pragma unroll
    for (int k = 0; k < PERH; ++k) {
      const int e = threadIdx.x + k * SOBEL_THREADS;
      if (e < NH) {
        const int yy = e / (2 * C), w = e - yy * (2 * C);
        const int side = w / C, c = w - side * C;
        const int gy = min(max(y0 + yy - 1, 0), Hp - 1);
        const int gx = side ? min(x0 + TILE_X, Wp - 1) : max(x0 - 1, 0);
        h[k] = __ldg(base + (static_cast<long long>(gy) * Wp + gx) * C + c);
      }
    }
#pragma unroll
    for (int k = 0; k < PERV; ++k) {
      const int e = threadIdx.x + k * SOBEL_THREADS;
      if (e < NV) {
        const int yy = e / V, m = e - yy * V;
        int px = (4 * m) / C, c = 4 * m - px * C;
        const float f[4] = {v[k].x, v[k].y, v[k].z, v[k].w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          tile[c][yy][1 + px] = f[i];
          if (++c == C) {
            c = 0;
            ++px;
          }
        }
      }
    }
#pragma unroll
    for (int k = 0; k < PERH; ++k) {
      const int e = threadIdx.x + k * SOBEL_THREADS;
      if (e < NH) {
        const int yy = e / (2 * C), w = e - yy * (2 * C);
        const int side = w / C, c = w - side * C;
        tile[c][yy][side ? TILE_X + 1 : 0] = h[k];
      }
    }
  } else {
    // partial tiles (right image edge) and unaligned images: one clamped
    // float per element
    constexpr int ROW = (TILE_X + 2) * C;
    constexpr int TOTAL = (TILE_Y + 2) * ROW;
    for (int e = threadIdx.x; e < TOTAL; e += SOBEL_THREADS) {
      const int yy = e / ROW, w = e - yy * ROW;
      const int xx = w / C, c = w - xx * C;
      const int gy = min(max(y0 + yy - 1, 0), Hp - 1);
      const int gx = min(max(x0 + xx - 1, 0), Wp - 1);
      tile[c][yy][xx] = __ldg(base + (static_cast<long long>(gy) * Wp + gx) * C + c);
    }
  }
  __syncthreads();
  // Thread t takes pixel column tx = t % 64 and the ROWS consecutive rows
  // from ty0 = (t / 64) ROWS; ROWS divides P, so they all lie in token row
  // ty0 / P. A warp covers 32 consecutive columns (32 / P tokens).
  static_assert(SOBEL_THREADS % TILE_X == 0 && 32 % P == 0 && P % ROWS == 0, "tile mapping");
  const int tx = threadIdx.x % TILE_X, ty0 = (threadIdx.x / TILE_X) * ROWS;
  const int q = tx + 1;  // column in the padded tile
  // sliding 3-row window per channel: up/mid/dn rows at columns q-1, q, q+1,
  // and the horizontal sums of the up and mid rows
  float up[C][3], mid[C][3], hup[C], hmid[C];
#pragma unroll
  for (int c = 0; c < C; ++c) {
#pragma unroll
    for (int i = 0; i < 3; ++i) {
      up[c][i] = tile[c][ty0][q - 1 + i];
      mid[c][i] = tile[c][ty0 + 1][q - 1 + i];
    }
    hup[c] = sobel_sum3(up[c][0], up[c][1], up[c][2]);
    hmid[c] = sobel_sum3(mid[c][0], mid[c][1], mid[c][2]);
  }
  const bool col_ok = x0 + tx < Wp;
  uint32_t mx = 0u;
#pragma unroll
  for (int j = 0; j < ROWS; ++j) {
    const int r = ty0 + 1 + j;  // row in the padded tile
    float acc = 0.0f;
#pragma unroll
    for (int c = 0; c < C; ++c) {
      float dn[3];
#pragma unroll
      for (int i = 0; i < 3; ++i) dn[i] = tile[c][r + 1][q - 1 + i];
      const float hdn = sobel_sum3(dn[0], dn[1], dn[2]);                  // bottom
      const float right = sobel_sum3(up[c][2], mid[c][2], dn[2]);
      const float left = sobel_sum3(up[c][0], mid[c][0], dn[0]);
      const float gx = __fsub_rn(right, left);
      const float gy = __fsub_rn(hdn, hup[c]);                            // bottom - top
      acc = __fadd_rn(acc, __fadd_rn(__fmul_rn(gx, gx), __fmul_rn(gy, gy)));
#pragma unroll
      for (int i = 0; i < 3; ++i) {
        up[c][i] = mid[c][i];
        mid[c][i] = dn[i];
      }
      hup[c] = hmid[c];
      hmid[c] = hdn;
    }
    if (col_ok && y0 + ty0 + j < Hp) mx = max(mx, __float_as_uint(__fsqrt_rn(acc)));
  }
  const int lane = threadIdx.x & 31;
  const uint32_t seg = (P >= 32 ? 0xffffffffu : ((1u << P) - 1u)) << (lane & ~(P - 1));
  const uint32_t m = __reduce_max_sync(seg, mx);
  if ((lane & (P - 1)) == 0) atomicMax(&tmax[(ty0 / P) * TOK_X + tx / P], m);
  __syncthreads();
  if (threadIdx.x < 32) {
    uint32_t t = 0u;
    if (threadIdx.x < TOK_Y * TOK_X) {
      const int ti = blockIdx.y * TOK_Y + threadIdx.x / TOK_X;
      const int tj = blockIdx.x * TOK_X + threadIdx.x % TOK_X;
      if (ti < H && tj < W) {
        t = tmax[threadIdx.x];
        tokmax[(static_cast<long long>(b) * H + ti) * W + tj] = __uint_as_float(t);
      }
    }
    t = __reduce_max_sync(0xffffffffu, t);
    if (threadIdx.x == 0) tilemax[(static_cast<long long>(b) * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x] = t;
  }
}

// One CTA per 16 x 16 tokens: the image maximum from the tile slots, the
// mask tile with a halo of `radius` tokens in shared memory, then each
// token's normalised maximum and its dilation window (radius <= MAX_RADIUS).
constexpr int KEEP_T = 16;
constexpr int MAX_RADIUS = 64;

__global__ void __launch_bounds__(KEEP_T * KEEP_T) sobel_keep_kernel(const float* __restrict__ tokmax,
                                                                   const uint32_t* __restrict__ tilemax,
                                                                   int ntiles, const uint8_t* __restrict__ mask,
                                                                   uint8_t* __restrict__ keep, int H, int W,
                                                                   int radius, float threshold) {
  pdl_trigger();
  pdl_wait();
  __shared__ uint8_t mt[KEEP_T + 2 * MAX_RADIUS][KEEP_T + 2 * MAX_RADIUS];
  __shared__ uint32_t wred[KEEP_T * KEEP_T / 32];
  const int b = blockIdx.z;
  const int i0 = blockIdx.y * KEEP_T - radius, j0 = blockIdx.x * KEEP_T - radius;
  const int S = KEEP_T + 2 * radius;
  const uint8_t* mb = mask + static_cast<long long>(b) * H * W;
  for (int e = threadIdx.x; e < S * S; e += blockDim.x) {
    const int ii = i0 + e / S, jj = j0 + e % S;
    mt[e / S][e % S] = (ii >= 0 && ii < H && jj >= 0 && jj < W) ? mb[ii * W + jj] : 0;
  }
  uint32_t gm = 0u;
  const uint32_t* tb = tilemax + static_cast<long long>(b) * ntiles;
  for (int e = threadIdx.x; e < ntiles; e += blockDim.x) gm = max(gm, tb[e]);
  gm = __reduce_max_sync(0xffffffffu, gm);
  if ((threadIdx.x & 31) == 0) wred[threadIdx.x >> 5] = gm;
  __syncthreads();
  gm = wred[0];
#pragma unroll
  for (int w = 1; w < KEEP_T * KEEP_T / 32; ++w) gm = max(gm, wred[w]);
  const int ti = threadIdx.x / KEEP_T, tj = threadIdx.x % KEEP_T;
  const int i = blockIdx.y * KEEP_T + ti, j = blockIdx.x * KEEP_T + tj;
  if (i >= H || j >= W) return;
  const long long t = (static_cast<long long>(b) * H + i) * W + j;
  // 0 / 0 (an image without any gradient) is NaN and selects nothing
  const float f = __fdiv_rn(tokmax[t], __uint_as_float(gm));
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
  // token maxima, then one slot per tokmax tile at the larger tile count of
  // the two patch sizes (16 pixels per token)
  return static_cast<size_t>(B) * H * W * sizeof(float) + 256 +
         static_cast<size_t>(B) * sobel_tiles(H, W, 16) * sizeof(uint32_t);
}

cudaError_t launch_sobel_select(const float* img, int B, int H, int W, int C, int patch,
                                const uint8_t* mask, int radius, float threshold, uint8_t* keep, void* ws,
                                int num_sms, cudaStream_t st) {
  (void)num_sms;
  if (radius > MAX_RADIUS) return cudaErrorInvalidValue;
  float* tokmax = static_cast<float*>(ws);
  uint32_t* tilemax = reinterpret_cast<uint32_t*>(
      (reinterpret_cast<uintptr_t>(tokmax + static_cast<size_t>(B) * H * W) + 255) & ~static_cast<uintptr_t>(255));
  const int vec_ok = (reinterpret_cast<uintptr_t>(img) & 15) == 0;
  const dim3 grid((W * patch + TILE_X - 1) / TILE_X, (H * patch + TILE_Y - 1) / TILE_Y, B);
  cudaError_t e = cudaErrorInvalidValue;
#define HILO_SOBEL_CASE(PP, CC)                                                                         \
  if (patch == PP && C == CC)                                                                           \
    e = launch_pdl(sobel_tokmax_kernel<PP, CC>, grid, dim3(SOBEL_THREADS), 0, st, img, tokmax, tilemax, H, W, \
                   vec_ok);
  HILO_SOBEL_CASE(16, 1) HILO_SOBEL_CASE(16, 2) HILO_SOBEL_CASE(16, 3) HILO_SOBEL_CASE(16, 4)
  HILO_SOBEL_CASE(8, 1) HILO_SOBEL_CASE(8, 2) HILO_SOBEL_CASE(8, 3) HILO_SOBEL_CASE(8, 4)
#undef HILO_SOBEL_CASE
  if (e != cudaSuccess) return e;
  const dim3 kgrid((W + KEEP_T - 1) / KEEP_T, (H + KEEP_T - 1) / KEEP_T, B);
  return launch_pdl(sobel_keep_kernel, kgrid, dim3(KEEP_T * KEEP_T), 0, st, static_cast<const float*>(tokmax),
                    static_cast<const uint32_t*>(tilemax), sobel_tiles(H, W, patch), mask, keep, H, W, radius,
                    threshold);
}

}  // namespace hilo
