// Epilogue of the tcgen05 GEMMs (gemm_tc.cu, gemm2_tc.cu): one warp turns
// the 32 accumulator rows of its TMEM lane quarter into output rows.
//
// For each 32-row slab the warp reads the accumulator 32 (fp32 outputs) or
// 64 (16-bit outputs) columns at a time with tcgen05.ld (lane = row), applies
// the bias and the epilogue function, and writes the 128-byte row pieces into
// a 128-byte-swizzled shared-memory box (32 rows x 128 B, two per warp, used
// in turn). One lane then hands the box to the TMA engine:
//   bf16 / fp16 outputs      bulk tensor store
//   fp32 += (residual in C)  bulk tensor reduce-add, so the old value is
//                            never loaded by the SM (and partial sums of a
//                            tile cut along K can be added independently)
//   fp32 = residual + ...    bulk tensor store; the residual rows are loaded
//                            one column chunk ahead of their use
// so every global write leaves the SM as whole 128-byte lines and the
// epilogue does not wait on memory latency. A slab that is only partly inside
// its row group (the ragged last tile of the image rows) is written with
// per-lane stores (atomic adds for +=) of the valid rows instead.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "common.cuh"
#include "internal.h"

namespace hilo {

constexpr int EPI_BOX_BYTES = 32 * 128;                   // one staging box
constexpr int EPI_WARP_BYTES = 2 * EPI_BOX_BYTES;         // two per warp
constexpr int EPI_SMEM_BYTES = 4 * EPI_WARP_BYTES;        // four epilogue warps

// GELU in its tanh form, 0.5 z (1 + tanh(u)) with u = sqrt(2/pi) (z + 0.044715 z^3).
// Since 0.5 (1 + tanh(u)) = 1 / (1 + e^(-2u)), it is evaluated as
// z / (1 + 2^(-2u log2 e)): one exp2 and one division.
__device__ __forceinline__ float gelu_tanh(float z) {
  constexpr float k = 2.0f * 0.7978845608028654f * 1.4426950408889634f;  // 2 sqrt(2/pi) log2(e)
  const float t = z * fmaf(0.044715f * z, z, 1.0f);
  float e;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(e) : "f"(-k * t));
  return __fdividef(z, 1.0f + e);
}

__device__ __forceinline__ void bf16x8(const uint4& v, float* f) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

// Byte offset of 16-byte unit j of row r in a 128-byte-swizzled box.
__device__ __forceinline__ uint32_t sw128_off(int r, int j) {
  return static_cast<uint32_t>(r * 128 + ((j ^ (r & 7)) << 4));
}

// This lane's 8 bias values, columns n0 + 8 lane .. + 7 of the tile (zero
// past N or past the tile's NC columns). Loaded before the accumulator is
// ready, so the load's latency is hidden behind the main loop; the chunks
// then take their values from the owning lane by shuffles.
template <int NC>
__device__ __forceinline__ uint4 epi_bias_preload(const __nv_bfloat16* bias, int n0, int N) {
  const int col = n0 + 8 * lane_id();
  if (8 * lane_id() < NC && col < N) return __ldg(reinterpret_cast<const uint4*>(bias + col));
  return make_uint4(0u, 0u, 0u, 0u);
}

// The 8 bias values held by lane `src` (warp-uniform).
__device__ __forceinline__ void epi_bias8(const uint4& b, int src, float* f) {
  uint4 v;
  v.x = __shfl_sync(0xffffffffu, b.x, src);
  v.y = __shfl_sync(0xffffffffu, b.y, src);
  v.z = __shfl_sync(0xffffffffu, b.z, src);
  v.w = __shfl_sync(0xffffffffu, b.w, src);
  bf16x8(v, f);
}

// FP8 dequantisation of one warp's slab: this lane's row scale and 8 column
// scales per lane (columns n0 + 8 lane .. + 7), taken per chunk by shuffles
// like the bias. `on` false: no scaling.
struct EpiScale {
  bool on = false;
  float sa = 1.0f;
  uint4 s0 = make_uint4(0u, 0u, 0u, 0u), s1 = make_uint4(0u, 0u, 0u, 0u);
};

template <int NC>
__device__ __forceinline__ EpiScale epi_scale_preload(const float* a_scale, const float* w_scale, int row0,
                                                      int nvalid, int n0, int N) {
  EpiScale e;
  e.on = true;
  const int lane = lane_id();
  e.sa = lane < nvalid ? __ldg(a_scale + row0 + lane) : 0.0f;
  const int col = n0 + 8 * lane;
  if (8 * lane < NC && col < N) {
    e.s0 = __ldg(reinterpret_cast<const uint4*>(w_scale + col));
    e.s1 = __ldg(reinterpret_cast<const uint4*>(w_scale + col + 4));
  }
  return e;
}

// The 8 column scales held by lane `src` (warp-uniform), times the row's.
__device__ __forceinline__ void epi_scale8(const EpiScale& e, int src, float* f) {
  const uint32_t w[8] = {__shfl_sync(0xffffffffu, e.s0.x, src), __shfl_sync(0xffffffffu, e.s0.y, src),
                         __shfl_sync(0xffffffffu, e.s0.z, src), __shfl_sync(0xffffffffu, e.s0.w, src),
                         __shfl_sync(0xffffffffu, e.s1.x, src), __shfl_sync(0xffffffffu, e.s1.y, src),
                         __shfl_sync(0xffffffffu, e.s1.z, src), __shfl_sync(0xffffffffu, e.s1.w, src)};
#pragma unroll
  for (int i = 0; i < 8; ++i) f[i] = e.sa * __uint_as_float(w[i]);
}

struct EpiSlab {
  int g;         // row group (weights / bias / residual source)
  int row0;      // row of lane 0 in the row space
  int nvalid;    // rows of the slab inside the group: 0..32
  int row_base;  // first row of the group
  int n0;        // first output column of the tile
};

// Hands a finished box to the TMA engine (lane 0) after all lanes wrote it.
template <bool kReduce>
__device__ __forceinline__ void epi_issue(const CUtensorMap* tm, unsigned char* box, int x, int y) {
  fence_proxy_async_smem();
  __syncwarp();
  if (lane_id() == 0) {
    if (kReduce)
      tma_reduce_add_2d(tm, box, x, y);
    else
      tma_store_2d(tm, box, x, y);
    bulk_commit();
  }
}

// The staging box `buf` may be rewritten once the copy issued from it two
// boxes ago has read it.
__device__ __forceinline__ unsigned char* epi_box(unsigned char* stage, int& buf) {
  unsigned char* box = stage + buf * EPI_BOX_BYTES;
  buf ^= 1;
  if (lane_id() == 0) bulk_wait_read<1>();
  __syncwarp();
  return box;
}

// Epilogue of one warp over NC accumulator columns at TMEM address `taddr`
// (lane quarter already applied); `bpre` is epi_bias_preload's value for the
// tile, `sc` the FP8 dequantisation scales (acc * row scale * column scale
// + bias) or off. `release()` is called by the whole warp once the last
// tcgen05.ld of the accumulator has completed.
template <int NC, class P, class Release>
__device__ __forceinline__ void epilogue_warp(const P& p, const CUtensorMap* tm_out, uint32_t taddr,
                                              const EpiSlab& s, const uint4& bpre, const EpiScale& sc,
                                              unsigned char* stage, int& buf, Release release) {
  static_assert(NC <= 256, "one bias uint4 per lane covers 256 columns");
  // parameters held in registers for the whole tile (the asm statements
  // below clobber memory, which would otherwise force them to be re-read)
  const int lane = lane_id();
  const bool full = s.nvalid == 32;
  const bool mine = lane < s.nvalid;
  const int N = p.N;
  const int epi = p.epilogue;
  void* const out = p.out;
  if (epi == EPI_BIAS_BF16 || epi == EPI_BIAS_GELU_F16) {
    const bool gelu = epi == EPI_BIAS_GELU_F16;
#pragma unroll 1
    for (int c = 0; c < NC / 64; ++c) {
      float v[64];
      tmem_ld32(taddr + c * 64, v);
      tmem_ld32(taddr + c * 64 + 32, v + 32);
      tmem_ld_wait();
      if (c == NC / 64 - 1) release();
      const int col0 = s.n0 + c * 64;
      if (col0 >= N || s.nvalid == 0) continue;
      uint4 o[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        float bv[8];
        epi_bias8(bpre, 8 * c + j, bv);
        float w[8];
        if (sc.on) {
          float sv[8];
          epi_scale8(sc, 8 * c + j, sv);
#pragma unroll
          for (int i = 0; i < 8; ++i) v[8 * j + i] *= sv[i];
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          w[i] = v[8 * j + i] + bv[i];
          if (gelu) w[i] = gelu_tanh(w[i]);
        }
        if (gelu) {
          o[j].x = pack_f16x2_sat(w[0], w[1]);
          o[j].y = pack_f16x2_sat(w[2], w[3]);
          o[j].z = pack_f16x2_sat(w[4], w[5]);
          o[j].w = pack_f16x2_sat(w[6], w[7]);
        } else {
          o[j].x = pack_bf16x2(w[0], w[1]);
          o[j].y = pack_bf16x2(w[2], w[3]);
          o[j].z = pack_bf16x2(w[4], w[5]);
          o[j].w = pack_bf16x2(w[6], w[7]);
        }
      }
      if (full) {
        unsigned char* box = epi_box(stage, buf);
#pragma unroll
        for (int j = 0; j < 8; ++j) *reinterpret_cast<uint4*>(box + sw128_off(lane, j)) = o[j];
        epi_issue<false>(tm_out, box, col0, s.row0);
      } else if (mine) {
        uint4* dst = reinterpret_cast<uint4*>(static_cast<uint16_t*>(out) +
                                              static_cast<long long>(s.row0 + lane) * N + col0);
#pragma unroll
        for (int j = 0; j < 8; ++j)
          if (col0 + 8 * j < N) dst[j] = o[j];
      }
    }
    return;
  }
  // fp32 outputs, 32 columns at a time
  const bool inplace = epi == EPI_BIAS_RESID_F32;
  const bool resid_f32 = p.resid_f32 != 0;
  const void* const resid = s.g ? p.resid_src[1] : p.resid_src[0];
  const long long rrow = static_cast<long long>(s.row0 + lane - s.row_base) * N;
  uint4 rn[8];  // residual of the next chunk (bf16: rn[0..3], fp32: rn[0..7])
  auto load_resid = [&](int col0) {
    if (resid_f32) {
      const uint4* src = reinterpret_cast<const uint4*>(static_cast<const float*>(resid) + rrow + col0);
#pragma unroll
      for (int j = 0; j < 8; ++j) rn[j] = __ldg(src + j);
    } else {
      const uint4* src =
          reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(resid) + rrow + col0);
#pragma unroll
      for (int j = 0; j < 4; ++j) rn[j] = __ldg(src + j);
    }
  };
  if (!inplace && mine && s.n0 < N) load_resid(s.n0);
#pragma unroll 1
  for (int c = 0; c < NC / 32; ++c) {
    float v[32];
    tmem_ld32(taddr + c * 32, v);
    tmem_ld_wait();
    if (c == NC / 32 - 1) release();
    const int col0 = s.n0 + c * 32;
    if (col0 >= N || s.nvalid == 0) continue;
    float bv[32];
#pragma unroll
    for (int j = 0; j < 4; ++j) epi_bias8(bpre, 4 * c + j, bv + 8 * j);
    if (sc.on) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        float sv[8];
        epi_scale8(sc, 4 * c + j, sv);
#pragma unroll
        for (int i = 0; i < 8; ++i) v[8 * j + i] *= sv[i];
      }
    }
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] += bv[i];
    if (!inplace) {
      float rv[32];
      if (resid_f32) {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          rv[4 * j] = __uint_as_float(rn[j].x);
          rv[4 * j + 1] = __uint_as_float(rn[j].y);
          rv[4 * j + 2] = __uint_as_float(rn[j].z);
          rv[4 * j + 3] = __uint_as_float(rn[j].w);
        }
      } else {
#pragma unroll
        for (int j = 0; j < 4; ++j) bf16x8(rn[j], rv + 8 * j);
      }
      if (mine && c + 1 < NC / 32 && col0 + 32 < N) load_resid(col0 + 32);
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = rv[i] + v[i];
    }
    if (full) {
      unsigned char* box = epi_box(stage, buf);
#pragma unroll
      for (int j = 0; j < 8; ++j)
        *reinterpret_cast<float4*>(box + sw128_off(lane, j)) =
            make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
      if (inplace)
        epi_issue<true>(tm_out, box, col0, s.row0);
      else
        epi_issue<false>(tm_out, box, col0, s.row0);
    } else if (mine) {
      float4* dst = reinterpret_cast<float4*>(static_cast<float*>(out) +
                                              static_cast<long long>(s.row0 + lane) * N + col0);
      if (inplace) {
        // atomic: pieces of a tile cut along K may add to the same rows
        float* d = reinterpret_cast<float*>(dst);
#pragma unroll
        for (int i = 0; i < 32; ++i) atomicAdd(d + i, v[i]);
      } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) dst[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
      }
    }
  }
}

// Waits until every bulk copy this warp issued has completed (before exit).
__device__ __forceinline__ void epilogue_drain() {
  if (lane_id() == 0) bulk_wait<0>();
  __syncwarp();
}

// The output tensor map of an epilogue: 32-row boxes of 128 bytes.
inline bool encode_epilogue_map(CUtensorMap* map, const GemmArgs& a) {
  if (a.epilogue == EPI_BIAS_RESID_F32 || a.epilogue == EPI_BIAS_RESIDIN_F32)
    return encode_tmap_2d(map, TMAP_F32, a.out, a.N, a.R, a.N, 32, 32);
  return encode_tmap_2d(map, a.epilogue == EPI_BIAS_GELU_F16 ? TMAP_F16 : TMAP_BF16, a.out, a.N, a.R, a.N,
                        64, 32);
}

}  // namespace hilo
