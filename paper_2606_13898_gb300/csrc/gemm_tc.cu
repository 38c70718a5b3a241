// Grouped bf16 GEMM on the 5th-generation tensor cores (tcgen05) for the
// MMDiT block's linear layers: C[r, n] = sum_k A[r, k] * W_g[n, k] + b_g[n]
// with the text rows (group 0) and the packed image rows (group 1) of the
// row space using their own weights. The image row count is read on the
// device, so no host synchronisation is needed between split and block.
//
// Design (one persistent CTA per SM, 192 threads):
//   warp 0     TMA producer: 128x64 A and 256x64 W tiles, 128-byte swizzle,
//              into a 4-stage shared-memory ring (48 KB per stage)
//   warp 1     MMA issuer: tcgen05.mma M=128 N=256 K=16, fp32 accumulator in
//              TMEM, two accumulators (2 x 256 columns) so the epilogue of one
//              tile overlaps the main loop of the next
//   warps 2-5  epilogue: tcgen05.ld 32 columns at a time, bias / GELU /
//              residual add, vector stores
// Every mbarrier wait is bounded; on a timeout the CTA latches an error code
// (read by hilo_sync_status), stops, frees its TMEM and returns.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "common.cuh"
#include "internal.h"

namespace hilo {

__device__ int g_gemm_err;

namespace {

constexpr int BM = 128, BK = 64;
constexpr int GEMM_THREADS = 192;

// Tile configuration by tile width: 128x256 tiles with a 4-stage ring, or
// 128x128 tiles with a 6-stage ring (for narrow outputs, N <= 1024).
template <int BN>
struct TileCfg {
  static constexpr int STAGES = BN == 256 ? 4 : 6;
  static constexpr int A_STAGE_BYTES = BM * BK * 2;
  static constexpr int B_STAGE_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_STAGE_BYTES + B_STAGE_BYTES;
  static constexpr uint32_t TMEM_COLS = 2 * BN;  // two accumulators
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 + 256;
};

struct GemmParams {
  int N, K;
  uint32_t idesc;
  int row_base[2];
  int rows_static[2];
  const int32_t* rows_dev[2];
  const __nv_bfloat16* bias[2];
  int epilogue;
  void* out;
  const void* resid_src[2];
  int resid_f32;
};

struct Tile {
  int g, m0, n0, rows, row_base;
};

template <int BN>
struct Sched {
  int mt[2], rows[2], nt, total;
  __device__ void init(const GemmParams& p) {
    nt = (p.N + BN - 1) / BN;
    total = 0;
#pragma unroll
    for (int g = 0; g < 2; ++g) {
      rows[g] = p.rows_dev[g] ? *p.rows_dev[g] : p.rows_static[g];
      mt[g] = (rows[g] + BM - 1) / BM;
      total += mt[g] * nt;
    }
  }
  __device__ Tile get(const GemmParams& p, int t) const {
    Tile r;
    r.g = t < mt[0] * nt ? 0 : 1;
    if (r.g) t -= mt[0] * nt;
    const int mtg = mt[r.g];
    r.m0 = p.row_base[r.g] + (t % mtg) * BM;
    r.n0 = (t / mtg) * BN;
    r.rows = rows[r.g];
    r.row_base = p.row_base[r.g];
    return r;
  }
};

__device__ __forceinline__ float gelu_tanh(float z) {
  const float k0 = 0.7978845608028654f;  // sqrt(2/pi)
  return 0.5f * z * (1.0f + tanhf(k0 * (z + 0.044715f * z * z * z)));
}

__device__ __forceinline__ void bf16x8(const uint4& v, float* f) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

template <int BN>
__global__ void __launch_bounds__(GEMM_THREADS, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB0,
                const __grid_constant__ CUtensorMap tmB1, const GemmParams p) {
  using Cfg = TileCfg<BN>;
  constexpr int STAGES = Cfg::STAGES;
  constexpr int STAGE_BYTES = Cfg::STAGE_BYTES;
  constexpr int A_STAGE_BYTES = Cfg::A_STAGE_BYTES;
  constexpr uint32_t TMEM_COLS = Cfg::TMEM_COLS;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* err = &g_gemm_err;

  pdl_trigger();
  const int warp = warp_id(), lane = lane_id();
  Sched<BN> sc;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 4);  // one arrive per epilogue warp
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB0);
    tma_prefetch_desc(&tmB1);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int kblocks = p.K / BK;
  pdl_wait();  // the row counts and A are written by the previous kernel
  sc.init(p);

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer
      int stage = 0;
      uint32_t phase = 0;
      int armed[STAGES];  // parity of the last phase armed on full[s], or -1
      for (int s = 0; s < STAGES; ++s) armed[s] = -1;
      bool ok = true;
      for (int t = blockIdx.x; t < sc.total && ok; t += gridDim.x) {
        const Tile tl = sc.get(p, t);
        const CUtensorMap* tb = tl.g ? &tmB1 : &tmB0;
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, err, DEV_TIMEOUT_GEMM)) {
            ok = false;
            break;
          }
          unsigned char* sa = smem + stage * STAGE_BYTES;
          mbar_arrive_expect_tx(&full[stage], STAGE_BYTES);
          tma_load_2d(sa, &tmA, &full[stage], kb * BK, tl.m0);
          tma_load_2d(sa + A_STAGE_BYTES, tb, &full[stage], kb * BK, tl.n0);
          armed[stage] = static_cast<int>(phase);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        // wait (bounded) for the bulk copies already in flight, so that none
        // lands in shared memory after this CTA has exited
        for (int s = 0; s < STAGES; ++s) {
          if (armed[s] < 0) continue;
          const uint64_t t0 = globaltimer_ns();
          while (!mbar_try_wait(smem_u32(&full[s]), static_cast<uint32_t>(armed[s]))) {
            if (globaltimer_ns() - t0 > HILO_WAIT_LIMIT_NS / 4) break;
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer
      const uint32_t idesc = p.idesc;
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < sc.total && ok; t += gridDim.x) {
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, err, DEV_TIMEOUT_GEMM)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem + static_cast<uint32_t>(acc * BN);
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_flag, err, DEV_TIMEOUT_GEMM)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_base = smem_u32(smem + stage * STAGE_BYTES);
          const uint32_t b_base = a_base + A_STAGE_BYTES;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            const uint64_t ad = sw128_desc(a_base + k * 32, 16, 1024);
            const uint64_t bd = sw128_desc(b_base + k * 32, 16, 1024);
            umma_bf16(d_tmem, ad, bd, idesc, (kb | k) != 0 ? 1u : 0u);
          }
          umma_commit(&empty[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit(&tfull[acc]);
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
      }
      // every MMA this thread issued has completed before TMEM is freed
      umma_commit(drain);
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(smem_u32(drain), 0u)) {
        if (globaltimer_ns() - t0 > HILO_WAIT_LIMIT_NS) {
          atomicExch(err, DEV_TIMEOUT_GEMM);
          break;
        }
      }
    }
  } else {
    // ---------------- epilogue (warps 2..5 -> TMEM lane quarters 2,3,0,1)
    const int q = warp & 3;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int t = blockIdx.x; t < sc.total; t += gridDim.x) {
      const Tile tl = sc.get(p, t);
      if (!mbar_wait_warp(&tfull[acc], acc_phase, abort_flag, err, DEV_TIMEOUT_GEMM)) break;
      tc_fence_after();
      const int rit = q * 32 + lane;
      const int grow = tl.m0 + rit;
      const bool valid = (tl.m0 - tl.row_base) + rit < tl.rows;
      const uint32_t taddr = tmem + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * BN);
      const __nv_bfloat16* bias = p.bias[tl.g];
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        float v[32];
        tmem_ld32(taddr + c * 32, v);
        tmem_ld_wait();
        if (c == BN / 32 - 1) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&tempty[acc]);
        }
        const int col0 = tl.n0 + c * 32;
        if (!valid || col0 >= p.N) continue;
        float bv[32];
#pragma unroll
        for (int j = 0; j < 4; ++j) bf16x8(__ldg(reinterpret_cast<const uint4*>(bias + col0) + j), bv + 8 * j);
        if (p.epilogue == EPI_BIAS_RESID_F32 || p.epilogue == EPI_BIAS_RESIDIN_F32) {
          float4* dst = reinterpret_cast<float4*>(static_cast<float*>(p.out) +
                                                  static_cast<long long>(grow) * p.N + col0);
          float rv[32];
          if (p.epilogue == EPI_BIAS_RESID_F32) {
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float4 r = dst[j];
              rv[4 * j] = r.x;
              rv[4 * j + 1] = r.y;
              rv[4 * j + 2] = r.z;
              rv[4 * j + 3] = r.w;
            }
          } else {
            const long long off = static_cast<long long>(grow - tl.row_base) * p.N + col0;
            if (p.resid_f32) {
              const float4* src = reinterpret_cast<const float4*>(static_cast<const float*>(p.resid_src[tl.g]) + off);
#pragma unroll
              for (int j = 0; j < 8; ++j) {
                const float4 r = __ldg(src + j);
                rv[4 * j] = r.x;
                rv[4 * j + 1] = r.y;
                rv[4 * j + 2] = r.z;
                rv[4 * j + 3] = r.w;
              }
            } else {
              const uint4* src =
                  reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(p.resid_src[tl.g]) + off);
#pragma unroll
              for (int j = 0; j < 4; ++j) bf16x8(__ldg(src + j), rv + 8 * j);
            }
          }
#pragma unroll
          for (int j = 0; j < 8; ++j)
            dst[j] = make_float4(rv[4 * j] + (v[4 * j] + bv[4 * j]), rv[4 * j + 1] + (v[4 * j + 1] + bv[4 * j + 1]),
                                 rv[4 * j + 2] + (v[4 * j + 2] + bv[4 * j + 2]),
                                 rv[4 * j + 3] + (v[4 * j + 3] + bv[4 * j + 3]));
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] += bv[i];
          uint4* dst = reinterpret_cast<uint4*>(static_cast<uint16_t*>(p.out) +
                                                static_cast<long long>(grow) * p.N + col0);
          if (p.epilogue == EPI_BIAS_GELU_F16) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = gelu_tanh(v[i]);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              uint4 o;
              o.x = pack_f16x2_sat(v[8 * j], v[8 * j + 1]);
              o.y = pack_f16x2_sat(v[8 * j + 2], v[8 * j + 3]);
              o.z = pack_f16x2_sat(v[8 * j + 4], v[8 * j + 5]);
              o.w = pack_f16x2_sat(v[8 * j + 6], v[8 * j + 7]);
              dst[j] = o;
            }
          } else {
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              uint4 o;
              o.x = pack_bf16x2(v[8 * j], v[8 * j + 1]);
              o.y = pack_bf16x2(v[8 * j + 2], v[8 * j + 3]);
              o.z = pack_bf16x2(v[8 * j + 4], v[8 * j + 5]);
              o.w = pack_bf16x2(v[8 * j + 6], v[8 * j + 7]);
              dst[j] = o;
            }
          }
        }
      }
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

template <int BN>
cudaError_t launch_bn(const GemmArgs& a, int num_sms, cudaStream_t st) {
  using Cfg = TileCfg<BN>;
  CUtensorMap tA, tB0, tB1;
  if (!encode_tmap_bf16_2d(&tA, a.A, a.K, a.R, a.K, BK, BM)) return cudaErrorInvalidValue;
  if (!encode_tmap_bf16_2d(&tB0, a.g[0].weight ? a.g[0].weight : a.g[1].weight, a.K, a.N, a.K,
                           BK, BN))
    return cudaErrorInvalidValue;
  if (!encode_tmap_bf16_2d(&tB1, a.g[1].weight ? a.g[1].weight : a.g[0].weight, a.K, a.N, a.K,
                           BK, BN))
    return cudaErrorInvalidValue;
  GemmParams p;
  p.N = a.N;
  p.K = a.K;
  p.idesc = idesc_kind_f16(BM, BN, 0, 0, a.op_f16 ? 0 : 1);
  long long upper = 0;
  for (int g = 0; g < 2; ++g) {
    p.row_base[g] = a.g[g].row_base;
    p.rows_static[g] = a.g[g].rows_static;
    p.rows_dev[g] = a.g[g].rows_dev;
    p.bias[g] = static_cast<const __nv_bfloat16*>(a.g[g].bias);
    upper += (a.g[g].rows_cap + BM - 1) / BM;
  }
  upper *= (a.N + BN - 1) / BN;
  p.epilogue = a.epilogue;
  p.out = a.out;
  p.resid_src[0] = a.resid_src[0];
  p.resid_src[1] = a.resid_src[1];
  p.resid_f32 = a.resid_f32;
  if (upper <= 0) return cudaSuccess;
  const int grid = static_cast<int>(upper < num_sms ? upper : num_sms);
  cudaError_t e = cudaFuncSetAttribute(gemm_kernel<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Cfg::SMEM_BYTES);
  if (e != cudaSuccess) return e;
  return launch_pdl(gemm_kernel<BN>, dim3(grid), dim3(GEMM_THREADS), Cfg::SMEM_BYTES, st, tA, tB0, tB1,
                    p);
}

}  // namespace

cudaError_t launch_gemm(const GemmArgs& a, int num_sms, cudaStream_t st) {
  if (a.K % BK != 0 || a.N % 32 != 0) return cudaErrorInvalidValue;
  // CTA pairs with 256x256 tiles where N allows (half the W traffic per SM);
  // else one CTA per tile: 256-wide tiles, or 128-wide where N is so small
  // that 256 would leave SMs idle.
  if (a.N >= 1024 && gemm_pair_supported(a)) return launch_gemm_pair(a, num_sms, st);
  if (a.N <= 1024) return launch_bn<128>(a, num_sms, st);
  return launch_bn<256>(a, num_sms, st);
}

int gemm_take_device_error() {
  int v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_gemm_err, sizeof(int)) != cudaSuccess) return -1;
  if (v) cudaMemcpyToSymbol(g_gemm_err, &z, sizeof(int));
  return v;
}

}  // namespace hilo
