// Joint variable-length softmax attention of the MMDiT block on tcgen05.
//
// Image b attends over its joint sequence [T text rows ; L_b packed image
// rows] (non-causal, scale 1/sqrt(head_dim)); L_b comes from the device
// array cu_img, so the compressed sequence lengths never travel to the host.
// The text rows and the image rows of one image live in two separate ranges
// of the row space; queries and keys/values are tiled per range (128 rows per
// tile, the ragged last tile masked).
//
// One CTA per (image, head, 128-query tile), 192 threads:
//   warp 0     TMA: Q once, then K and V tiles (two-stage ring), 128-byte
//              swizzled boxes of 64 columns
//   warp 1     MMA: S = Q K^T into TMEM (two S buffers so S_{t+1} overlaps
//              the softmax of S_t), then O_t = P_t V_t into TMEM (V is the
//              MN-major operand, no transpose pass)
//   warps 2-5  softmax, one query row per thread: row max, exp2, bf16 P into
//              swizzled shared memory, running sum; the output accumulator
//              lives in registers and is rescaled there (online softmax)
// Every mbarrier wait is bounded (error latched, TMEM freed, CTA returns).
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace hilo {

__device__ int g_attn_err;

namespace {

constexpr int BQ = 128;
constexpr int BKV = 128;
constexpr int ATTN_THREADS = 192;
constexpr uint32_t ATTN_TMEM_COLS = 512;  // S0 | S1 | O
constexpr int BOX_BYTES = 128 * 128;       // 128 rows x 64 bf16

template <int HD>
struct Cfg {
  static constexpr int NBOX = HD / 64;
  static constexpr int TILE_BYTES = NBOX * BOX_BYTES;  // 128 rows x HD
  static constexpr int P_BYTES = 2 * BOX_BYTES;        // 128 x 128 bf16
  // Q | K0 | V0 | K1 | V1 | P
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K0 = TILE_BYTES;
  static constexpr int OFF_P = 5 * TILE_BYTES;
  static constexpr int DATA_BYTES = 5 * TILE_BYTES + P_BYTES;
  static constexpr int SMEM_BYTES = DATA_BYTES + 1024 + 256;
};

struct AttnParams {
  const int32_t* cu_img;
  __nv_bfloat16* out;
  int B, T, heads, d, qt_txt, qt_img_max;
  float scale_log2;  // log2(e) / sqrt(head_dim)
};

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Row range of KV tile t of image b: text tiles first, then image tiles.
__device__ __forceinline__ void kv_tile(const AttnParams& p, int b, int L, int t, int& row0,
                                        int& valid) {
  if (t < p.qt_txt) {
    row0 = b * p.T + t * BKV;
    valid = min(BKV, p.T - t * BKV);
  } else {
    const int j = t - p.qt_txt;
    row0 = p.B * p.T + p.cu_img[b] + j * BKV;
    valid = min(BKV, L - j * BKV);
  }
}

template <int HD>
__global__ void __launch_bounds__(ATTN_THREADS, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tm, const AttnParams p) {
  using C = Cfg<HD>;
  // ---- work item
  const int per = p.qt_txt + p.qt_img_max;
  const int item = blockIdx.x;
  const int b = item / (p.heads * per);
  const int h = (item / per) % p.heads;
  const int qt = item % per;
  const int L = p.cu_img[b + 1] - p.cu_img[b];
  const int nkv_img = (L + BKV - 1) / BKV;
  int q_row0, q_valid;
  if (qt < p.qt_txt) {
    q_row0 = b * p.T + qt * BQ;
    q_valid = min(BQ, p.T - qt * BQ);
  } else {
    const int j = qt - p.qt_txt;
    if (j >= nkv_img) return;  // beyond this image's compressed length
    q_row0 = p.B * p.T + p.cu_img[b] + j * BQ;
    q_valid = min(BQ, L - j * BQ);
  }
  const int nkv = p.qt_txt + nkv_img;

  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  unsigned char* sQ = smem + C::OFF_Q;
  unsigned char* sP = smem + C::OFF_P;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::DATA_BYTES);
  uint64_t* q_full = bars + 0;
  uint64_t* kv_full = bars + 1;   // [2]
  uint64_t* kv_empty = bars + 3;  // [2]
  uint64_t* s_full = bars + 5;    // [2]
  uint64_t* p_full = bars + 7;
  uint64_t* o_full = bars + 8;
  uint64_t* drain = bars + 9;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 10);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* err = &g_attn_err;
  auto sK = [&](int st) { return smem + C::OFF_K0 + st * 2 * C::TILE_BYTES; };
  auto sV = [&](int st) { return smem + C::OFF_K0 + st * 2 * C::TILE_BYTES + C::TILE_BYTES; };

  const int warp = warp_id(), lane = lane_id();
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&kv_full[i], 1);
      mbar_init(&kv_empty[i], 1);
      mbar_init(&s_full[i], 1);
    }
    mbar_init(p_full, 128);
    mbar_init(o_full, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, ATTN_TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tS[2] = {tmem, tmem + 128u};
  const uint32_t tO = tmem + 256u;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer
      tma_prefetch_desc(&tm);
      int armed[2] = {-1, -1};
      mbar_arrive_expect_tx(q_full, C::TILE_BYTES);
#pragma unroll
      for (int j = 0; j < C::NBOX; ++j)
        tma_load_2d(sQ + j * BOX_BYTES, &tm, q_full, h * HD + 64 * j, q_row0);
      bool ok = true;
      for (int t = 0; t < nkv; ++t) {
        const int st = t & 1;
        const uint32_t ph = static_cast<uint32_t>((t >> 1) & 1);
        if (!mbar_wait(&kv_empty[st], ph ^ 1u, abort_flag, err, DEV_TIMEOUT_ATTN)) {
          ok = false;
          break;
        }
        int row0, valid;
        kv_tile(p, b, L, t, row0, valid);
        mbar_arrive_expect_tx(&kv_full[st], 2 * C::TILE_BYTES);
#pragma unroll
        for (int j = 0; j < C::NBOX; ++j) {
          tma_load_2d(sK(st) + j * BOX_BYTES, &tm, &kv_full[st], p.d + h * HD + 64 * j, row0);
          tma_load_2d(sV(st) + j * BOX_BYTES, &tm, &kv_full[st], 2 * p.d + h * HD + 64 * j, row0);
        }
        armed[st] = static_cast<int>(ph);
      }
      if (!ok) {
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(smem_u32(q_full), 0u) && globaltimer_ns() - t0 < HILO_WAIT_LIMIT_NS / 4) {
        }
        for (int st = 0; st < 2; ++st) {
          if (armed[st] < 0) continue;
          const uint64_t t1 = globaltimer_ns();
          while (!mbar_try_wait(smem_u32(&kv_full[st]), static_cast<uint32_t>(armed[st])) &&
                 globaltimer_ns() - t1 < HILO_WAIT_LIMIT_NS / 4) {
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer
      const uint32_t idesc_s = idesc_bf16(BQ, BKV, 0, 0);
      const uint32_t idesc_o = idesc_bf16(BQ, HD, 0, 1);
      const uint32_t q_base = smem_u32(sQ);
      const uint32_t p_base = smem_u32(sP);
      auto issue_s = [&](int t) {
        const uint32_t k_base = smem_u32(sK(t & 1));
#pragma unroll
        for (int k = 0; k < HD / 16; ++k) {
          const uint32_t off = (k >> 2) * BOX_BYTES + (k & 3) * 32;
          umma_bf16(tS[t & 1], sw128_desc(q_base + off, 16, 1024), sw128_desc(k_base + off, 16, 1024),
                    idesc_s, k > 0 ? 1u : 0u);
        }
        umma_commit(&s_full[t & 1]);
      };
      bool ok = mbar_wait(q_full, 0u, abort_flag, err, DEV_TIMEOUT_ATTN) &&
                mbar_wait(&kv_full[0], 0u, abort_flag, err, DEV_TIMEOUT_ATTN);
      if (ok) {
        tc_fence_after();
        issue_s(0);
      }
      for (int t = 0; t < nkv && ok; ++t) {
        if (t + 1 < nkv) {
          if (!mbar_wait(&kv_full[(t + 1) & 1], static_cast<uint32_t>(((t + 1) >> 1) & 1), abort_flag,
                         err, DEV_TIMEOUT_ATTN))
            break;
          tc_fence_after();
          issue_s(t + 1);
        }
        if (!mbar_wait(p_full, static_cast<uint32_t>(t & 1), abort_flag, err, DEV_TIMEOUT_ATTN)) break;
        tc_fence_after();
        const uint32_t v_base = smem_u32(sV(t & 1));
#pragma unroll
        for (int k = 0; k < BKV / 16; ++k) {
          const uint64_t ad = sw128_desc(p_base + (k >> 2) * BOX_BYTES + (k & 3) * 32, 16, 1024);
          const uint64_t bd = sw128_desc(v_base + k * 2048, BOX_BYTES, 1024);
          umma_bf16(tO, ad, bd, idesc_o, k > 0 ? 1u : 0u);
        }
        umma_commit(o_full);
        umma_commit(&kv_empty[t & 1]);
      }
      umma_commit(drain);
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(smem_u32(drain), 0u)) {
        if (globaltimer_ns() - t0 > HILO_WAIT_LIMIT_NS) {
          atomicExch(err, DEV_TIMEOUT_ATTN);
          break;
        }
      }
    }
  } else {
    // ---------------- softmax (warps 2..5 -> TMEM lane quarters 2,3,0,1)
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    float acc[HD];
#pragma unroll
    for (int i = 0; i < HD; ++i) acc[i] = 0.f;
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int t = 0; t < nkv; ++t) {
      int row0, valid;
      kv_tile(p, b, L, t, row0, valid);
      if (!mbar_wait(&s_full[t & 1], static_cast<uint32_t>((t >> 1) & 1), abort_flag, err,
                     DEV_TIMEOUT_ATTN)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t sb = tS[t & 1] + lane_off;
      float mx = -INFINITY;
#pragma unroll 1
      for (int c = 0; c < BKV / 32; ++c) {
        float v[32];
        tmem_ld32(sb + c * 32, v);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (c * 32 + i < valid) mx = fmaxf(mx, v[i]);
      }
      const float m_new = fmaxf(m, mx * p.scale_log2);
      const float alpha = ex2(m - m_new);
      // rows of a ragged last tile hold other tokens' (or stale) values:
      // zero them in V so that 0-probability columns contribute exactly 0
      if (valid < BKV) {
        if (!mbar_wait(&kv_full[t & 1], static_cast<uint32_t>((t >> 1) & 1), abort_flag, err,
                       DEV_TIMEOUT_ATTN)) {
          ok = false;
          break;
        }
        if (row >= valid) {
          unsigned char* vr = sV(t & 1) + row * 128;
#pragma unroll
          for (int j = 0; j < C::NBOX; ++j)
#pragma unroll
            for (int c16 = 0; c16 < 8; ++c16)
              *reinterpret_cast<uint4*>(vr + j * BOX_BYTES + c16 * 16) = make_uint4(0, 0, 0, 0);
        }
      }
      float lsum = 0.f;
      unsigned char* prow = sP + row * 128;
#pragma unroll 1
      for (int c = 0; c < BKV / 32; ++c) {
        float v[32];
        tmem_ld32(sb + c * 32, v);
        tmem_ld_wait();
        float pv[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          pv[i] = (c * 32 + i < valid) ? ex2(v[i] * p.scale_log2 - m_new) : 0.f;
          lsum += pv[i];
        }
        unsigned char* pbox = prow + (c >> 1) * BOX_BYTES;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int chunk = (c & 1) * 4 + j;
          uint4 o;
          o.x = pack_bf16x2(pv[8 * j], pv[8 * j + 1]);
          o.y = pack_bf16x2(pv[8 * j + 2], pv[8 * j + 3]);
          o.z = pack_bf16x2(pv[8 * j + 4], pv[8 * j + 5]);
          o.w = pack_bf16x2(pv[8 * j + 6], pv[8 * j + 7]);
          *reinterpret_cast<uint4*>(pbox + ((chunk ^ (row & 7)) << 4)) = o;
        }
      }
      l = l * alpha + lsum;
      m = m_new;
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(p_full);
      if (!mbar_wait(o_full, static_cast<uint32_t>(t & 1), abort_flag, err, DEV_TIMEOUT_ATTN)) {
        ok = false;
        break;
      }
      tc_fence_after();
#pragma unroll
      for (int c = 0; c < HD / 32; ++c) {
        float v[32];
        tmem_ld32(tO + lane_off + c * 32, v);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; ++i) acc[c * 32 + i] = acc[c * 32 + i] * alpha + v[i];
      }
    }
    if (ok && row < q_valid) {
      const float inv = 1.0f / l;
      uint4* dst = reinterpret_cast<uint4*>(p.out + static_cast<long long>(q_row0 + row) * p.d + h * HD);
#pragma unroll
      for (int j = 0; j < HD / 8; ++j) {
        uint4 o;
        o.x = pack_bf16x2(acc[8 * j] * inv, acc[8 * j + 1] * inv);
        o.y = pack_bf16x2(acc[8 * j + 2] * inv, acc[8 * j + 3] * inv);
        o.z = pack_bf16x2(acc[8 * j + 4] * inv, acc[8 * j + 5] * inv);
        o.w = pack_bf16x2(acc[8 * j + 6] * inv, acc[8 * j + 7] * inv);
        dst[j] = o;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, ATTN_TMEM_COLS);
  }
}

template <int HD>
cudaError_t launch_hd(const AttnArgs& a, const AttnParams& p, int grid, cudaStream_t st) {
  CUtensorMap tm;
  if (!encode_tmap_bf16_2d(&tm, a.qkv, 3ull * a.d, a.R, 3ull * a.d, 64, 128))
    return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(attn_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Cfg<HD>::SMEM_BYTES);
  if (e != cudaSuccess) return e;
  attn_kernel<HD><<<grid, ATTN_THREADS, Cfg<HD>::SMEM_BYTES, st>>>(tm, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_attention(const AttnArgs& a, int num_sms, cudaStream_t st) {
  (void)num_sms;
  AttnParams p;
  p.cu_img = a.cu_img;
  p.out = static_cast<__nv_bfloat16*>(a.out);
  p.B = a.B;
  p.T = a.T;
  p.heads = a.heads;
  p.d = a.d;
  p.qt_txt = (a.T + BQ - 1) / BQ;
  p.qt_img_max = (a.max_img_rows + BQ - 1) / BQ;
  p.scale_log2 = static_cast<float>(1.4426950408889634 / sqrt(static_cast<double>(a.head_dim)));
  const long long items = static_cast<long long>(a.B) * a.heads * (p.qt_txt + p.qt_img_max);
  if (items <= 0) return cudaSuccess;
  if (items > 0x7fffffffLL) return cudaErrorInvalidValue;
  if (a.head_dim == 128) return launch_hd<128>(a, p, static_cast<int>(items), st);
  if (a.head_dim == 64) return launch_hd<64>(a, p, static_cast<int>(items), st);
  return cudaErrorInvalidValue;
}

int attn_take_device_error() {
  int v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_attn_err, sizeof(int)) != cudaSuccess) return -1;
  if (v) cudaMemcpyToSymbol(g_attn_err, &z, sizeof(int));
  return v;
}

}  // namespace hilo
