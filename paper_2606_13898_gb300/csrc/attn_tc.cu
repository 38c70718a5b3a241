// Joint variable-length softmax attention of the MMDiT block on tcgen05
// (paper Sec. 2.1: the DiT of the editing generalist; Sec. 2.3: the
// compressed image tokens attend jointly with the text tokens).
//
// Image b attends over its joint sequence [T text rows ; L_b packed image
// rows] (non-causal, scale 1/sqrt(head_dim)); L_b comes from the device
// array cu_img, so the compressed sequence lengths never travel to the host.
// The text rows and the image rows of one image live in two separate ranges
// of the row space; queries and keys/values are tiled per range (128 rows per
// tile, the ragged last tile masked).
//
// One CTA per (image, head, pair of 128-query tiles), 384 threads in three
// warpgroups:
//   warps 0-3    softmax of query tile 0 (one query row per thread)
//   warps 4-7    softmax of query tile 1
//   warp 8       TMA: Q tiles once, then K and V tiles (two stages each),
//                128-byte swizzled boxes of 64 columns
//   warp 9       MMA: S_i = Q_i K^T into TMEM, O_i += P_i V into TMEM
//   warps 10-11  idle (the third warpgroup gives its registers away)
// Tensor memory holds S_0 | S_1 | O_0 | O_1 (128 columns each). A softmax
// warpgroup reads S_i once into registers and writes the probabilities P_i
// back over the first 64 columns of S_i as packed bf16; the PV product takes
// P_i from tensor memory (A operand) and V from shared memory (MN-major, no
// transpose pass). The two query tiles ping-pong on the tensor core (MMA
// order PV_0(t), S_0(t+1), PV_1(t), S_1(t+1)); S_i(t+1) overwrites P_i(t)
// only after PV_i(t), in issue order. When a softmax warpgroup sees S_i(t),
// every earlier MMA has completed, so O_i may be rescaled and P_i written
// without a further wait. The output accumulators are rescaled only when a
// row's running maximum grows by more than 2^8 (until then the
// probabilities are formed against the older, smaller maximum, so they stay
// <= 256, well inside bf16 range).
// With proportional attention (PROP) every key j carries a weight n_j (the
// number of grid tokens a packed image row stands for; text keys weigh 1):
// softmax(s + ln n) = n e^s / sum(n e^s), so each probability is multiplied
// by its key's weight before the row sum and the bf16 packing, and the row
// maxima (the stabiliser) stay those of the raw logits. Each softmax warp
// fetches the next key tile's 128 weights with asynchronous 4-byte copies
// (zero-filled past the ragged end) into its own double-buffered shared slot
// while it works on the current tile, and reads them back as 16-byte
// broadcasts; no barrier spans warps.
// Every mbarrier wait is bounded (error latched, TMEM freed, CTA returns).
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace hilo {

__device__ int g_attn_err;
// Set when an image has more packed rows than the launch's query tiles cover
// (cu_img describes more than hilo_shape allows per image); those rows'
// attention output would be left unwritten, so the call is reported failed.
__device__ int g_attn_rows_err;

namespace {

constexpr int BQ = 128;
constexpr int BKV = 128;
// Three warpgroups: two softmax warpgroups and one for TMA, MMA and two idle
// warps. The control warpgroup gives registers to the softmax warpgroups
// (setmaxnreg); launch_hd checks that the shares fit the launch allocation.
constexpr int ATTN_THREADS = 384;
constexpr int PRODUCER_WARP = 8;
constexpr int MMA_WARP = 9;
constexpr uint32_t SOFTMAX_REGS = 216;
constexpr uint32_t CONTROL_REGS = 72;
constexpr uint32_t ATTN_TMEM_COLS = 512;  // S0 | S1 | O0 | O1
constexpr int BOX_BYTES = 128 * 128;       // 128 rows x 64 16-bit elements
constexpr float RESCALE_LOG2 = 8.0f;

template <int HD, bool PROP>
struct Cfg {
  static constexpr int NBOX = HD / 64;
  static constexpr int TILE_BYTES = NBOX * BOX_BYTES;  // 128 rows x HD
  // Q0 | Q1 | K0 | K1 | V0 | V1
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = 2 * TILE_BYTES;
  static constexpr int OFF_V = 4 * TILE_BYTES;
  static constexpr int DATA_BYTES = 6 * TILE_BYTES;
  // barriers (256 B) and, with PROP, 8 softmax warps x 2 slots x 128 weights
  static constexpr int OFF_W = DATA_BYTES + 256;
  static constexpr int SMEM_BYTES = DATA_BYTES + 1024 + 256 + (PROP ? 8 * 2 * BKV * 4 : 0);
};

struct AttnParams {
  const int32_t* cu_img;
  const float* n_img;  // PROP: weight of each packed image row
  __nv_bfloat16* out;
  int B, T, heads, d, qt_txt, pairs_max;
  int cap;           // image-row capacity: row offsets are clamped to it
  float scale_log2;  // log2(e) / sqrt(head_dim)
};

// 4-byte asynchronous global -> shared copy; bytes past src_bytes (0 or 4)
// are zero-filled
__device__ __forceinline__ void cp_async4(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Pairs of fp32 values in one 64-bit register pair: Blackwell's paired fp32
// instructions (fma/mul/add .f32x2) apply the same IEEE operation to both
// halves at one issue slot per pair.
__device__ __forceinline__ uint64_t f2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f2_split(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}
__device__ __forceinline__ uint64_t f2_mul(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// The largest of three floats in one instruction (three-input max.f32). A
// maximum is exact, so grouping the row's values by threes gives the same
// result as any other order.
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float y;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(y) : "f"(a), "f"(b), "f"(c));
  return y;
}

// Row range of tile j of image b (text tiles first, then image tiles); used
// for both query and key/value tiles.
__device__ __forceinline__ void seq_tile(const AttnParams& p, int b, int L, int j, int& row0,
                                         int& valid) {
  if (j < p.qt_txt) {
    row0 = b * p.T + j * BKV;
    valid = min(BKV, p.T - j * BKV);
  } else {
    const int k = j - p.qt_txt;
    row0 = p.B * p.T + min(p.cu_img[b], p.cap) + k * BKV;
    valid = min(BKV, L - k * BKV);
  }
}

template <int HD, bool PROP>
__global__ void __launch_bounds__(ATTN_THREADS, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tm, const __grid_constant__ AttnParams p) {
  using C = Cfg<HD, PROP>;
  pdl_trigger();
  pdl_wait();  // cu_img and q/k/v are written by the previous kernels
  // ---- work item: (image, head, query-tile pair)
  const int item = blockIdx.x;
  const int b = item / (p.heads * p.pairs_max);
  const int h = (item / p.pairs_max) % p.heads;
  const int pair = item % p.pairs_max;
  // image rows [cu_img[b], cu_img[b+1]) within the capacity
  const int L = min(p.cu_img[b + 1], p.cap) - min(p.cu_img[b], p.cap);
  const int nkv = p.qt_txt + (L + BKV - 1) / BKV;  // also the number of query tiles
  if (pair == 0 && h == 0 && threadIdx.x == 0 && nkv > 2 * p.pairs_max) atomicExch(&g_attn_rows_err, b + 1);
  if (2 * pair >= nkv) return;                     // beyond this image's compressed length
  const bool has1 = 2 * pair + 1 < nkv;
  // the two query tiles (scalars: a runtime-indexed array would live in
  // local memory)
  int q_row0_0, q_valid_0, q_row0_1, q_valid_1;
  seq_tile(p, b, L, 2 * pair, q_row0_0, q_valid_0);
  q_row0_1 = q_row0_0;
  q_valid_1 = 0;
  if (has1) seq_tile(p, b, L, 2 * pair + 1, q_row0_1, q_valid_1);

  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::DATA_BYTES);
  uint64_t* q_full = bars + 0;
  uint64_t* k_full = bars + 1;    // [2]
  uint64_t* k_empty = bars + 3;   // [2]
  uint64_t* v_full = bars + 5;    // [2]
  uint64_t* v_empty = bars + 7;   // [2]
  uint64_t* s_full = bars + 9;    // [2] per query tile
  uint64_t* p_full = bars + 11;   // [2] per query tile
  uint64_t* o_done = bars + 13;   // [2] per query tile
  uint64_t* drain = bars + 15;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 16);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* err = &g_attn_err;
  auto sQ = [&](int i) { return smem + C::OFF_Q + i * C::TILE_BYTES; };
  auto sK = [&](int st) { return smem + C::OFF_K + st * C::TILE_BYTES; };
  auto sV = [&](int st) { return smem + C::OFF_V + st * C::TILE_BYTES; };

  const int warp = warp_id(), lane = lane_id();
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&k_full[i], 1);
      mbar_init(&k_empty[i], 1);
      mbar_init(&v_full[i], 1);
      mbar_init(&v_empty[i], 1);
      mbar_init(&s_full[i], 1);
      mbar_init(&p_full[i], 128);
      mbar_init(&o_done[i], 1);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == MMA_WARP) {
    tmem_alloc(tmem_slot, ATTN_TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  if (warp >= 8) {
    // control warpgroup: TMA producer, MMA issuer, two idle warps
    setmaxnreg_dec<CONTROL_REGS>();
    if (warp == PRODUCER_WARP) {
    if (lane == 0) {
      // ---------------- TMA producer
      tma_prefetch_desc(&tm);
      // per stage (bit st): armed at least once, and the parity of the last arming
      uint32_t armed_k = 0, par_k = 0, armed_v = 0, par_v = 0;
      mbar_arrive_expect_tx(q_full, (has1 ? 2 : 1) * C::TILE_BYTES);
#pragma unroll
      for (int j = 0; j < C::NBOX; ++j) {
        tma_load_2d(sQ(0) + j * BOX_BYTES, &tm, q_full, h * HD + 64 * j, q_row0_0);
        if (has1) tma_load_2d(sQ(1) + j * BOX_BYTES, &tm, q_full, h * HD + 64 * j, q_row0_1);
      }
      bool ok = true;
      for (int t = 0; t < nkv && ok; ++t) {
        const int st = t & 1;
        const uint32_t ph = static_cast<uint32_t>((t >> 1) & 1);
        int row0, valid;
        seq_tile(p, b, L, t, row0, valid);
        if (!mbar_wait(&k_empty[st], ph ^ 1u, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 1)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&k_full[st], C::TILE_BYTES);
#pragma unroll
        for (int j = 0; j < C::NBOX; ++j)
          tma_load_2d(sK(st) + j * BOX_BYTES, &tm, &k_full[st], p.d + h * HD + 64 * j, row0);
        armed_k |= 1u << st;
        par_k = (par_k & ~(1u << st)) | (ph << st);
        if (!mbar_wait(&v_empty[st], ph ^ 1u, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 2)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&v_full[st], C::TILE_BYTES);
#pragma unroll
        for (int j = 0; j < C::NBOX; ++j)
          tma_load_2d(sV(st) + j * BOX_BYTES, &tm, &v_full[st], 2 * p.d + h * HD + 64 * j, row0);
        armed_v |= 1u << st;
        par_v = (par_v & ~(1u << st)) | (ph << st);
      }
      if (!ok) {
        // wait (bounded) for the bulk copies in flight before the CTA exits
        const uint64_t t0 = globaltimer_ns();
        const uint64_t lim = HILO_WAIT_LIMIT_NS / 4;
        while (!mbar_try_wait(smem_u32(q_full), 0u) && globaltimer_ns() - t0 < lim) {
        }
        for (int st = 0; st < 2; ++st) {
          if ((armed_k >> st) & 1u)
            while (!mbar_try_wait(smem_u32(&k_full[st]), (par_k >> st) & 1u) &&
                   globaltimer_ns() - t0 < lim) {
            }
          if ((armed_v >> st) & 1u)
            while (!mbar_try_wait(smem_u32(&v_full[st]), (par_v >> st) & 1u) &&
                   globaltimer_ns() - t0 < lim) {
            }
        }
      }
    }
  } else if (warp == MMA_WARP) {
    if (lane == 0) {
      // ---------------- MMA issuer
      const uint32_t idesc_s = idesc_bf16(BQ, BKV, 0, 0);
      const uint32_t idesc_o = idesc_bf16(BQ, HD, 0, 1);
      auto issue_s = [&](int i, int t) {
        const uint32_t q_base = smem_u32(sQ(i));
        const uint32_t k_base = smem_u32(sK(t & 1));
#pragma unroll
        for (int k = 0; k < HD / 16; ++k) {
          const uint32_t off = (k >> 2) * BOX_BYTES + (k & 3) * 32;
          umma_bf16(tmem + 128u * i, sw128_desc(q_base + off, 16, 1024),
                    sw128_desc(k_base + off, 16, 1024), idesc_s, k > 0 ? 1u : 0u);
        }
        umma_commit(&s_full[i]);
      };
      // O_i += P_i V: P_i from the first 64 TMEM columns of S_i (8 columns =
      // 16 keys per MMA), V from shared memory
      auto issue_pv = [&](int i, int t) {
        const uint32_t v_base = smem_u32(sV(t & 1));
#pragma unroll
        for (int k = 0; k < BKV / 16; ++k) {
          const uint64_t bd = sw128_desc(v_base + k * 2048, BOX_BYTES, 1024);
          umma_bf16_tmem_a(tmem + 256u + 128u * i, tmem + 128u * i + 8u * k, bd, idesc_o,
                           (t > 0 || k > 0) ? 1u : 0u);
        }
        umma_commit(&o_done[i]);
      };
      bool ok = mbar_wait(q_full, 0u, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 3) &&
                mbar_wait(&k_full[0], 0u, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 4);
      if (ok) {
        tc_fence_after();
        issue_s(0, 0);
        if (has1) issue_s(1, 0);
        umma_commit(&k_empty[0]);
      }
      for (int t = 0; t < nkv && ok; ++t) {
        const int st = t & 1;
        const uint32_t ph = static_cast<uint32_t>((t >> 1) & 1);
        const uint32_t tp = static_cast<uint32_t>(t & 1);
        const bool more = t + 1 < nkv;
        const int st1 = (t + 1) & 1;
        const uint32_t ph1 = static_cast<uint32_t>(((t + 1) >> 1) & 1);
        if (!mbar_wait(&p_full[0], tp, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 5) ||
            !mbar_wait(&v_full[st], ph, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 6)) {
          ok = false;
          break;
        }
        tc_fence_after();
        issue_pv(0, t);
        if (!has1) umma_commit(&v_empty[st]);
        if (more) {
          if (!mbar_wait(&k_full[st1], ph1, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 7)) {
            ok = false;
            break;
          }
          tc_fence_after();
          issue_s(0, t + 1);
          if (!has1) umma_commit(&k_empty[st1]);
        }
        if (has1) {
          if (!mbar_wait(&p_full[1], tp, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 8)) {
            ok = false;
            break;
          }
          tc_fence_after();
          issue_pv(1, t);
          umma_commit(&v_empty[st]);
          if (more) {
            issue_s(1, t + 1);
            umma_commit(&k_empty[st1]);
          }
        }
      }
      umma_commit(drain);
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(smem_u32(drain), 0u)) {
        if (globaltimer_ns() - t0 > HILO_WAIT_LIMIT_NS) {
          atomicExch(err, DEV_TIMEOUT_ATTN + 256 * 9);
          break;
        }
      }
    }
    }
  } else {
    setmaxnreg_inc<SOFTMAX_REGS>();
    // ---------------- softmax: warpgroup i = warps 4i..4i+3, TMEM lane quarter warp % 4
    const int i = warp >> 2;
    const int row = (warp & 3) * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t tS = tmem + 128u * i + lane_off;
    const uint32_t tO = tmem + 256u + 128u * i + lane_off;
    const bool active = i == 0 || has1;
    float m = -INFINITY, l = 0.f;
    bool ok = active;
    // PROP: key weights of tile tt into the warp's slot tt & 1 (text tiles
    // weigh 1; columns past the ragged end 0), one commit group per call
    float* wslots = reinterpret_cast<float*>(smem + C::OFF_W) + warp * 2 * BKV;
    auto fetch_weights = [&](int tt) {
      if (tt < nkv) {
        float* wb = wslots + (tt & 1) * BKV;
        if (tt < p.qt_txt) {
#pragma unroll
          for (int u = 0; u < 4; ++u) wb[lane + 32 * u] = 1.0f;
        } else {
          int r0, v;
          seq_tile(p, b, L, tt, r0, v);
          const float* src = p.n_img + (min(p.cu_img[b], p.cap) + (tt - p.qt_txt) * BKV);
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int col = lane + 32 * u;
            cp_async4(smem_u32(wb + col), col < v ? src + col : p.n_img, col < v ? 4u : 0u);
          }
        }
      }
      cp_async_commit();
    };
    // ragged key tile: rows past `valid` hold other tokens (or stale data);
    // zero them in V so that the zero-probability columns add exactly 0.
    // Returns false when the wait for V gave up.
    auto zero_v_tail = [&](int t, int valid) -> bool {
      if (i == 0 && valid < BKV) {
        if (!mbar_wait_warp(&v_full[t & 1], static_cast<uint32_t>((t >> 1) & 1), abort_flag, err,
                            DEV_TIMEOUT_ATTN + 256 * 11))
          return false;
        if (row >= valid) {
          unsigned char* vr = sV(t & 1) + row * 128;
#pragma unroll
          for (int j = 0; j < C::NBOX; ++j)
#pragma unroll
            for (int c16 = 0; c16 < 8; ++c16)
              *reinterpret_cast<uint4*>(vr + j * BOX_BYTES + c16 * 16) = make_uint4(0, 0, 0, 0);
        }
      }
      return true;
    };
    // S_i(t) complete means every earlier MMA is too (PV_i(t-1) included),
    // so O_i can be rescaled and P_i written over S_i without another wait.
    // tcgen05.ld / tcgen05.st are warp-collective: the whole warp rescales
    // when any of its rows needs it (rows that do not use alpha = 1)
    auto rescale_o = [&](bool rescale, float m_use) {
      if (__any_sync(0xffffffffu, rescale)) {
        const float alpha = rescale ? ex2(m - m_use) : 1.0f;
#pragma unroll 1
        for (int c = 0; c < HD / 32; ++c) {
          float o[32];
          tmem_ld32(tO + c * 32, o);
          tmem_ld_wait();
#pragma unroll
          for (int j = 0; j < 32; ++j) o[j] *= alpha;
          tmem_st32(tO + c * 32, o);
        }
        l *= alpha;
      }
    };
    if (PROP && active) fetch_weights(0);
    for (int t = 0; t < nkv && ok; ++t) {
      int row0, valid;
      seq_tile(p, b, L, t, row0, valid);
      const uint32_t tp = static_cast<uint32_t>(t & 1);
      if (PROP) {
        // every lane is done with slot (t + 1) & 1 (read for tile t - 1)
        // before the next tile's weights are fetched into it
        __syncwarp();
        fetch_weights(t + 1);
      }
      if (!mbar_wait_warp(&s_full[i], tp, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 10)) {
        ok = false;
        break;
      }
      tc_fence_after();
      // row max and row sum with 8 independent partials combined by a tree,
      // so the reductions do not form one 128-long dependent chain (the max
      // of a full tile takes two keys per three-input max); only the
      // last key tile of a segment is ragged and needs masking
      const bool full_tile = valid == BKV;
      float s[BKV];
#pragma unroll
      for (int c = 0; c < BKV / 32; ++c) tmem_ld32(tS + c * 32, s + c * 32);
      tmem_ld_wait();
      float mx8[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) mx8[u] = -INFINITY;
      if (full_tile) {
#pragma unroll
        for (int j = 0; j < BKV; j += 16)
#pragma unroll
          for (int u = 0; u < 8; ++u) mx8[u] = fmax3(mx8[u], s[j + u], s[j + 8 + u]);
      } else {
#pragma unroll
        for (int j = 0; j < BKV; ++j)
          if (j < valid) mx8[j & 7] = fmaxf(mx8[j & 7], s[j]);
      }
      const float mx = fmax3(fmax3(mx8[0], mx8[1], mx8[2]), fmax3(mx8[3], mx8[4], mx8[5]),
                             fmaxf(mx8[6], mx8[7]));
      const float m_tile = mx * p.scale_log2;
      bool rescale = false;
      float m_use = m;
      if (t == 0) {
        m_use = m_tile;
      } else if (m_tile > m + RESCALE_LOG2) {
        m_use = m_tile;
        rescale = true;
      }
      float ls8[8];
      if (PROP) {
        // probabilities by key pairs: exponent argument s*scale - m as one
        // paired fma, two exp2, times the pair's weights (one paired mul);
        // the row sum's partials (2u, 2u+1) for pair c with u = c mod 4 are
        // the same partition and order as key j into partial j mod 8.
        // Masked columns are 0, selected, never computed from their stale
        // logits. First: this tile's weights have landed (all groups but the
        // newest) and are visible to the whole warp.
        cp_async_wait<1>();
        __syncwarp();
        const uint64_t* w2 = reinterpret_cast<const uint64_t*>(wslots + (t & 1) * BKV);
        const uint64_t sc2 = f2(p.scale_log2, p.scale_log2), nm2 = f2(-m_use, -m_use);
        uint64_t ls4[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) ls4[u] = 0ull;
#pragma unroll
        for (int c = 0; c < BKV / 2; ++c) {
          float a, a1;
          f2_split(f2_fma(f2(s[2 * c], s[2 * c + 1]), sc2, nm2), a, a1);
          a = (full_tile || 2 * c < valid) ? ex2(a) : 0.f;
          a1 = (full_tile || 2 * c + 1 < valid) ? ex2(a1) : 0.f;
          const uint64_t pr = f2_mul(f2(a, a1), w2[c]);
          f2_split(pr, s[2 * c], s[2 * c + 1]);
          ls4[c & 3] = f2_add(ls4[c & 3], pr);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) f2_split(ls4[u], ls8[2 * u], ls8[2 * u + 1]);
      } else {
#pragma unroll
        for (int u = 0; u < 8; ++u) ls8[u] = 0.f;
        if (full_tile) {
#pragma unroll
          for (int j = 0; j < BKV; ++j) {
            const float pj = ex2(fmaf(s[j], p.scale_log2, -m_use));
            s[j] = pj;
            ls8[j & 7] += pj;
          }
        } else {
#pragma unroll
          for (int j = 0; j < BKV; ++j) {
            const float pj = j < valid ? ex2(fmaf(s[j], p.scale_log2, -m_use)) : 0.f;
            s[j] = pj;
            ls8[j & 7] += pj;
          }
        }
      }
      const float lsum = ((ls8[0] + ls8[1]) + (ls8[2] + ls8[3])) + ((ls8[4] + ls8[5]) + (ls8[6] + ls8[7]));
      if (!zero_v_tail(t, valid)) {
        ok = false;
        break;
      }
      rescale_o(rescale, m_use);
      m = m_use;
      l += lsum;
      // P_i as bf16 pairs (keys 2c, 2c+1 in column c) over the first 64
      // columns of S_i, the A operand of the PV product
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
        float pk[32];
#pragma unroll
        for (int c = 0; c < 32; ++c)
          pk[c] = __uint_as_float(pack_bf16x2(s[64 * h2 + 2 * c], s[64 * h2 + 2 * c + 1]));
        tmem_st32(tS + 32 * h2, pk);
      }
      tmem_st_wait();
      fence_proxy_async_smem();  // the zeroed V rows, if any, are read by the tensor core
      tc_fence_before();
      mbar_arrive(&p_full[i]);
    }
    if (PROP) cp_async_wait<0>();  // no copy in flight when the CTA leaves
    if (ok && mbar_wait_warp(&o_done[i], static_cast<uint32_t>((nkv - 1) & 1), abort_flag, err,
                        DEV_TIMEOUT_ATTN + 256 * 14)) {
      tc_fence_after();
      const float inv = 1.0f / l;
      const int qr0 = i ? q_row0_1 : q_row0_0, qv = i ? q_valid_1 : q_valid_0;
      // O_i normalised to bf16 rows, staged through shared memory so that the
      // global stores leave as whole 128-byte lines (one row per lane would
      // write 16 bytes into 32 different rows per instruction). Each warp
      // owns a slice of the K stages: every S product, the last reader of K,
      // completed before O_i did, and no K copy is left to come. The 16-byte
      // units of a row are XOR-swizzled by the row, so neither the writes
      // (one row per lane) nor the reads (consecutive units of a row) collide
      // in the shared-memory banks.
      constexpr int UNITS = HD / 8;   // 16-byte units per row
      constexpr int RPI = 32 / UNITS;  // rows per store instruction
      uint4* stage = reinterpret_cast<uint4*>(smem + C::OFF_K) + warp * 32 * UNITS;
#pragma unroll 1
      for (int c = 0; c < HD / 32; ++c) {
        float o[32];
        tmem_ld32(tO + c * 32, o);
        tmem_ld_wait();
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          uint4 v;
          v.x = pack_bf16x2(o[8 * j] * inv, o[8 * j + 1] * inv);
          v.y = pack_bf16x2(o[8 * j + 2] * inv, o[8 * j + 3] * inv);
          v.z = pack_bf16x2(o[8 * j + 4] * inv, o[8 * j + 5] * inv);
          v.w = pack_bf16x2(o[8 * j + 6] * inv, o[8 * j + 7] * inv);
          stage[lane * UNITS + ((4 * c + j) ^ (lane & (UNITS - 1)))] = v;
        }
      }
      __syncwarp();
      const int u = lane % UNITS;
#pragma unroll 4
      for (int k = 0; k < 32 / RPI; ++k) {
        const int rr = k * RPI + lane / UNITS;  // row within the warp's 32
        const int qrow = (warp & 3) * 32 + rr;  // row within the query tile
        if (qrow < qv)
          reinterpret_cast<uint4*>(p.out + static_cast<long long>(qr0 + qrow) * p.d + h * HD)[u] =
              stage[rr * UNITS + (u ^ (rr & (UNITS - 1)))];
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == MMA_WARP) {
    tc_fence_after();
    tmem_dealloc(tmem, ATTN_TMEM_COLS);
  }
}

template <int HD, bool PROP>
cudaError_t launch_hd(const AttnArgs& a, const AttnParams& p, int grid, cudaStream_t st) {
  CUtensorMap tm;
  if (!encode_tmap_bf16_2d(&tm, a.qkv, 3ull * a.d, a.R, 3ull * a.d, 64, 128))
    return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(attn_kernel<HD, PROP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Cfg<HD, PROP>::SMEM_BYTES);
  if (e != cudaSuccess) return e;
  // the register split must fit what the CTA is launched with, or the
  // softmax warpgroups' setmaxnreg.inc would wait for registers forever
  static int regs = -1;
  if (regs < 0) {
    cudaFuncAttributes fa;
    e = cudaFuncGetAttributes(&fa, attn_kernel<HD, PROP>);
    if (e != cudaSuccess) return e;
    regs = fa.numRegs;
  }
  if (static_cast<long long>(regs) * ATTN_THREADS < 256LL * SOFTMAX_REGS + 128LL * CONTROL_REGS)
    return cudaErrorInvalidConfiguration;
  return launch_pdl(attn_kernel<HD, PROP>, dim3(grid), dim3(ATTN_THREADS), Cfg<HD, PROP>::SMEM_BYTES, st, tm,
                    p);
}

}  // namespace

cudaError_t launch_attention(const AttnArgs& a, int num_sms, cudaStream_t st) {
  (void)num_sms;
  AttnParams p;
  p.cu_img = a.cu_img;
  p.n_img = a.n_img;
  p.out = static_cast<__nv_bfloat16*>(a.out);
  p.B = a.B;
  p.T = a.T;
  p.heads = a.heads;
  p.d = a.d;
  p.qt_txt = (a.T + BQ - 1) / BQ;
  p.cap = a.R - a.B * a.T;
  const int qt_img_max = (a.max_img_rows + BQ - 1) / BQ;
  p.pairs_max = (p.qt_txt + qt_img_max + 1) / 2;
  p.scale_log2 = static_cast<float>(1.4426950408889634 / sqrt(static_cast<double>(a.head_dim)));
  const long long items = static_cast<long long>(a.B) * a.heads * p.pairs_max;
  if (items <= 0) return cudaSuccess;
  if (items > 0x7fffffffLL) return cudaErrorInvalidValue;
  if (a.n_img) {
    if (a.head_dim == 128) return launch_hd<128, true>(a, p, static_cast<int>(items), st);
    if (a.head_dim == 64) return launch_hd<64, true>(a, p, static_cast<int>(items), st);
    return cudaErrorInvalidValue;
  }
  if (a.head_dim == 128) return launch_hd<128, false>(a, p, static_cast<int>(items), st);
  if (a.head_dim == 64) return launch_hd<64, false>(a, p, static_cast<int>(items), st);
  return cudaErrorInvalidValue;
}

int attn_take_device_error() {
  int v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_attn_err, sizeof(int)) != cudaSuccess) return -1;
  if (v) cudaMemcpyToSymbol(g_attn_err, &z, sizeof(int));
  return v;
}

int attn_take_rows_error() {
  int v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_attn_rows_err, sizeof(int)) != cudaSuccess) return -1;
  if (v) cudaMemcpyToSymbol(g_attn_rows_err, &z, sizeof(int));
  return v;
}

}  // namespace hilo
