// extern "C" entry points of libhilo (declared in include/hilo.h): argument
// and shape validation on the host, workspace layout, launch orchestration
// of the kernels, device error reporting. The path they run is paper
// Sec. 2.3 (selection, pooling, the DiT on the compressed sequence,
// restoration); each entry point's passage is cited in include/hilo.h.
#include <cuda.h>
#include <cuda_runtime.h>
#include <atomic>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include "../../include/hilo.h"
#include "internal.h"

namespace {

thread_local char g_last_error[512] = "";
thread_local cudaEvent_t g_stage_ev[16];
thread_local int g_stage_n = 0;
std::atomic<unsigned long long> g_launches{0};

void stage_mark(int k, cudaStream_t s) {
  if (k < g_stage_n && g_stage_ev[k]) cudaEventRecord(g_stage_ev[k], s);
}

void count(int n) { g_launches.fetch_add(static_cast<unsigned long long>(n), std::memory_order_relaxed); }

int fail(int status, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_last_error, sizeof(g_last_error), fmt, ap);
  va_end(ap);
  return status;
}

int cuda_fail(cudaError_t e, const char* where) {
  return fail(HILO_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

struct DevInfo {
  int num_sms = 0;
  int major = 0, minor = 0;
};

// per-device cache (index = device ordinal)
DevInfo g_dev[64];

int current_device(DevInfo** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= 64) return fail(HILO_ERR_UNSUPPORTED, "device ordinal %d", dev);
  DevInfo& d = g_dev[dev];
  if (d.num_sms == 0) {
    e = cudaDeviceGetAttribute(&d.major, cudaDevAttrComputeCapabilityMajor, dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&d.minor, cudaDevAttrComputeCapabilityMinor, dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&d.num_sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) {
      d.num_sms = 0;
      return cuda_fail(e, "cudaDeviceGetAttribute");
    }
  }
  if (d.major != 10 || d.minor != 3)
    return fail(HILO_ERR_UNSUPPORTED, "libhilo is built for sm_103a; device is sm_%d%d", d.major,
                d.minor);
  *out = &d;
  return HILO_OK;
}

int check_shape(const hilo_shape* s, bool need_block) {
  if (!s) return fail(HILO_ERR_ARG, "shape is NULL");
  if (s->B < 1) return fail(HILO_ERR_SHAPE, "B=%d must be >= 1", s->B);
  if (s->H < 2 || s->W < 2 || (s->H & 1) || (s->W & 1))
    return fail(HILO_ERR_SHAPE, "H=%d, W=%d must be even and >= 2", s->H, s->W);
  if (s->levels != 1 && s->levels != 2) return fail(HILO_ERR_SHAPE, "levels=%d must be 1 or 2", s->levels);
  if (s->levels == 2 && ((s->H & 3) || (s->W & 3)))
    return fail(HILO_ERR_SHAPE, "H=%d, W=%d must be multiples of 4 for two-level pooling", s->H, s->W);
  if (s->lf != 0 && s->lf != 2 && s->lf != 4 && s->lf != 8)
    return fail(HILO_ERR_SHAPE, "lf=%d must be 0, 2, 4 or 8", s->lf);
  if (s->lf && (s->levels != 1 || s->H % s->lf || s->W % s->lf))
    return fail(HILO_ERR_SHAPE, "lf=%d needs levels=1 and H=%d, W=%d multiples of lf", s->lf, s->H, s->W);
  if (static_cast<long long>(s->H) * s->W > 32768)
    return fail(HILO_ERR_SHAPE, "H*W=%lld exceeds 32768 tokens per image",
                static_cast<long long>(s->H) * s->W);
  if (s->d < 128 || s->d % 128 || s->d > 4096)
    return fail(HILO_ERR_SHAPE, "d=%d must be a multiple of 128 in [128, 4096]", s->d);
  {
    // row indices (packed rows, cu_img, the block's row space) are int32
    const long long N = static_cast<long long>(s->H) * s->W;
    const long long per_image = N + (s->lf ? N / (s->lf * s->lf) : 0) + (s->T > 0 ? s->T : 0);
    if (static_cast<long long>(s->B) * per_image > 0x7FFFFFFFLL)
      return fail(HILO_ERR_SHAPE, "B=%d images of %lld rows exceed the int32 row space", s->B, per_image);
  }
  if (need_block) {
    if (s->T < 0) return fail(HILO_ERR_SHAPE, "T=%d must be >= 0", s->T);
    if (s->heads < 1 || s->d % s->heads) return fail(HILO_ERR_SHAPE, "heads=%d must divide d=%d", s->heads, s->d);
    const int hd = s->d / s->heads;
    if (hd != 64 && hd != 128) return fail(HILO_ERR_SHAPE, "head_dim=%d must be 64 or 128", hd);
    if (s->mlp != 0 && s->mlp != 1) return fail(HILO_ERR_SHAPE, "mlp=%d must be 0 or 1", s->mlp);
  }
  return HILO_OK;
}

int check_split(const hilo_split_out* sp) {
  if (!sp || !sp->labels || !sp->row_src || !sp->counts || !sp->cu_img || !sp->tok_row)
    return fail(HILO_ERR_ARG, "split output pointer is NULL");
  return HILO_OK;
}

inline size_t align256(size_t v) { return (v + 255) & ~static_cast<size_t>(255); }

struct BlockWs {
  size_t ln, qkv, attn, hid, total;
};

BlockWs block_ws_layout(const hilo_shape* s, int32_t cap) {
  const size_t R = static_cast<size_t>(s->B) * s->T + static_cast<size_t>(cap);
  const size_t d = static_cast<size_t>(s->d);
  BlockWs w;
  w.ln = 0;
  w.qkv = w.ln + align256(R * d * 2);
  w.attn = w.qkv + align256(R * 3 * d * 2);
  w.hid = w.attn + align256(R * d * 2);
  w.total = w.hid + (s->mlp ? align256(R * 4 * d * 2) : 0);
  return w;
}

// FP8 block: one e4m3 buffer for the A operand of every GEMM (LayerNorm
// outputs, attention output, MLP hidden; each used before the next is
// written, in stream order) with its per-row scales, then bf16 q|k|v and
// attention rows and the fp16 MLP hidden rows.
struct BlockWs8 {
  size_t q8, qs, qkv, attn, hid, total;
};

BlockWs8 block_fp8_ws_layout(const hilo_shape* s, int32_t cap) {
  const size_t R = static_cast<size_t>(s->B) * s->T + static_cast<size_t>(cap);
  const size_t d = static_cast<size_t>(s->d);
  BlockWs8 w;
  w.q8 = 0;
  w.qs = w.q8 + align256(R * (s->mlp ? 4 * d : d));
  w.qkv = w.qs + align256(R * 4);
  w.attn = w.qkv + align256(R * 3 * d * 2);
  w.hid = w.attn + align256(R * d * 2);
  w.total = w.hid + (s->mlp ? align256(R * 4 * d * 2) : 0);
  return w;
}

}  // namespace

namespace hilo {

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                    const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                    const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                    CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// The driver's tensor-map encoder, resolved through the runtime so that the
// library does not link libcuda (and loads on hosts without a driver).
static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

bool encode_tmap_2d(CUtensorMap* map, TmapType type, const void* base, uint64_t inner, uint64_t outer,
                    uint64_t row_stride_elems, uint32_t box_inner, uint32_t box_outer) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  CUtensorMapDataType dt = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  uint64_t esize = 2;
  if (type == TMAP_F16) dt = CU_TENSOR_MAP_DATA_TYPE_FLOAT16;
  if (type == TMAP_F32) {
    dt = CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
    esize = 4;
  }
  if (type == TMAP_U8) {
    dt = CU_TENSOR_MAP_DATA_TYPE_UINT8;
    esize = 1;
  }
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_stride_elems * esize};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, dt, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool encode_tmap_bf16_2d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
                         uint64_t row_stride_elems, uint32_t box_inner, uint32_t box_outer) {
  return encode_tmap_2d(map, TMAP_BF16, base, inner, outer, row_stride_elems, box_inner, box_outer);
}

// Sets the calling thread's hilo_last_error() text and returns `status`
// (for entry points defined in other files).
int set_error(int status, const char* msg) { return fail(status, "%s", msg); }

int check_block_shape(const hilo_shape* shape) { return check_shape(shape, true); }

}  // namespace hilo

extern "C" {

const char* hilo_status_string(int status) {
  switch (status) {
    case HILO_OK: return "HILO_OK";
    case HILO_ERR_ARG: return "HILO_ERR_ARG";
    case HILO_ERR_SHAPE: return "HILO_ERR_SHAPE";
    case HILO_ERR_CUDA: return "HILO_ERR_CUDA";
    case HILO_ERR_WORKSPACE: return "HILO_ERR_WORKSPACE";
    case HILO_ERR_TIMEOUT: return "HILO_ERR_TIMEOUT";
    case HILO_ERR_UNSUPPORTED: return "HILO_ERR_UNSUPPORTED";
    case HILO_ERR_CHECK: return "HILO_ERR_CHECK";
    default: return "HILO_ERR_UNKNOWN";
  }
}

const char* hilo_last_error(void) { return g_last_error; }

int hilo_device_info(int* num_sms, int* is_sm103) {
  int dev = 0, major = 0, minor = 0, n = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return cuda_fail(e, "hilo_device_info");
  if (num_sms) *num_sms = n;
  if (is_sm103) *is_sm103 = (major == 10 && minor == 3) ? 1 : 0;
  return HILO_OK;
}

int hilo_sync_status(void* stream) {
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "hilo_sync_status: stream");
  const int g = hilo::gemm_take_device_error();
  const int g2 = hilo::gemm2_take_device_error();
  const int a = hilo::attn_take_device_error();
  const int pr = hilo::probe_take_device_error();
  const int dc = hilo::dcheck_take_bw();
  if (g < 0 || g2 < 0 || a < 0 || pr < 0 || dc < 0)
    return fail(HILO_ERR_CUDA, "hilo_sync_status: reading the device error word failed");
  if (g || g2 || a || pr)
    return fail(HILO_ERR_TIMEOUT, "device-side wait ran out (gemm=%d, gemm pair=%d, attention=%d, probe=%d)", g,
                g2, a, pr);
  if (dc) return fail(HILO_ERR_CHECK, "device-side index check %d failed (checks build)", dc);
  return HILO_OK;
}

int hilo_debug_wait_timeout(void* stream) {
  const cudaError_t e = hilo::launch_wait_probe(static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? HILO_OK : cuda_fail(e, "hilo_debug_wait_timeout");
}

int hilo_score(const hilo_shape* shape, const void* x, float* score, void* stream) {
  int st = check_shape(shape, false);
  if (st) return st;
  if (!x || !score) return fail(HILO_ERR_ARG, "hilo_score: NULL pointer");
  DevInfo* dev;
  if ((st = current_device(&dev))) return st;
  cudaError_t e = hilo::launch_score(x, score, shape->B, shape->H, shape->W, shape->d, dev->num_sms,
                                     static_cast<cudaStream_t>(stream));
  if (e == cudaSuccess) count(1);
  return e == cudaSuccess ? HILO_OK : cuda_fail(e, "hilo_score");
}

size_t hilo_split_workspace_bytes(const hilo_shape* shape) {
  (void)shape;
  return 0;
}

static int split_common(const char* name, const hilo_shape* shape, const float* score, const uint8_t* mask,
                        const int32_t* k_keep, const int32_t* k_mid, const hilo_split_out* out, int granular,
                        void* stream) {
  int st = check_shape(shape, false);
  if (st) return st;
  if ((st = check_split(out))) return st;
  if (!score || !mask || !k_keep) return fail(HILO_ERR_ARG, "%s: NULL pointer", name);
  if (shape->levels == 2 && !k_mid) return fail(HILO_ERR_ARG, "%s: k_mid is NULL with levels=2", name);
  DevInfo* dev;
  if ((st = current_device(&dev))) return st;
  cudaError_t e = hilo::launch_split(score, mask, k_keep, shape->levels == 2 ? k_mid : k_keep,
                                     out->labels, out->row_src, out->counts, out->cu_img,
                                     out->tok_row, shape->B, shape->H, shape->W, shape->levels, granular,
                                     shape->lf, static_cast<cudaStream_t>(stream));
  if (e == cudaSuccess) count(shape->B == 1 ? 1 : 2);  // one image: the select kernel also compacts
  return e == cudaSuccess ? HILO_OK : cuda_fail(e, name);
}

int hilo_split(const hilo_shape* shape, const float* score, const uint8_t* mask,
               const int32_t* k_keep, const int32_t* k_mid, const hilo_split_out* out, void* ws,
               size_t ws_bytes, void* stream) {
  (void)ws;
  (void)ws_bytes;
  return split_common("hilo_split", shape, score, mask, k_keep, k_mid, out, 0, stream);
}

int hilo_split_regions(const hilo_shape* shape, const float* score, const uint8_t* mask,
                       const int32_t* k_keep, const int32_t* k_mid, const hilo_split_out* out, void* ws,
                       size_t ws_bytes, void* stream) {
  (void)ws;
  (void)ws_bytes;
  if (shape && shape->lf)
    return fail(HILO_ERR_ARG, "hilo_split_regions: the window-granular split has no low-frequency mode");
  return split_common("hilo_split_regions", shape, score, mask, k_keep, k_mid, out, 1, stream);
}

size_t hilo_sobel_workspace_bytes(const hilo_shape* shape) {
  if (check_shape(shape, false)) return 0;
  return hilo::sobel_workspace_bytes(shape->B, shape->H, shape->W);
}

int hilo_sobel_select(const hilo_shape* shape, const float* img, int channels, int patch,
                      const uint8_t* mask, int radius, float threshold, uint8_t* keep, void* ws,
                      size_t ws_bytes, void* stream) {
  int st = check_shape(shape, false);
  if (st) return st;
  if (!img || !mask || !keep || !ws) return fail(HILO_ERR_ARG, "hilo_sobel_select: NULL pointer");
  if (channels < 1 || channels > 4)
    return fail(HILO_ERR_ARG, "hilo_sobel_select: channels=%d must be in [1, 4]", channels);
  if (patch != 8 && patch != 16) return fail(HILO_ERR_ARG, "hilo_sobel_select: patch=%d must be 8 or 16", patch);
  if (radius < 0 || radius > 64) return fail(HILO_ERR_ARG, "hilo_sobel_select: radius=%d must be in [0, 64]", radius);
  if (!(threshold == threshold) || threshold > 3.0e38f || threshold < -3.0e38f)
    return fail(HILO_ERR_ARG, "hilo_sobel_select: threshold must be finite");
  if (reinterpret_cast<uintptr_t>(ws) & 15)
    return fail(HILO_ERR_ARG, "hilo_sobel_select: workspace must be 16-byte aligned");
  const size_t need = hilo::sobel_workspace_bytes(shape->B, shape->H, shape->W);
  if (ws_bytes < need)
    return fail(HILO_ERR_WORKSPACE, "hilo_sobel_select: workspace %zu < %zu bytes", ws_bytes, need);
  DevInfo* dev;
  if ((st = current_device(&dev))) return st;
  cudaError_t e = hilo::launch_sobel_select(img, shape->B, shape->H, shape->W, channels, patch, mask, radius,
                                            threshold, keep, ws, dev->num_sms, static_cast<cudaStream_t>(stream));
  if (e == cudaSuccess) count(2);
  return e == cudaSuccess ? HILO_OK : cuda_fail(e, "hilo_sobel_select");
}

int hilo_pack(const hilo_shape* shape, const void* x, const hilo_split_out* split, void* packed,
              int32_t cap, void* stream) {
  int st = check_shape(shape, false);
  if (st) return st;
  if ((st = check_split(split))) return st;
  if (!x || !packed) return fail(HILO_ERR_ARG, "hilo_pack: NULL pointer");
  if (cap < 0) return fail(HILO_ERR_ARG, "hilo_pack: cap=%d", cap);
  DevInfo* dev;
  if ((st = current_device(&dev))) return st;
  cudaError_t e = hilo::launch_pack(x, split->labels, split->row_src, split->counts, split->cu_img,
                                    packed, shape->B, shape->H, shape->W, shape->d, cap, shape->lf,
                                    dev->num_sms, static_cast<cudaStream_t>(stream));
  if (e == cudaSuccess) count(1);
  return e == cudaSuccess ? HILO_OK : cuda_fail(e, "hilo_pack");
}

size_t hilo_row_capacity(const hilo_shape* shape) {
  if (check_shape(shape, false)) return 0;
  const size_t N = static_cast<size_t>(shape->H) * shape->W;
  return static_cast<size_t>(shape->B) * (N + (shape->lf ? N / (shape->lf * shape->lf) : 0));
}

size_t hilo_block_workspace_bytes(const hilo_shape* shape, int32_t cap) {
  if (!shape || cap < 0) return 0;
  return block_ws_layout(shape, cap).total;
}

// The block of hilo_block_forward; n_img != NULL selects proportional
// attention (hilo_block_forward_prop).
static int block_forward_impl(const hilo_shape* shape, const hilo_block_weights* w, const int32_t* cu_img,
                              int32_t cap, const void* in_txt, const void* in_img, int in_dtype,
                              const float* n_img, float* out, void* ws, size_t ws_bytes, void* stream) {
  int st = check_shape(shape, true);
  if (st) return st;
  if (!w || !cu_img || !in_img || !out) return fail(HILO_ERR_ARG, "hilo_block_forward: NULL pointer");
  if (shape->T > 0 && !in_txt) return fail(HILO_ERR_ARG, "hilo_block_forward: in_txt is NULL with T>0");
  if ((reinterpret_cast<uintptr_t>(in_txt) | reinterpret_cast<uintptr_t>(in_img) |
       reinterpret_cast<uintptr_t>(out)) & 15)
    return fail(HILO_ERR_ARG, "hilo_block_forward: in_txt, in_img and out must be 16-byte aligned");
  if (in_dtype != HILO_BF16 && in_dtype != HILO_F32)
    return fail(HILO_ERR_ARG, "hilo_block_forward: in_dtype=%d", in_dtype);
  if (cap < 0) return fail(HILO_ERR_ARG, "hilo_block_forward: cap=%d", cap);
  const hilo_stream_weights* sw[2] = {&w->txt, &w->img};
  for (int i = 0; i < 2; ++i) {
    if (i == 0 && shape->T == 0) continue;
    if (!sw[i]->w_qkv || !sw[i]->b_qkv || !sw[i]->w_o || !sw[i]->b_o)
      return fail(HILO_ERR_ARG, "hilo_block_forward: %s attention weight is NULL", i ? "image" : "text");
    if (shape->mlp && (!sw[i]->w_1 || !sw[i]->b_1 || !sw[i]->w_2 || !sw[i]->b_2))
      return fail(HILO_ERR_ARG, "hilo_block_forward: %s MLP weight is NULL", i ? "image" : "text");
  }
  const BlockWs L = block_ws_layout(shape, cap);
  if (!ws || ws_bytes < L.total)
    return fail(HILO_ERR_WORKSPACE, "hilo_block_forward: workspace %zu < %zu bytes", ws_bytes, L.total);
  DevInfo* dev;
  if ((st = current_device(&dev))) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int B = shape->B, T = shape->T, d = shape->d;
  const int BT = B * T;
  const int R = BT + cap;
  char* base = static_cast<char*>(ws);
  void* ln = base + L.ln;
  void* qkv = base + L.qkv;
  void* attn = base + L.attn;
  void* hid = base + L.hid;
  const int in_f32 = in_dtype == HILO_F32;
  const bool in_place = in_f32 && in_txt == out && in_img == out + static_cast<size_t>(BT) * d;
  const bool in_place_img = in_f32 && BT == 0 && in_img == out;

  stage_mark(0, s);
  // the residual is read from the input by the out-projection epilogue (no
  // fp32 copy of it is made) unless the input already is the output buffer
  cudaError_t e = hilo::launch_layernorm(in_txt, in_img, in_f32, nullptr, ln, 0, nullptr, cu_img, B, BT, cap, d,
                                         dev->num_sms, s);
  if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward: layernorm 1");
  count(1);
  stage_mark(1, s);

  auto gemm = [&](const void* A, int op_f16, int N, int K, int epi, void* o,
                  const void* wt, const void* bt, const void* wi, const void* bi) {
    hilo::GemmArgs g;
    if (epi == hilo::EPI_BIAS_RESIDIN_F32) {
      g.resid_src[0] = in_txt;
      g.resid_src[1] = in_img;
      g.resid_f32 = in_f32;
    }
    g.A = A;
    g.op_f16 = op_f16;
    g.R = R;
    g.N = N;
    g.K = K;
    g.epilogue = epi;
    g.out = o;
    g.g[0] = {0, BT, nullptr, wt, bt, BT};
    g.g[1] = {BT, 0, cu_img + B, wi, bi, cap};
    cudaError_t ge = hilo::launch_gemm(g, dev->num_sms, s);
    if (ge == cudaSuccess) count(1);
    return ge;
  };
  e = gemm(ln, 0, 3 * d, d, hilo::EPI_BIAS_BF16, qkv, w->txt.w_qkv, w->txt.b_qkv, w->img.w_qkv, w->img.b_qkv);
  if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward: qkv gemm");
  stage_mark(2, s);

  hilo::AttnArgs aa;
  aa.qkv = qkv;
  aa.out = attn;
  aa.cu_img = cu_img;
  aa.n_img = n_img;
  aa.B = B;
  aa.T = T;
  aa.heads = shape->heads;
  aa.head_dim = d / shape->heads;
  aa.d = d;
  aa.R = R;
  e = hilo::launch_attention(aa, dev->num_sms, s);
  if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward: attention");
  count(1);
  stage_mark(3, s);

  e = gemm(attn, 0, d, d, (in_place || in_place_img) ? hilo::EPI_BIAS_RESID_F32 : hilo::EPI_BIAS_RESIDIN_F32, out, w->txt.w_o, w->txt.b_o, w->img.w_o, w->img.b_o);
  if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward: out-projection gemm");
  stage_mark(4, s);
  if (shape->mlp) {
    e = hilo::launch_layernorm(out, out + static_cast<size_t>(BT) * d, 1, nullptr, ln, 1, nullptr, cu_img, B, BT,
                               cap, d, dev->num_sms, s);
    if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward: layernorm 2");
    count(1);
    stage_mark(5, s);
    e = gemm(ln, 1, 4 * d, d, hilo::EPI_BIAS_GELU_F16, hid, w->txt.w_1, w->txt.b_1, w->img.w_1, w->img.b_1);
    if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward: mlp1 gemm");
    stage_mark(6, s);
    e = gemm(hid, 1, d, 4 * d, hilo::EPI_BIAS_RESID_F32, out, w->txt.w_2, w->txt.b_2, w->img.w_2, w->img.b_2);
    if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward: mlp2 gemm");
    stage_mark(7, s);
  }
  return HILO_OK;
}

int hilo_block_forward(const hilo_shape* shape, const hilo_block_weights* w, const int32_t* cu_img,
                       int32_t cap, const void* in_txt, const void* in_img, int in_dtype,
                       float* out, void* ws, size_t ws_bytes, void* stream) {
  return block_forward_impl(shape, w, cu_img, cap, in_txt, in_img, in_dtype, nullptr, out, ws, ws_bytes,
                            stream);
}

int hilo_block_forward_prop(const hilo_shape* shape, const hilo_block_weights* w, const int32_t* cu_img,
                            int32_t cap, const void* in_txt, const void* in_img, int in_dtype,
                            const float* n_img, float* out, void* ws, size_t ws_bytes, void* stream) {
  if (!n_img) return fail(HILO_ERR_ARG, "hilo_block_forward_prop: n_img is NULL");
  if (reinterpret_cast<uintptr_t>(n_img) & 3)
    return fail(HILO_ERR_ARG, "hilo_block_forward_prop: n_img must be 4-byte aligned");
  return block_forward_impl(shape, w, cu_img, cap, in_txt, in_img, in_dtype, n_img, out, ws, ws_bytes,
                            stream);
}

int hilo_quantize_rows_e4m3(const void* src, int src_dtype, int64_t rows, int32_t cols, uint8_t* dst,
                            float* scale, void* stream) {
  if (!src || !dst || !scale) return fail(HILO_ERR_ARG, "hilo_quantize_rows_e4m3: NULL pointer");
  if (src_dtype != HILO_BF16 && src_dtype != HILO_F16 && src_dtype != HILO_F32)
    return fail(HILO_ERR_ARG, "hilo_quantize_rows_e4m3: src_dtype=%d", src_dtype);
  if (rows < 0 || rows > 0x7fffffff || cols < 0 || cols % 8)
    return fail(HILO_ERR_ARG, "hilo_quantize_rows_e4m3: rows=%lld, cols=%d (a multiple of 8)",
                static_cast<long long>(rows), cols);
  if ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15)
    return fail(HILO_ERR_ARG, "hilo_quantize_rows_e4m3: src and dst must be 16-byte aligned");
  DevInfo* dev;
  int st;
  if ((st = current_device(&dev))) return st;
  if (rows == 0 || cols == 0) return HILO_OK;
  const int type = src_dtype == HILO_BF16 ? 0 : (src_dtype == HILO_F16 ? 1 : 2);
  cudaError_t e = hilo::launch_quant_rows(src, type, cols, static_cast<int>(rows), nullptr, 0, 0, 0, dst, scale,
                                          dev->num_sms, static_cast<cudaStream_t>(stream));
  if (e == cudaSuccess) count(1);
  return e == cudaSuccess ? HILO_OK : cuda_fail(e, "hilo_quantize_rows_e4m3");
}

size_t hilo_block_fp8_workspace_bytes(const hilo_shape* shape, int32_t cap) {
  if (!shape || cap < 0) return 0;
  return block_fp8_ws_layout(shape, cap).total;
}

// The block of hilo_block_forward_fp8; n_img != NULL selects proportional
// attention (hilo_block_forward_fp8_prop).
static int block_forward_fp8_impl(const hilo_shape* shape, const hilo_block_weights_fp8* w,
                                  const int32_t* cu_img, int32_t cap, const void* in_txt, const void* in_img,
                                  int in_dtype, const float* n_img, float* out, void* ws, size_t ws_bytes,
                                  void* stream) {
  int st = check_shape(shape, true);
  if (st) return st;
  if (shape->d < 1024 || shape->d % 256)
    return fail(HILO_ERR_SHAPE, "hilo_block_forward_fp8: d=%d must be a multiple of 256, at least 1024",
                shape->d);
  if (!w || !cu_img || !in_img || !out) return fail(HILO_ERR_ARG, "hilo_block_forward_fp8: NULL pointer");
  if (shape->T > 0 && !in_txt) return fail(HILO_ERR_ARG, "hilo_block_forward_fp8: in_txt is NULL with T>0");
  if ((reinterpret_cast<uintptr_t>(in_txt) | reinterpret_cast<uintptr_t>(in_img) |
       reinterpret_cast<uintptr_t>(out)) & 15)
    return fail(HILO_ERR_ARG, "hilo_block_forward_fp8: in_txt, in_img and out must be 16-byte aligned");
  if (in_dtype != HILO_BF16 && in_dtype != HILO_F32)
    return fail(HILO_ERR_ARG, "hilo_block_forward_fp8: in_dtype=%d", in_dtype);
  if (cap < 0) return fail(HILO_ERR_ARG, "hilo_block_forward_fp8: cap=%d", cap);
  const hilo_stream_weights_fp8* sw[2] = {&w->txt, &w->img};
  for (int i = 0; i < 2; ++i) {
    if (i == 0 && shape->T == 0) continue;
    const hilo_stream_weights_fp8& x = *sw[i];
    if (!x.w_qkv || !x.s_qkv || !x.b_qkv || !x.w_o || !x.s_o || !x.b_o)
      return fail(HILO_ERR_ARG, "hilo_block_forward_fp8: %s attention weight is NULL", i ? "image" : "text");
    if (shape->mlp && (!x.w_1 || !x.s_1 || !x.b_1 || !x.w_2 || !x.s_2 || !x.b_2))
      return fail(HILO_ERR_ARG, "hilo_block_forward_fp8: %s MLP weight is NULL", i ? "image" : "text");
    if ((reinterpret_cast<uintptr_t>(x.s_qkv) | reinterpret_cast<uintptr_t>(x.s_o) |
         reinterpret_cast<uintptr_t>(x.s_1) | reinterpret_cast<uintptr_t>(x.s_2)) & 15)
      return fail(HILO_ERR_ARG, "hilo_block_forward_fp8: weight scales must be 16-byte aligned");
  }
  const BlockWs8 L = block_fp8_ws_layout(shape, cap);
  if (!ws || ws_bytes < L.total)
    return fail(HILO_ERR_WORKSPACE, "hilo_block_forward_fp8: workspace %zu < %zu bytes", ws_bytes, L.total);
  DevInfo* dev;
  if ((st = current_device(&dev))) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int B = shape->B, T = shape->T, d = shape->d;
  const int BT = B * T;
  const int R = BT + cap;
  char* base = static_cast<char*>(ws);
  uint8_t* q8 = reinterpret_cast<uint8_t*>(base + L.q8);
  float* qs = reinterpret_cast<float*>(base + L.qs);
  void* qkv = base + L.qkv;
  void* attn = base + L.attn;
  void* hid = base + L.hid;
  const int in_f32 = in_dtype == HILO_F32;
  const bool in_place = in_f32 && in_txt == out && in_img == out + static_cast<size_t>(BT) * d;
  const bool in_place_img = in_f32 && BT == 0 && in_img == out;

  stage_mark(0, s);
  cudaError_t e = hilo::launch_layernorm(in_txt, in_img, in_f32, nullptr, q8, 2, qs, cu_img, B, BT, cap, d,
                                         dev->num_sms, s);
  if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward_fp8: layernorm 1");
  count(1);
  stage_mark(1, s);
  auto gemm = [&](int N, int K, int epi, void* o, const void* wt, const float* st_, const void* bt,
                  const void* wi, const float* si, const void* bi) {
    hilo::GemmArgs g;
    if (epi == hilo::EPI_BIAS_RESIDIN_F32) {
      g.resid_src[0] = in_txt;
      g.resid_src[1] = in_img;
      g.resid_f32 = in_f32;
    }
    g.A = q8;
    g.op_f16 = 0;
    g.fp8 = 1;
    g.a_scale = qs;
    g.R = R;
    g.N = N;
    g.K = K;
    g.epilogue = epi;
    g.out = o;
    g.g[0] = {0, BT, nullptr, wt, bt, BT, st_};
    g.g[1] = {BT, 0, cu_img + B, wi, bi, cap, si};
    cudaError_t ge = hilo::launch_gemm(g, dev->num_sms, s);
    if (ge == cudaSuccess) count(1);
    return ge;
  };
  const hilo_stream_weights_fp8 &wt = w->txt, &wi = w->img;
  e = gemm(3 * d, d, hilo::EPI_BIAS_BF16, qkv, wt.w_qkv, wt.s_qkv, wt.b_qkv, wi.w_qkv, wi.s_qkv, wi.b_qkv);
  if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward_fp8: qkv gemm");
  stage_mark(2, s);
  hilo::AttnArgs aa;
  aa.qkv = qkv;
  aa.out = attn;
  aa.cu_img = cu_img;
  aa.n_img = n_img;
  aa.B = B;
  aa.T = T;
  aa.heads = shape->heads;
  aa.head_dim = d / shape->heads;
  aa.d = d;
  aa.R = R;
  e = hilo::launch_attention(aa, dev->num_sms, s);
  if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward_fp8: attention");
  count(1);
  e = hilo::launch_quant_rows(attn, 0, d, 0, cu_img, B, BT, cap, q8, qs, dev->num_sms, s);
  if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward_fp8: attention quantisation");
  count(1);
  stage_mark(3, s);
  e = gemm(d, d, (in_place || in_place_img) ? hilo::EPI_BIAS_RESID_F32 : hilo::EPI_BIAS_RESIDIN_F32, out, wt.w_o,
           wt.s_o, wt.b_o, wi.w_o, wi.s_o, wi.b_o);
  if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward_fp8: out-projection gemm");
  stage_mark(4, s);
  if (shape->mlp) {
    e = hilo::launch_layernorm(out, out + static_cast<size_t>(BT) * d, 1, nullptr, q8, 2, qs, cu_img, B, BT, cap,
                               d, dev->num_sms, s);
    if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward_fp8: layernorm 2");
    count(1);
    stage_mark(5, s);
    e = gemm(4 * d, d, hilo::EPI_BIAS_GELU_F16, hid, wt.w_1, wt.s_1, wt.b_1, wi.w_1, wi.s_1, wi.b_1);
    if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward_fp8: mlp1 gemm");
    e = hilo::launch_quant_rows(hid, 1, 4 * d, 0, cu_img, B, BT, cap, q8, qs, dev->num_sms, s);
    if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward_fp8: hidden quantisation");
    count(1);
    stage_mark(6, s);
    e = gemm(d, 4 * d, hilo::EPI_BIAS_RESID_F32, out, wt.w_2, wt.s_2, wt.b_2, wi.w_2, wi.s_2, wi.b_2);
    if (e != cudaSuccess) return cuda_fail(e, "hilo_block_forward_fp8: mlp2 gemm");
    stage_mark(7, s);
  }
  return HILO_OK;
}

int hilo_block_forward_fp8(const hilo_shape* shape, const hilo_block_weights_fp8* w, const int32_t* cu_img,
                           int32_t cap, const void* in_txt, const void* in_img, int in_dtype, float* out,
                           void* ws, size_t ws_bytes, void* stream) {
  return block_forward_fp8_impl(shape, w, cu_img, cap, in_txt, in_img, in_dtype, nullptr, out, ws, ws_bytes,
                                stream);
}

int hilo_block_forward_fp8_prop(const hilo_shape* shape, const hilo_block_weights_fp8* w, const int32_t* cu_img,
                                int32_t cap, const void* in_txt, const void* in_img, int in_dtype,
                                const float* n_img, float* out, void* ws, size_t ws_bytes, void* stream) {
  if (!n_img) return fail(HILO_ERR_ARG, "hilo_block_forward_fp8_prop: n_img is NULL");
  if (reinterpret_cast<uintptr_t>(n_img) & 3)
    return fail(HILO_ERR_ARG, "hilo_block_forward_fp8_prop: n_img must be 4-byte aligned");
  return block_forward_fp8_impl(shape, w, cu_img, cap, in_txt, in_img, in_dtype, n_img, out, ws, ws_bytes,
                                stream);
}

int hilo_row_sizes(const hilo_shape* shape, const hilo_split_out* split, float* n_img, int32_t cap,
                   void* stream) {
  int st = check_shape(shape, false);
  if (st) return st;
  if ((st = check_split(split))) return st;
  if (!n_img) return fail(HILO_ERR_ARG, "hilo_row_sizes: NULL pointer");
  if (cap < 0) return fail(HILO_ERR_ARG, "hilo_row_sizes: cap=%d", cap);
  DevInfo* dev;
  if ((st = current_device(&dev))) return st;
  cudaError_t e = hilo::launch_row_sizes(split->labels, split->row_src, split->counts, split->cu_img, n_img,
                                         shape->B, shape->H, shape->W, cap, shape->lf, dev->num_sms,
                                         static_cast<cudaStream_t>(stream));
  if (e == cudaSuccess && cap > 0) count(1);
  return e == cudaSuccess ? HILO_OK : cuda_fail(e, "hilo_row_sizes");
}

int hilo_unpack(const hilo_shape* shape, const float* out_img, const hilo_split_out* split, float* y,
                void* stream) {
  int st = check_shape(shape, false);
  if (st) return st;
  if ((st = check_split(split))) return st;
  if (!out_img || !y) return fail(HILO_ERR_ARG, "hilo_unpack: NULL pointer");
  DevInfo* dev;
  if ((st = current_device(&dev))) return st;
  const long long ntok = static_cast<long long>(shape->B) * shape->H * shape->W;
  const long long rows_max = static_cast<long long>(hilo_row_capacity(shape));
  cudaError_t e = hilo::launch_unpack(out_img, split->tok_row, y, ntok, shape->d, rows_max, dev->num_sms,
                                      static_cast<cudaStream_t>(stream));
  if (e == cudaSuccess) count(1);
  return e == cudaSuccess ? HILO_OK : cuda_fail(e, "hilo_unpack");
}

int hilo_unpack_delta(const hilo_shape* shape, const float* out_img, const void* packed, const void* x,
                      const hilo_split_out* split, float* y, void* stream) {
  int st = check_shape(shape, false);
  if (st) return st;
  if ((st = check_split(split))) return st;
  if (!out_img || !packed || !x || !y) return fail(HILO_ERR_ARG, "hilo_unpack_delta: NULL pointer");
  if ((reinterpret_cast<uintptr_t>(out_img) | reinterpret_cast<uintptr_t>(packed) |
       reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(y)) & 15)
    return fail(HILO_ERR_ARG, "hilo_unpack_delta: pointers must be 16-byte aligned");
  DevInfo* dev;
  if ((st = current_device(&dev))) return st;
  const long long ntok = static_cast<long long>(shape->B) * shape->H * shape->W;
  cudaError_t e = hilo::launch_unpack_delta(out_img, packed, x, split->labels, split->tok_row, y, ntok,
                                            shape->d, static_cast<long long>(hilo_row_capacity(shape)),
                                            dev->num_sms, static_cast<cudaStream_t>(stream));
  if (e == cudaSuccess) count(1);
  return e == cudaSuccess ? HILO_OK : cuda_fail(e, "hilo_unpack_delta");
}

int hilo_unpack_update(const hilo_shape* shape, const float* out_img, const hilo_split_out* split,
                       void* x, float alpha, void* stream) {
  int st = check_shape(shape, false);
  if (st) return st;
  if ((st = check_split(split))) return st;
  if (!out_img || !x) return fail(HILO_ERR_ARG, "hilo_unpack_update: NULL pointer");
  DevInfo* dev;
  if ((st = current_device(&dev))) return st;
  const long long ntok = static_cast<long long>(shape->B) * shape->H * shape->W;
  cudaError_t e = hilo::launch_unpack_update(out_img, split->tok_row, x, ntok, shape->d, alpha,
                                             static_cast<long long>(hilo_row_capacity(shape)), dev->num_sms,
                                             static_cast<cudaStream_t>(stream));
  if (e == cudaSuccess) count(1);
  return e == cudaSuccess ? HILO_OK : cuda_fail(e, "hilo_unpack_update");
}

int hilo_convert_bf16_to_f16(const void* src, void* dst, size_t n, void* stream) {
  if (!src || !dst) return fail(HILO_ERR_ARG, "hilo_convert_bf16_to_f16: NULL pointer");
  if (n % 8) return fail(HILO_ERR_ARG, "hilo_convert_bf16_to_f16: n=%zu is not a multiple of 8", n);
  if ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15)
    return fail(HILO_ERR_ARG, "hilo_convert_bf16_to_f16: pointers must be 16-byte aligned");
  DevInfo* dev;
  int st;
  if ((st = current_device(&dev))) return st;
  if (n == 0) return HILO_OK;
  cudaError_t e = hilo::launch_bf16_to_f16(src, dst, static_cast<long long>(n), dev->num_sms,
                                           static_cast<cudaStream_t>(stream));
  if (e == cudaSuccess) count(1);
  return e == cudaSuccess ? HILO_OK : cuda_fail(e, "hilo_convert_bf16_to_f16");
}

int hilo_set_stage_events(void* const* events, int n) {
  if (n < 0 || n > 16 || (n > 0 && !events)) return fail(HILO_ERR_ARG, "hilo_set_stage_events: n=%d", n);
  for (int i = 0; i < n; ++i) g_stage_ev[i] = static_cast<cudaEvent_t>(events[i]);
  g_stage_n = n;
  return HILO_OK;
}

unsigned long long hilo_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

}  // extern "C"
