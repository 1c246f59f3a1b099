// Host side of the C ABI (include/dfs.h): plan construction (index tables I_t and
// compacted per-step panels, Sec. 4.3), the per-step block forward, the few-step loop
// and the test hooks.  All device work goes to the caller's stream.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <mutex>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "../../include/dfs.h"
#include "kernels.cuh"

using dfs::bf16;

namespace {

thread_local std::string g_last_error;

dfs_status fail(dfs_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

#define DFS_CK(expr)                                                                           \
  do {                                                                                         \
    cudaError_t e_ = (expr);                                                                   \
    if (e_ != cudaSuccess) return fail(DFS_ECUDA, "%s failed: %s", #expr, cudaGetErrorString(e_)); \
  } while (0)

// ------------------------------------------------------------------ tensor maps

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
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

// 2D bf16 map over a row-major [outer, inner] array with row pitch `ld` elements, a box
// of box_inner x box_outer elements (box_inner * 2 = 128 B) and 128-byte swizzle;
// out-of-range elements read as zero.
bool make_map(CUtensorMap* m, const void* base, long long inner, long long outer, long long ld, int box_inner,
              int box_outer) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || inner <= 0 || outer <= 0) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(outer)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(box_inner), static_cast<cuuint32_t>(box_outer)};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Tensor map of an fp32 [outer, inner] row-major matrix (leading dimension ld elements) with a
// {32, 32} box and the 128-byte swizzle: the GEMM epilogue's TMA output stores.
bool make_map_out_f32(CUtensorMap* m, const void* base, long long inner, long long outer, long long ld) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || inner <= 0 || outer <= 0) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(outer)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 4};
  cuuint32_t box[2] = {32, 32};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

long long round_up(long long v, long long m) { return (v + m - 1) / m * m; }

}  // namespace

// ------------------------------------------------------------------ plan

struct Panel {
  bf16* p = nullptr;
  long long rows = 0, cols = 0, ld = 0;
};

struct StepLayer {
  int h_s = 0, f_s = 0, hc = 0;
  std::vector<int> heads, chunks, xheads;
  std::vector<int> pos_heads, pos_chunks, pos_xheads;  // positions inside the layer's union
  int* up_rows_u = nullptr;    // union engine: union W_up rows of the step's FFN channels [f_s]
  int* down_segs_u = nullptr;  // union engine: union W_down 8-column segments of its chunks [f_s / 8]
  Panel P[15];       // indexed like dfs_plan_panel's `which`
  bf16* kc = nullptr;    // cross-attention context keys, normalised [ctx_len, hc dh]
  bf16* vct = nullptr;   // cross-attention context values, transposed [hc dh, ctx_ld]
  dfs::GemmArgs g_qkv, g_o, g_up, g_down, g_cq, g_co;
  dfs::AttnArgs a_self, a_cross;
  double flops = 0;
};

// The union super-model of one layer (Sec. 4.3): ids of the units retained at any step and,
// under DFS_ENGINE_UNION, the weights of exactly those units.
struct LayerUnion {
  std::vector<int> heads, chunks, xheads;
  Panel wqkv, wo, wup, wdown, cwq, cwo;  // indexed like dfs_plan_union_panel's `which`
};

struct LayerConst {
  bf16* bo = nullptr;
  bf16* bdown = nullptr;
  bf16* emod = nullptr;
  bf16* cbo = nullptr;
  float* cln_w = nullptr;
  float* cln_b = nullptr;
};

struct dfs_plan {
  dfs_config cfg;
  int N = 0, T = 0, L = 0, num_sms = 0, device = 0;
  std::vector<uint8_t> block_gate;
  std::vector<StepLayer> sl;  // [T * L]
  std::vector<LayerConst> lc;
  std::vector<LayerUnion> lu;  // [L]
  bool uni = false;            // DFS_ENGINE_UNION
  bf16* ffn_up_s = nullptr;    // union engine: the forward's FFN panels, gathered from the
  bf16* ffn_down_s = nullptr;  //   union at every forward ([f_s, d] and [d, f_s], largest step)
  long long bytes_total = 0, bytes_weights = 0;
  std::vector<void*> temps;    // device buffers needed only during plan creation
  // model around the blocks (dfs_model_attach)
  bool has_model = false;
  int mC = 0, mD = 0;
  bf16 *m_patch_w = nullptr, *m_patch_b = nullptr, *m_t_w1 = nullptr, *m_t_b1 = nullptr, *m_t_w2 = nullptr,
       *m_t_b2 = nullptr, *m_head_mod = nullptr, *m_head_w = nullptr, *m_head_b = nullptr;
  bf16 *m_tok = nullptr, *m_x0 = nullptr, *m_vtok = nullptr, *m_temb = nullptr;
  float *m_freq = nullptr, *m_h1 = nullptr, *m_temb_f = nullptr, *m_hm = nullptr;
  dfs::GemmArgs g_embed, g_head;
  bf16* w_t = nullptr;
  bf16* b_t = nullptr;
  dfs::RopeTables rope{};
  float* mod = nullptr;       // [6, d] for the current layer
  float* mod_base = nullptr;  // [T, 6, d] W_t t_emb + b_t per step (denoise)
  bf16* xm = nullptr;
  bf16* qk = nullptr;
  bf16* vt = nullptr;
  long long vt_ld = 0, ctx_ld = 0;
  bf16* attn = nullptr;
  float* x1 = nullptr;
  bf16* h = nullptr;
  bf16* qc = nullptr;
  bf16* act[2] = {nullptr, nullptr};
  bf16* stage_x = nullptr;
  bf16* stage_out = nullptr;
  bf16* stage_t = nullptr;
  // Two-slot staging ring of dfs_block_forward_host_async (slot 0 is stage_x / stage_out /
  // stage_t): host->device copies on `h2d`, device->host copies on `d2h`, ordered against
  // the caller's stream by per-slot events.
  struct HostRing {
    bool ready = false;
    int next = 0;
    bf16* x[2] = {nullptr, nullptr};
    bf16* out[2] = {nullptr, nullptr};
    bf16* t[2] = {nullptr, nullptr};
    cudaStream_t h2d = nullptr, d2h = nullptr;
    cudaEvent_t loaded[2] = {nullptr, nullptr};    // slot's inputs on the device
    cudaEvent_t computed[2] = {nullptr, nullptr};  // slot's forward done (inputs free, output ready)
    cudaEvent_t drained[2] = {nullptr, nullptr};   // slot's output copied to the host
  } ring;
  int* err = nullptr;
  std::vector<void*> allocs;
  int last_step = -1, last_layer = -1;
  int fault_alloc = -1, n_alloc = 0;  // host-side fault injection (DFS_FAULT_ALLOC=n)
  long long fault_launch = -1, n_launch = 0;  // (DFS_FAULT_LAUNCH=n: the n-th launch fails)
  // per-kernel profiling: event pairs recorded around launches while prof_on
  bool prof_on = false;
  std::vector<cudaEvent_t> ev;  // pool, pairs (2i, 2i+1)
  std::vector<int> ev_kind;     // kind of each recorded pair
  size_t ev_used = 0;
  long long launches[DFS_K_COUNT] = {0};
};

namespace {

dfs_status dev_alloc(dfs_plan* P, void** out, size_t bytes) {
  *out = nullptr;
  ++P->n_alloc;
  if (P->fault_alloc > 0 && P->n_alloc == P->fault_alloc)
    return fail(DFS_ENOMEM, "injected allocation failure at allocation %d", P->n_alloc);
  if (bytes == 0) return DFS_OK;
  cudaError_t e = cudaMalloc(out, bytes);
  if (e != cudaSuccess) {
    *out = nullptr;
    (void)cudaGetLastError();
    return fail(DFS_ENOMEM, "cudaMalloc(%zu) failed: %s", bytes, cudaGetErrorString(e));
  }
  P->allocs.push_back(*out);
  P->bytes_total += static_cast<long long>(bytes);
  return DFS_OK;
}

template <typename T>
dfs_status alloc_n(dfs_plan* P, T** out, long long n) {
  return dev_alloc(P, reinterpret_cast<void**>(out), static_cast<size_t>(n) * sizeof(T));
}

// A weight panel of the plan (counted in bytes_weights).
dfs_status alloc_weights(dfs_plan* P, bf16** out, long long n) {
  dfs_status e = alloc_n(P, out, n);
  if (!e) P->bytes_weights += 2 * n;
  return e;
}

// A device buffer freed at the end of plan creation (not counted as held by the plan).
dfs_status alloc_temp(dfs_plan* P, bf16** out, long long n) {
  *out = nullptr;
  ++P->n_alloc;
  if (P->fault_alloc > 0 && P->n_alloc == P->fault_alloc)
    return fail(DFS_ENOMEM, "injected allocation failure at allocation %d", P->n_alloc);
  if (n == 0) return DFS_OK;
  cudaError_t e = cudaMalloc(reinterpret_cast<void**>(out), static_cast<size_t>(n) * sizeof(bf16));
  if (e != cudaSuccess) {
    *out = nullptr;
    (void)cudaGetLastError();
    return fail(DFS_ENOMEM, "cudaMalloc(%lld) failed: %s", 2 * n, cudaGetErrorString(e));
  }
  P->temps.push_back(*out);
  return DFS_OK;
}

void free_plan(dfs_plan* P) {
  if (!P) return;
  for (cudaEvent_t e : P->ev) cudaEventDestroy(e);
  {
    dfs_plan::HostRing& R = P->ring;
    if (R.h2d) cudaStreamSynchronize(R.h2d);
    if (R.d2h) cudaStreamSynchronize(R.d2h);
    for (int b = 0; b < 2; ++b)
      for (cudaEvent_t e : {R.loaded[b], R.computed[b], R.drained[b]})
        if (e) cudaEventDestroy(e);
    if (R.h2d) cudaStreamDestroy(R.h2d);
    if (R.d2h) cudaStreamDestroy(R.d2h);
  }
  for (void* p : P->allocs) cudaFree(p);
  for (void* p : P->temps) cudaFree(p);
  delete P;
}

// ------------------------------------------------------------------ per-kernel profiling

const char* const kKindNames[DFS_K_COUNT] = {"dfs modulation", "dfs adaln", "dfs gemm_qkv", "dfs qk_norm_rope",
                                             "dfs attention", "dfs gemm_o", "dfs gemm_up", "dfs gemm_down",
                                             "dfs cross", "dfs other", "dfs gather", "dfs model"};

// Brackets one kernel launch: an NVTX range named by its kind (seen by Nsight tools, free
// without one), an event before and after it on `st` while profiling is on, and the launch
// count.  `inject` is set for the launch DFS_FAULT_LAUNCH names, which is then skipped and
// reported as a failed launch (host-side fault injection; nothing reaches the GPU).
struct ProfScope {
  dfs_plan* P;
  int kind;
  cudaStream_t st;
  int pair = -1;
  bool inject = false;
  ProfScope(dfs_plan* p, int k, cudaStream_t s) : P(p), kind(k), st(s) {
    nvtxRangePushA(kKindNames[kind]);
    ++P->launches[kind];
    inject = ++P->n_launch == P->fault_launch;
    if (!P->prof_on || inject) return;
    if (2 * P->ev_used + 2 > P->ev.size()) {
      cudaEvent_t a, b;
      if (cudaEventCreate(&a) != cudaSuccess) return;
      if (cudaEventCreate(&b) != cudaSuccess) { cudaEventDestroy(a); return; }
      P->ev.push_back(a);
      P->ev.push_back(b);
      P->ev_kind.push_back(kind);
    }
    pair = static_cast<int>(P->ev_used++);
    P->ev_kind[pair] = kind;
    cudaEventRecord(P->ev[2 * pair], st);
  }
  ~ProfScope() {
    if (pair >= 0) cudaEventRecord(P->ev[2 * pair + 1], st);
    nvtxRangePop();
  }
};

#define DFS_LAUNCH(kind, expr)                                                                  \
  do {                                                                                          \
    ProfScope prof_(P, (kind), st);                                                             \
    if (prof_.inject) return fail(DFS_ECUDA, "injected launch failure at launch %lld", P->n_launch); \
    DFS_CK(expr);                                                                               \
  } while (0)

// ------------------------------------------------------------------ validation (host only)

// Device buffers are read and written with 16-byte vectors and TMA (cudaMalloc and torch
// allocations are at least 256-byte aligned).
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

dfs_status validate(const dfs_config* c, const dfs_layer_weights* layers, const void* w_t, const void* b_t,
                    const dfs_masks* m, const void* ctx, dfs_plan** out) {
  if (!out) return fail(DFS_EINVAL, "out is NULL");
  *out = nullptr;
  if (!c) return fail(DFS_EINVAL, "cfg is NULL");
  if (c->head_dim != 64 && c->head_dim != 128) return fail(DFS_EINVAL, "head_dim must be 64 or 128");
  if (c->n_heads < 1 || c->dim != c->n_heads * c->head_dim)
    return fail(DFS_EINVAL, "dim (%d) must equal n_heads * head_dim", c->dim);
  if (c->dim > 8192) return fail(DFS_EUNSUPPORTED, "dim > 8192");
  if (c->ffn_chunk != 8) return fail(DFS_EINVAL, "ffn_chunk must be 8");
  if (c->ffn_dim < 8 || c->ffn_dim % c->ffn_chunk != 0)
    return fail(DFS_EINVAL, "ffn_dim (%d) must be a positive multiple of ffn_chunk", c->ffn_dim);
  if (c->n_layers < 1 || c->n_layers > 4096) return fail(DFS_EINVAL, "n_layers out of range");
  if (c->n_steps < 1 || c->n_steps > 8) return fail(DFS_EINVAL, "n_steps must be in 1..8");
  if (c->grid_t < 1 || c->grid_h < 1 || c->grid_w < 1) return fail(DFS_EINVAL, "grid dims must be >= 1");
  const long long N = static_cast<long long>(c->grid_t) * c->grid_h * c->grid_w;
  if (N > (1LL << 22)) return fail(DFS_EUNSUPPORTED, "more than 2^22 tokens");
  if (c->has_cross != 0 && c->has_cross != 1) return fail(DFS_EINVAL, "has_cross must be 0 or 1");
  if (c->has_cross && (c->ctx_len < 1 || c->ctx_len > 4096 || c->ctx_len % 8 != 0))
    return fail(DFS_EINVAL, "ctx_len must be a multiple of 8 in 8..4096");
  if (c->has_cross && !ctx) return fail(DFS_EINVAL, "ctx is NULL with has_cross");
  if (c->qk_norm_mode != 0 && c->qk_norm_mode != 1) return fail(DFS_EINVAL, "qk_norm_mode must be 0 or 1");
  if (c->engine != DFS_ENGINE_COMPACTED && c->engine != DFS_ENGINE_UNION)
    return fail(DFS_EINVAL, "engine must be DFS_ENGINE_COMPACTED or DFS_ENGINE_UNION");
  if (!(c->ln_eps > 0.f) || !(c->rope_theta > 1.f)) return fail(DFS_EINVAL, "ln_eps / rope_theta out of range");
  if (!layers || !w_t || !b_t || !m) return fail(DFS_EINVAL, "NULL weights or masks");
  for (int l = 0; l < c->n_layers; ++l) {
    const dfs_layer_weights& w = layers[l];
    const void* req[] = {w.wq, w.bq, w.wk, w.bk, w.wv, w.bv, w.wo, w.bo, w.gq, w.gk, w.w_up, w.b_up, w.w_down,
                         w.b_down, w.e_mod};
    for (const void* p : req) {
      if (!p) return fail(DFS_EINVAL, "layer %d: NULL weight pointer", l);
      if (!aligned16(p)) return fail(DFS_EINVAL, "layer %d: weight pointers must be 16-byte aligned", l);
    }
    if (c->has_cross) {
      const void* rc[] = {w.cwq, w.cbq, w.cwk, w.cbk, w.cwv, w.cbv, w.cwo, w.cbo, w.cgq, w.cgk, w.cln_w, w.cln_b};
      for (const void* p : rc) {
        if (!p) return fail(DFS_EINVAL, "layer %d: NULL cross-attention weight pointer", l);
        if (!aligned16(p)) return fail(DFS_EINVAL, "layer %d: weight pointers must be 16-byte aligned", l);
      }
    }
  }
  if (!aligned16(w_t) || !aligned16(b_t) || (c->has_cross && !aligned16(ctx)))
    return fail(DFS_EINVAL, "w_t, b_t and ctx must be 16-byte aligned");
  if (!m->block_gate || !m->head_gate || !m->ffn_gate) return fail(DFS_EINVAL, "NULL gate array");
  const long long TL = static_cast<long long>(c->n_steps) * c->n_layers;
  auto check01 = [](const uint8_t* g, long long n) {
    for (long long i = 0; i < n; ++i)
      if (g[i] > 1) return false;
    return true;
  };
  if (!check01(m->block_gate, TL) || !check01(m->head_gate, TL * c->n_heads) ||
      !check01(m->ffn_gate, TL * (c->ffn_dim / c->ffn_chunk)) ||
      (m->xhead_gate && !check01(m->xhead_gate, TL * c->n_heads)))
    return fail(DFS_EINVAL, "gate values must be 0 or 1");
  return DFS_OK;
}

// ------------------------------------------------------------------ GEMM / attention args

dfs::GemmArgs gemm_args(dfs_plan* P, const CUtensorMap& a, const CUtensorMap& b, int M, int N, int K, int mode,
                        const bf16* bias) {
  dfs::GemmArgs g;
  memset(&g, 0, sizeof(g));
  g.tma_a = a;
  g.tma_b = b;
  g.M = M; g.N = N; g.K = K;
  g.mode = mode;
  g.bias = bias;
  g.split = N;
  g.group = dfs::gemm_group(K);
  g.epi_warps = dfs::gemm_epilogue_warps(K);
  g.err = P->err;
  return g;
}

dfs_status upload_ints(dfs_plan* P, const std::vector<int>& v, int** out, cudaStream_t st) {
  *out = nullptr;
  if (v.empty()) return DFS_OK;
  dfs_status s = alloc_n(P, out, static_cast<long long>(v.size()));
  if (s) return s;
  DFS_CK(cudaMemcpyAsync(*out, v.data(), v.size() * sizeof(int), cudaMemcpyHostToDevice, st));
  return DFS_OK;
}

// Positions of `ids` (ascending) inside `uni` (ascending, a superset): the I_t table that
// addresses a step's units inside the union super-model.
std::vector<int> positions_in(const std::vector<int>& ids, const std::vector<int>& uni) {
  std::vector<int> pos;
  pos.reserve(ids.size());
  for (int id : ids)
    pos.push_back(static_cast<int>(std::lower_bound(uni.begin(), uni.end(), id) - uni.begin()));
  return pos;
}

// Builds the index lists, gathers the panels and prebuilds every kernel argument of
// one (step, layer).
dfs_status build_step_layer(dfs_plan* P, int s, int l, const dfs_layer_weights& w, const dfs_masks* m,
                            const void* ctx, cudaStream_t st, std::vector<std::vector<int>>& keep_alive) {
  const dfs_config& c = P->cfg;
  const int d = c.dim, H = c.n_heads, dh = c.head_dim, NC = c.ffn_dim / c.ffn_chunk;
  StepLayer& S = P->sl[s * P->L + l];
  const LayerUnion& U = P->lu[l];
  const bool uni = P->uni;
  const long long base = static_cast<long long>(s) * c.n_layers + l;
  for (int h = 0; h < H; ++h)
    if (m->head_gate[base * H + h]) S.heads.push_back(h);
  for (int k = 0; k < NC; ++k)
    if (m->ffn_gate[base * NC + k]) S.chunks.push_back(k);
  if (c.has_cross)
    for (int h = 0; h < H; ++h)
      if (!m->xhead_gate || m->xhead_gate[base * H + h]) S.xheads.push_back(h);
  S.h_s = static_cast<int>(S.heads.size());
  S.f_s = static_cast<int>(S.chunks.size()) * c.ffn_chunk;
  S.hc = static_cast<int>(S.xheads.size());
  S.pos_heads = positions_in(S.heads, U.heads);
  S.pos_chunks = positions_in(S.chunks, U.chunks);
  S.pos_xheads = positions_in(S.xheads, U.xheads);
  const int hd = S.h_s * dh, hcd = S.hc * dh, fs = S.f_s;
  const int N = P->N;

  // index lists: rows (one per channel) and 16-byte segments (8 channels each)
  std::vector<int> qk_rows, qk_segs, ffn_rows, x_rows, x_segs;
  for (int h : S.heads)
    for (int j = 0; j < dh; ++j) qk_rows.push_back(h * dh + j);
  for (int h : S.heads)
    for (int j = 0; j < dh / 8; ++j) qk_segs.push_back(h * dh / 8 + j);
  for (int k : S.chunks)
    for (int j = 0; j < c.ffn_chunk; ++j) ffn_rows.push_back(k * c.ffn_chunk + j);
  for (int h : S.xheads)
    for (int j = 0; j < dh; ++j) x_rows.push_back(h * dh + j);
  for (int h : S.xheads)
    for (int j = 0; j < dh / 8; ++j) x_segs.push_back(h * dh / 8 + j);
  int *d_qk_rows, *d_qk_segs, *d_ffn_rows, *d_chunks, *d_x_rows, *d_x_segs;
  dfs_status e;
  if ((e = upload_ints(P, qk_rows, &d_qk_rows, st)) || (e = upload_ints(P, qk_segs, &d_qk_segs, st)) ||
      (e = upload_ints(P, ffn_rows, &d_ffn_rows, st)) || (e = upload_ints(P, S.chunks, &d_chunks, st)) ||
      (e = upload_ints(P, x_rows, &d_x_rows, st)) || (e = upload_ints(P, x_segs, &d_x_segs, st)))
    return e;
  keep_alive.push_back(qk_rows);
  keep_alive.push_back(qk_segs);
  keep_alive.push_back(ffn_rows);
  keep_alive.push_back(x_rows);
  keep_alive.push_back(x_segs);

  // Union engine: the union rows of the step's FFN channels, which K1 gathers at every
  // forward (the head-granular projections carry their maps in their kernel arguments).
  if (uni) {
    std::vector<int> up_rows;
    for (int p : S.pos_chunks)
      for (int j = 0; j < c.ffn_chunk; ++j) up_rows.push_back(p * c.ffn_chunk + j);
    if ((e = upload_ints(P, up_rows, &S.up_rows_u, st)) || (e = upload_ints(P, S.pos_chunks, &S.down_segs_u, st)))
      return e;
    keep_alive.push_back(up_rows);
  }

  // per-step panels; under the union engine only the vectors (the weight matrices are read
  // from the union through the maps) and, for the duration of plan creation, cWkv
  // W_down [d, f_s] (7) gets a row pitch of whole 128-byte lines: f_s is a multiple of 8 only,
  // and TMA rows that straddle L2 lines slowed its projection by a quarter
  auto mk = [&](int which, long long rows, long long cols) -> dfs_status {
    Panel& p = S.P[which];
    p.rows = rows; p.cols = cols; p.ld = which == 7 ? round_up(cols, 64) : cols;
    if (rows * cols == 0) return DFS_OK;
    const bool matrix = which == 0 || which == 4 || which == 5 || which == 7 || which == 8 || which == 10 ||
                        which == 14;
    if (uni && matrix) return which == 10 ? alloc_temp(P, &p.p, rows * p.ld) : DFS_OK;
    return alloc_weights(P, &p.p, rows * p.ld);
  };
  const bf16* wq = static_cast<const bf16*>(w.wq);
  const bf16* wk = static_cast<const bf16*>(w.wk);
  const bf16* wv = static_cast<const bf16*>(w.wv);
  if ((e = mk(0, 3LL * hd, d)) || (e = mk(1, 1, 3LL * hd)) || (e = mk(2, 1, hd)) || (e = mk(3, 1, hd)) ||
      (e = mk(4, d, hd)) || (e = mk(5, fs, d)) || (e = mk(6, 1, fs)) || (e = mk(7, d, fs)))
    return e;
  if (c.has_cross) {
    if ((e = mk(8, hcd, d)) || (e = mk(9, 1, hcd)) || (e = mk(10, 2LL * hcd, d)) || (e = mk(11, 1, 2LL * hcd)) ||
        (e = mk(12, 1, hcd)) || (e = mk(13, 1, hcd)) || (e = mk(14, d, hcd)))
      return e;
  }
  // K1 gathers
  if (hd > 0) {
    if (!uni) {
      bf16* Wqkv = S.P[0].p;
      DFS_CK(dfs::launch_gather_rows(Wqkv, d, wq, d, d_qk_rows, hd, d, st));
      DFS_CK(dfs::launch_gather_rows(Wqkv + static_cast<long long>(hd) * d, d, wk, d, d_qk_rows, hd, d, st));
      DFS_CK(dfs::launch_gather_rows(Wqkv + 2LL * hd * d, d, wv, d, d_qk_rows, hd, d, st));
      DFS_CK(dfs::launch_gather_segs(S.P[4].p, hd, static_cast<const bf16*>(w.wo), d, d_qk_segs, hd / 8, d, st));
    }
    bf16* b = S.P[1].p;
    DFS_CK(dfs::launch_gather_segs(b, 0, static_cast<const bf16*>(w.bq), 0, d_qk_segs, hd / 8, 1, st));
    DFS_CK(dfs::launch_gather_segs(b + hd, 0, static_cast<const bf16*>(w.bk), 0, d_qk_segs, hd / 8, 1, st));
    DFS_CK(dfs::launch_gather_segs(b + 2 * hd, 0, static_cast<const bf16*>(w.bv), 0, d_qk_segs, hd / 8, 1, st));
    DFS_CK(dfs::launch_gather_segs(S.P[2].p, 0, static_cast<const bf16*>(w.gq), 0, d_qk_segs, hd / 8, 1, st));
    DFS_CK(dfs::launch_gather_segs(S.P[3].p, 0, static_cast<const bf16*>(w.gk), 0, d_qk_segs, hd / 8, 1, st));
  }
  if (fs > 0) {
    const int nch = static_cast<int>(S.chunks.size());
    if (!uni) {
      DFS_CK(dfs::launch_gather_rows(S.P[5].p, d, static_cast<const bf16*>(w.w_up), d, d_ffn_rows, fs, d, st));
      DFS_CK(dfs::launch_gather_segs(S.P[7].p, S.P[7].ld, static_cast<const bf16*>(w.w_down), c.ffn_dim, d_chunks,
                                     nch, d, st));
    }
    DFS_CK(dfs::launch_gather_segs(S.P[6].p, 0, static_cast<const bf16*>(w.b_up), 0, d_chunks, nch, 1, st));
  }
  if (c.has_cross && hcd > 0) {
    if (!uni) {
      DFS_CK(dfs::launch_gather_rows(S.P[8].p, d, static_cast<const bf16*>(w.cwq), d, d_x_rows, hcd, d, st));
      DFS_CK(dfs::launch_gather_segs(S.P[14].p, hcd, static_cast<const bf16*>(w.cwo), d, d_x_segs, hcd / 8, d,
                                     st));
    }
    DFS_CK(dfs::launch_gather_segs(S.P[9].p, 0, static_cast<const bf16*>(w.cbq), 0, d_x_segs, hcd / 8, 1, st));
    DFS_CK(dfs::launch_gather_rows(S.P[10].p, d, static_cast<const bf16*>(w.cwk), d, d_x_rows, hcd, d, st));
    DFS_CK(dfs::launch_gather_rows(S.P[10].p + static_cast<long long>(hcd) * d, d,
                                   static_cast<const bf16*>(w.cwv), d, d_x_rows, hcd, d, st));
    DFS_CK(dfs::launch_gather_segs(S.P[11].p, 0, static_cast<const bf16*>(w.cbk), 0, d_x_segs, hcd / 8, 1, st));
    DFS_CK(dfs::launch_gather_segs(S.P[11].p + hcd, 0, static_cast<const bf16*>(w.cbv), 0, d_x_segs, hcd / 8, 1,
                                   st));
    DFS_CK(dfs::launch_gather_segs(S.P[12].p, 0, static_cast<const bf16*>(w.cgq), 0, d_x_segs, hcd / 8, 1, st));
    DFS_CK(dfs::launch_gather_segs(S.P[13].p, 0, static_cast<const bf16*>(w.cgk), 0, d_x_segs, hcd / 8, 1, st));
  }

  // Union engine: B of a head-granular projection read from the union panel through its
  // map, in head units of the union.  Rows: group g (dh rows) of the step's [q | k | v] (or
  // cross q) rows is head pos[g % h] of section g / h; padded to the B tiles of 256 rows.
  // K columns: block k (64 columns) of the step's attention output is column block
  // (pos[k dh_blocks] dh + ...) / 64 of the union.
  const int nu = static_cast<int>(U.heads.size());
  auto gather_rows = [&](dfs::GemmArgs& g, const std::vector<int>& pos, int sections, int nunion) -> dfs_status {
    const int h = static_cast<int>(pos.size());
    const size_t len = static_cast<size_t>((static_cast<long long>(sections) * h * dh + 255) / 256) * 256 / dh;
    if (len > static_cast<size_t>(dfs::kGemmMapMax)) return fail(DFS_EUNSUPPORTED, "gather map too long");
    g.b_gather = dfs::kGatherRows;
    g.b_group = dh;
    for (size_t i = 0; i < len; ++i) {
      const int gi = static_cast<int>(std::min(i, static_cast<size_t>(sections * h - 1)));
      g.b_idx[i] = static_cast<unsigned short>((gi / h) * nunion + pos[gi % h]);
    }
    return DFS_OK;
  };
  auto gather_kcols = [&](dfs::GemmArgs& g, const std::vector<int>& pos) -> dfs_status {
    const int kb = static_cast<int>(pos.size()) * dh / 64;
    if (kb > dfs::kGemmMapMax) return fail(DFS_EUNSUPPORTED, "gather map too long");
    g.b_gather = dfs::kGatherKCols;
    for (int k = 0; k < kb; ++k) g.b_idx[k] = static_cast<unsigned short>((pos[k * 64 / dh] * dh + (k * 64) % dh) / 64);
    return DFS_OK;
  };

  // kernel arguments
  const LayerConst& C = P->lc[l];
  CUtensorMap ma, mb;
  const float scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(dh)));
  if (hd > 0) {
    const bool okb = uni ? make_map(&mb, U.wqkv.p, d, U.wqkv.rows, d, 64, dh)
                         : make_map(&mb, S.P[0].p, d, 3LL * hd, d, 64, dfs::kGemmBRows);
    if (!make_map(&ma, P->xm, d, N, d, 64, 128) || !okb) return fail(DFS_ECUDA, "tensor map (QKV) failed");
    S.g_qkv = gemm_args(P, ma, mb, N, 3 * hd, d, dfs::kEpiBias, S.P[1].p);
    S.g_qkv.out = P->qk; S.g_qkv.ldo = 2 * hd; S.g_qkv.split = 2 * hd;
    S.g_qkv.out_t = P->vt; S.g_qkv.ldt = P->vt_ld;
    if (uni && (e = gather_rows(S.g_qkv, S.pos_heads, 3, nu))) return e;
    const bool okbo = uni ? make_map(&mb, U.wo.p, U.wo.cols, d, U.wo.cols, 64, dfs::kGemmBRows)
                          : make_map(&mb, S.P[4].p, hd, d, hd, 64, dfs::kGemmBRows);
    if (!make_map(&ma, P->attn, hd, N, hd, 64, 128) || !okbo) return fail(DFS_ECUDA, "tensor map (O) failed");
    S.g_o = gemm_args(P, ma, mb, N, d, hd, dfs::kEpiGatedRes, C.bo);
    S.g_o.out = P->x1; S.g_o.ldo = d; S.g_o.out_f32 = 1; S.g_o.ldr = d; S.g_o.res_f32 = 0;
    if (!make_map_out_f32(&S.g_o.tma_out, P->x1, d, N, d)) return fail(DFS_ECUDA, "tensor map (O output) failed");
    S.g_o.out_tma = 1;
    if (uni && (e = gather_kcols(S.g_o, S.pos_heads))) return e;
    dfs::AttnArgs& A = S.a_self;
    memset(&A, 0, sizeof(A));
    // a CTA pair of the attention kernel loads 64-key halves of K and DH/2-row halves of V^T
    if (!make_map(&A.tma_q, P->qk, 2LL * hd, N, 2LL * hd, 64, 128) ||
        !make_map(&A.tma_k, P->qk, 2LL * hd, N, 2LL * hd, 64, 64) ||
        !make_map(&A.tma_vt, P->vt, N, hd, P->vt_ld, 64, dh / 2))
      return fail(DFS_ECUDA, "tensor map (attention) failed");
    A.n_q = N; A.n_kv = N; A.n_heads = S.h_s; A.q_col0 = 0; A.k_col0 = hd;
    A.out = P->attn; A.ldo = hd; A.scale_log2 = scale_log2; A.err = P->err;
  }
  if (fs > 0) {
    // union engine: the FFN panels live in the plan's per-forward scratch (same layout)
    const bf16* wup = uni ? P->ffn_up_s : S.P[5].p;
    const bf16* wdown = uni ? P->ffn_down_s : S.P[7].p;
    const long long ldf = round_up(fs, 64);  // row pitch of h and W_down: whole 128-byte lines
    if (!make_map(&ma, P->xm, d, N, d, 64, 128) || !make_map(&mb, wup, d, fs, d, 64, dfs::kGemmBRows))
      return fail(DFS_ECUDA, "tensor map (up) failed");
    S.g_up = gemm_args(P, ma, mb, N, fs, d, dfs::kEpiBiasGelu, S.P[6].p);
    S.g_up.out = P->h; S.g_up.ldo = ldf;
    if (!make_map(&ma, P->h, fs, N, ldf, 64, 128) || !make_map(&mb, wdown, fs, d, ldf, 64, dfs::kGemmBRows))
      return fail(DFS_ECUDA, "tensor map (down) failed");
    S.g_down = gemm_args(P, ma, mb, N, d, fs, dfs::kEpiGatedRes, C.bdown);
    S.g_down.ldo = d; S.g_down.out_f32 = 0; S.g_down.res = P->x1; S.g_down.ldr = d; S.g_down.res_f32 = 1;
  }
  if (c.has_cross && hcd > 0) {
    // context keys / values of this step's cross heads, once per plan
    if ((e = alloc_n(P, &S.kc, static_cast<long long>(c.ctx_len) * hcd)) ||
        (e = alloc_n(P, &S.vct, static_cast<long long>(hcd) * P->ctx_ld)))
      return e;
    if (!make_map(&ma, ctx, d, c.ctx_len, d, 64, 128) || !make_map(&mb, S.P[10].p, d, 2LL * hcd, d, 64, dfs::kGemmBRows))
      return fail(DFS_ECUDA, "tensor map (cross kv) failed");
    dfs::GemmArgs kv = gemm_args(P, ma, mb, c.ctx_len, 2 * hcd, d, dfs::kEpiBias, S.P[11].p);
    kv.out = S.kc; kv.ldo = hcd; kv.split = hcd; kv.out_t = S.vct; kv.ldt = P->ctx_ld;
    DFS_CK(dfs::launch_gemm(kv, P->num_sms, st));
    DFS_CK(dfs::launch_qk_norm_rope(S.kc, hcd, c.ctx_len, 0, hcd, nullptr, S.P[13].p, dh, c.qk_norm_mode,
                                    c.ln_eps, nullptr, st));
    const bool okq = uni ? make_map(&mb, U.cwq.p, d, U.cwq.rows, d, 64, dh)
                         : make_map(&mb, S.P[8].p, d, hcd, d, 64, dfs::kGemmBRows);
    if (!make_map(&ma, P->xm, d, N, d, 64, 128) || !okq) return fail(DFS_ECUDA, "tensor map (cross q) failed");
    S.g_cq = gemm_args(P, ma, mb, N, hcd, d, dfs::kEpiBias, S.P[9].p);
    S.g_cq.out = P->qc; S.g_cq.ldo = hcd;
    if (uni && (e = gather_rows(S.g_cq, S.pos_xheads, 1, static_cast<int>(U.xheads.size())))) return e;
    const bool oko = uni ? make_map(&mb, U.cwo.p, U.cwo.cols, d, U.cwo.cols, 64, dfs::kGemmBRows)
                         : make_map(&mb, S.P[14].p, hcd, d, hcd, 64, dfs::kGemmBRows);
    if (!make_map(&ma, P->attn, hcd, N, hcd, 64, 128) || !oko) return fail(DFS_ECUDA, "tensor map (cross o) failed");
    S.g_co = gemm_args(P, ma, mb, N, d, hcd, dfs::kEpiGatedRes, C.cbo);
    S.g_co.out = P->x1; S.g_co.ldo = d; S.g_co.out_f32 = 1; S.g_co.res = P->x1; S.g_co.ldr = d;
    S.g_co.res_f32 = 1; S.g_co.gate = nullptr;
    if (!make_map_out_f32(&S.g_co.tma_out, P->x1, d, N, d)) return fail(DFS_ECUDA, "tensor map (cross O output) failed");
    S.g_co.out_tma = 1;
    if (uni && (e = gather_kcols(S.g_co, S.pos_xheads))) return e;
    dfs::AttnArgs& A = S.a_cross;
    memset(&A, 0, sizeof(A));
    if (!make_map(&A.tma_q, P->qc, hcd, N, hcd, 64, 128) || !make_map(&A.tma_k, S.kc, hcd, c.ctx_len, hcd, 64, 64) ||
        !make_map(&A.tma_vt, S.vct, c.ctx_len, hcd, P->ctx_ld, 64, dh / 2))
      return fail(DFS_ECUDA, "tensor map (cross attention) failed");
    A.n_q = N; A.n_kv = c.ctx_len; A.n_heads = S.hc; A.q_col0 = 0; A.k_col0 = 0;
    A.out = P->attn; A.ldo = hcd; A.scale_log2 = scale_log2; A.err = P->err;
  }
  const double Nd = N, dd = d;
  S.flops = 8 * Nd * dd * dh * S.h_s + 4 * Nd * Nd * dh * S.h_s + 4 * Nd * dd * S.f_s;
  if (c.has_cross)
    S.flops += 4 * Nd * dd * dh * S.hc + 4.0 * c.ctx_len * dd * dh * S.hc + 4 * Nd * c.ctx_len * dh * S.hc;
  return DFS_OK;
}

// The layer's union super-model (Sec. 4.3): ids retained at any step (OR of the step gates;
// block gates do not enter) and, under DFS_ENGINE_UNION, the weights of those units gathered
// from the full layer once: Wqkv, Wo, W_up, W_down, cWq, cWo.
dfs_status build_union(dfs_plan* P, int l, const dfs_layer_weights& w, const dfs_masks* m, cudaStream_t st,
                       std::vector<std::vector<int>>& keep_alive) {
  const dfs_config& c = P->cfg;
  const int d = c.dim, H = c.n_heads, dh = c.head_dim, NC = c.ffn_dim / c.ffn_chunk;
  LayerUnion& U = P->lu[l];
  for (int h = 0; h < H; ++h) {
    bool any = false, anyx = false;
    for (int s = 0; s < P->T; ++s) {
      const long long base = static_cast<long long>(s) * c.n_layers + l;
      any |= m->head_gate[base * H + h] != 0;
      anyx |= !m->xhead_gate || m->xhead_gate[base * H + h] != 0;
    }
    if (any) U.heads.push_back(h);
    if (c.has_cross && anyx) U.xheads.push_back(h);
  }
  for (int k = 0; k < NC; ++k) {
    bool any = false;
    for (int s = 0; s < P->T; ++s) any |= m->ffn_gate[(static_cast<long long>(s) * c.n_layers + l) * NC + k] != 0;
    if (any) U.chunks.push_back(k);
  }
  if (!P->uni) return DFS_OK;
  const int nu = static_cast<int>(U.heads.size()), nf = static_cast<int>(U.chunks.size());
  const int nx = static_cast<int>(U.xheads.size());
  std::vector<int> rows, segs, frows, xrows, xsegs;
  for (int h : U.heads)
    for (int j = 0; j < dh; ++j) rows.push_back(h * dh + j);
  for (int h : U.heads)
    for (int j = 0; j < dh / 8; ++j) segs.push_back(h * dh / 8 + j);
  for (int k : U.chunks)
    for (int j = 0; j < c.ffn_chunk; ++j) frows.push_back(k * c.ffn_chunk + j);
  for (int h : U.xheads)
    for (int j = 0; j < dh; ++j) xrows.push_back(h * dh + j);
  for (int h : U.xheads)
    for (int j = 0; j < dh / 8; ++j) xsegs.push_back(h * dh / 8 + j);
  int *d_rows, *d_segs, *d_frows, *d_chunks, *d_xrows, *d_xsegs;
  dfs_status e;
  if ((e = upload_ints(P, rows, &d_rows, st)) || (e = upload_ints(P, segs, &d_segs, st)) ||
      (e = upload_ints(P, frows, &d_frows, st)) || (e = upload_ints(P, U.chunks, &d_chunks, st)) ||
      (e = upload_ints(P, xrows, &d_xrows, st)) || (e = upload_ints(P, xsegs, &d_xsegs, st)))
    return e;
  for (auto* v : {&rows, &segs, &frows, &xrows, &xsegs}) keep_alive.push_back(*v);
  auto mk = [&](Panel& p, long long r, long long cols) -> dfs_status {
    p.rows = r; p.cols = cols; p.ld = cols;
    return r * cols ? alloc_weights(P, &p.p, r * cols) : DFS_OK;
  };
  const long long ud = static_cast<long long>(nu) * dh, xd = static_cast<long long>(nx) * dh;
  const long long uf = static_cast<long long>(nf) * c.ffn_chunk;
  if ((e = mk(U.wqkv, 3 * ud, d)) || (e = mk(U.wo, d, ud)) || (e = mk(U.wup, uf, d)) || (e = mk(U.wdown, d, uf)))
    return e;
  if (c.has_cross && ((e = mk(U.cwq, xd, d)) || (e = mk(U.cwo, d, xd)))) return e;
  if (ud > 0) {
    const void* src[3] = {w.wq, w.wk, w.wv};
    for (int q = 0; q < 3; ++q)
      DFS_CK(dfs::launch_gather_rows(U.wqkv.p + q * ud * d, d, static_cast<const bf16*>(src[q]), d, d_rows,
                                     static_cast<int>(ud), d, st));
    DFS_CK(dfs::launch_gather_segs(U.wo.p, ud, static_cast<const bf16*>(w.wo), d, d_segs, static_cast<int>(ud / 8),
                                   d, st));
  }
  if (uf > 0) {
    DFS_CK(dfs::launch_gather_rows(U.wup.p, d, static_cast<const bf16*>(w.w_up), d, d_frows, static_cast<int>(uf),
                                   d, st));
    DFS_CK(dfs::launch_gather_segs(U.wdown.p, uf, static_cast<const bf16*>(w.w_down), c.ffn_dim, d_chunks, nf, d,
                                   st));
  }
  if (c.has_cross && xd > 0) {
    DFS_CK(dfs::launch_gather_rows(U.cwq.p, d, static_cast<const bf16*>(w.cwq), d, d_xrows, static_cast<int>(xd),
                                   d, st));
    DFS_CK(dfs::launch_gather_segs(U.cwo.p, xd, static_cast<const bf16*>(w.cwo), d, d_xsegs,
                                   static_cast<int>(xd / 8), d, st));
  }
  return DFS_OK;
}

dfs_status create_impl(dfs_plan* P, const dfs_layer_weights* layers, const void* w_t, const void* b_t,
                       const dfs_masks* m, const void* ctx, cudaStream_t st) {
  const dfs_config& c = P->cfg;
  const int d = c.dim, dh = c.head_dim;
  DFS_CK(cudaGetDevice(&P->device));
  DFS_CK(cudaDeviceGetAttribute(&P->num_sms, cudaDevAttrMultiProcessorCount, P->device));
  if (!encode_fn()) return fail(DFS_ECUDA, "cuTensorMapEncodeTiled is unavailable");
  DFS_CK(dfs::gemm_prepare());
  DFS_CK(dfs::attention_prepare());
  const long long N = P->N;
  dfs_status e;
  if ((e = alloc_n(P, &P->err, 1))) return e;
  DFS_CK(cudaMemsetAsync(P->err, 0, sizeof(int), st));

  // shared adaLN linear and per-layer constants
  if ((e = alloc_n(P, &P->w_t, 6LL * d * d)) || (e = alloc_n(P, &P->b_t, 6LL * d))) return e;
  DFS_CK(cudaMemcpyAsync(P->w_t, w_t, 12LL * d * d, cudaMemcpyDeviceToDevice, st));
  DFS_CK(cudaMemcpyAsync(P->b_t, b_t, 12LL * d, cudaMemcpyDeviceToDevice, st));
  P->lc.resize(P->L);
  for (int l = 0; l < P->L; ++l) {
    LayerConst& C = P->lc[l];
    if ((e = alloc_n(P, &C.bo, d)) || (e = alloc_n(P, &C.bdown, d)) || (e = alloc_n(P, &C.emod, 6LL * d)))
      return e;
    DFS_CK(cudaMemcpyAsync(C.bo, layers[l].bo, 2LL * d, cudaMemcpyDeviceToDevice, st));
    DFS_CK(cudaMemcpyAsync(C.bdown, layers[l].b_down, 2LL * d, cudaMemcpyDeviceToDevice, st));
    DFS_CK(cudaMemcpyAsync(C.emod, layers[l].e_mod, 12LL * d, cudaMemcpyDeviceToDevice, st));
    if (c.has_cross) {
      if ((e = alloc_n(P, &C.cbo, d)) || (e = alloc_n(P, &C.cln_w, d)) || (e = alloc_n(P, &C.cln_b, d))) return e;
      DFS_CK(cudaMemcpyAsync(C.cbo, layers[l].cbo, 2LL * d, cudaMemcpyDeviceToDevice, st));
      DFS_CK(dfs::launch_to_f32(C.cln_w, static_cast<const bf16*>(layers[l].cln_w), d, st));
      DFS_CK(dfs::launch_to_f32(C.cln_b, static_cast<const bf16*>(layers[l].cln_b), d, st));
    }
  }

  // 3D RoPE tables (angles in double, stored fp32)
  {
    const int half = dh / 2, p_hw = dh / 6, p_t = half - 2 * p_hw;
    const int G[3] = {c.grid_t, c.grid_h, c.grid_w};
    const int Pn[3] = {p_t, p_hw, p_hw};
    std::vector<float> host;
    size_t off[6];
    for (int a = 0; a < 3; ++a) {
      off[2 * a] = host.size();
      for (int pos = 0; pos < G[a]; ++pos)
        for (int j = 0; j < Pn[a]; ++j)
          host.push_back(static_cast<float>(std::cos(pos * std::pow(static_cast<double>(c.rope_theta),
                                                                    -static_cast<double>(j) / Pn[a]))));
      off[2 * a + 1] = host.size();
      for (int pos = 0; pos < G[a]; ++pos)
        for (int j = 0; j < Pn[a]; ++j)
          host.push_back(static_cast<float>(std::sin(pos * std::pow(static_cast<double>(c.rope_theta),
                                                                    -static_cast<double>(j) / Pn[a]))));
    }
    float* t;
    if ((e = alloc_n(P, &t, static_cast<long long>(host.size())))) return e;
    DFS_CK(cudaMemcpy(t, host.data(), host.size() * sizeof(float), cudaMemcpyHostToDevice));
    P->rope.cos_t = t + off[0]; P->rope.sin_t = t + off[1];
    P->rope.cos_h = t + off[2]; P->rope.sin_h = t + off[3];
    P->rope.cos_w = t + off[4]; P->rope.sin_w = t + off[5];
    P->rope.grid_h = c.grid_h; P->rope.grid_w = c.grid_w;
    P->rope.p_t = p_t; P->rope.p_h = p_hw; P->rope.p_w = p_hw;
  }

  // workspace for N tokens, sized by the largest step structure
  int hmax = 0, fmax = 0, hcmax = 0;
  {
    const int H = c.n_heads, NC = c.ffn_dim / c.ffn_chunk;
    for (long long i = 0; i < static_cast<long long>(P->T) * P->L; ++i) {
      int hs = 0, ch = 0, xh = 0;
      for (int h = 0; h < H; ++h) hs += m->head_gate[i * H + h];
      for (int k = 0; k < NC; ++k) ch += m->ffn_gate[i * NC + k];
      if (c.has_cross)
        for (int h = 0; h < H; ++h) xh += m->xhead_gate ? m->xhead_gate[i * H + h] : 1;
      hmax = std::max(hmax, hs);
      fmax = std::max(fmax, ch * c.ffn_chunk);
      hcmax = std::max(hcmax, xh);
    }
  }
  P->vt_ld = round_up(N, 64);
  P->ctx_ld = round_up(c.has_cross ? c.ctx_len : 8, 64);
  const long long amax = static_cast<long long>(std::max(hmax, hcmax)) * dh;
  if ((e = alloc_n(P, &P->mod, 6LL * d)) || (e = alloc_n(P, &P->mod_base, 6LL * d * P->T)) ||
      (e = alloc_n(P, &P->xm, N * d)) || (e = alloc_n(P, &P->qk, N * 2 * hmax * dh)) ||
      (e = alloc_n(P, &P->vt, static_cast<long long>(hmax) * dh * P->vt_ld)) || (e = alloc_n(P, &P->attn, N * amax)) ||
      (e = alloc_n(P, &P->x1, N * d)) || (e = alloc_n(P, &P->h, N * round_up(fmax, 64))) ||
      (e = alloc_n(P, &P->qc, N * static_cast<long long>(hcmax) * dh)) || (e = alloc_n(P, &P->act[0], N * d)) ||
      (e = alloc_n(P, &P->act[1], N * d)) || (e = alloc_n(P, &P->stage_x, N * d)) ||
      (e = alloc_n(P, &P->stage_out, N * d)) || (e = alloc_n(P, &P->stage_t, d)))
    return e;
  if (hmax > 0) DFS_CK(cudaMemsetAsync(P->vt, 0, sizeof(bf16) * hmax * dh * P->vt_ld, st));
  if (P->uni && ((e = alloc_n(P, &P->ffn_up_s, static_cast<long long>(fmax) * d)) ||
                 (e = alloc_n(P, &P->ffn_down_s, round_up(fmax, 64) * d))))
    return e;

  // per layer: the union super-model; per (step, layer): index tables, compacted panels
  // (or gather maps into the union), kernel arguments
  std::vector<std::vector<int>> keep_alive;  // host index lists stay valid until the sync below
  P->lu.resize(P->L);
  for (int l = 0; l < P->L; ++l)
    if ((e = build_union(P, l, layers[l], m, st, keep_alive))) return e;
  P->sl.resize(static_cast<size_t>(P->T) * P->L);
  for (int s = 0; s < P->T; ++s)
    for (int l = 0; l < P->L; ++l)
      if ((e = build_step_layer(P, s, l, layers[l], m, ctx, st, keep_alive))) return e;
  DFS_CK(cudaStreamSynchronize(st));
  // buffers needed only while the plan was built (union engine: the context K/V weights)
  for (void* t : P->temps) cudaFree(t);
  P->temps.clear();
  for (StepLayer& S : P->sl) S.P[10].p = P->uni ? nullptr : S.P[10].p;
  int herr = 0;
  DFS_CK(cudaMemcpy(&herr, P->err, sizeof(int), cudaMemcpyDeviceToHost));
  if (herr) return fail(DFS_ETIMEOUT, "a kernel gave up waiting during plan creation");
  return DFS_OK;
}

// ------------------------------------------------------------------ forward

// Union engine: the step's FFN panels gathered from the layer's union (K1) into the plan's
// scratch, read by the FFN projections right after (the paper's gather through I_t).
// `profiled` = false launches without the per-kernel event bracket (the allocation-free
// forward creates no events).
dfs_status union_ffn_gather(dfs_plan* P, const StepLayer& S, int l, cudaStream_t st, bool profiled = true) {
  if (!P->uni || S.f_s == 0) return DFS_OK;
  const LayerUnion& U = P->lu[l];
  const int d = P->cfg.dim, fs = S.f_s;
  if (profiled) {
    DFS_LAUNCH(DFS_K_GATHER, dfs::launch_gather_rows(P->ffn_up_s, d, U.wup.p, d, S.up_rows_u, fs, d, st));
    DFS_LAUNCH(DFS_K_GATHER, dfs::launch_gather_segs(P->ffn_down_s, round_up(fs, 64), U.wdown.p, U.wdown.ld,
                                                     S.down_segs_u, fs / P->cfg.ffn_chunk, d, st));
  } else {
    DFS_CK(dfs::launch_gather_rows(P->ffn_up_s, d, U.wup.p, d, S.up_rows_u, fs, d, st));
    DFS_CK(dfs::launch_gather_segs(P->ffn_down_s, round_up(fs, 64), U.wdown.p, U.wdown.ld, S.down_segs_u,
                                   fs / P->cfg.ffn_chunk, d, st));
  }
  return DFS_OK;
}

dfs_status forward_impl(dfs_plan* P, int s, int l, const bf16* x, bf16* out, cudaStream_t st) {
  // P->mod holds this layer's six modulation vectors
  const dfs_config& c = P->cfg;
  const int d = c.dim, dh = c.head_dim;
  const int N = P->N;
  StepLayer& S = P->sl[s * P->L + l];
  const LayerConst& C = P->lc[l];
  const float* shift_a = P->mod;
  const float* scale_a = P->mod + d;
  const float* gate_a = P->mod + 2 * d;
  const float* shift_f = P->mod + 3 * d;
  const float* scale_f = P->mod + 4 * d;
  const float* gate_f = P->mod + 5 * d;
  P->last_step = s;
  P->last_layer = l;

  DFS_LAUNCH(DFS_K_ADALN, dfs::launch_row_norm(P->xm, x, 0, N, d, scale_a, 1.f, shift_a, c.ln_eps, st));
  if (S.h_s > 0) {
    const int hd = S.h_s * dh;
    DFS_LAUNCH(DFS_K_GEMM_QKV, dfs::launch_gemm(S.g_qkv, P->num_sms, st));
    DFS_LAUNCH(DFS_K_QK_NORM_ROPE, dfs::launch_qk_norm_rope(P->qk, 2LL * hd, N, hd, hd, S.P[2].p, S.P[3].p, dh, c.qk_norm_mode, c.ln_eps,
                                    &P->rope, st));
    DFS_LAUNCH(DFS_K_ATTENTION, dfs::launch_attention(S.a_self, dh, st));
    dfs::GemmArgs g = S.g_o;
    g.res = x;
    g.gate = gate_a;
    DFS_LAUNCH(DFS_K_GEMM_O, dfs::launch_gemm(g, P->num_sms, st));
  } else {
    DFS_LAUNCH(DFS_K_OTHER, dfs::launch_bias_residual(P->x1, 1, x, 0, gate_a, C.bo, N, d, st));
  }
  if (c.has_cross) {
    DFS_LAUNCH(DFS_K_CROSS, dfs::launch_row_norm(P->xm, P->x1, 1, N, d, C.cln_w, 0.f, C.cln_b, c.ln_eps, st));
    if (S.hc > 0) {
      const int hcd = S.hc * dh;
      DFS_LAUNCH(DFS_K_CROSS, dfs::launch_gemm(S.g_cq, P->num_sms, st));
      DFS_LAUNCH(DFS_K_CROSS, dfs::launch_qk_norm_rope(P->qc, hcd, N, hcd, 0, S.P[12].p, nullptr, dh, c.qk_norm_mode, c.ln_eps,
                                      nullptr, st));
      DFS_LAUNCH(DFS_K_CROSS, dfs::launch_attention(S.a_cross, dh, st));
      DFS_LAUNCH(DFS_K_CROSS, dfs::launch_gemm(S.g_co, P->num_sms, st));
    } else {
      DFS_LAUNCH(DFS_K_CROSS, dfs::launch_bias_residual(P->x1, 1, P->x1, 1, nullptr, C.cbo, N, d, st));
    }
  }
  DFS_LAUNCH(DFS_K_ADALN, dfs::launch_row_norm(P->xm, P->x1, 1, N, d, scale_f, 1.f, shift_f, c.ln_eps, st));
  if (S.f_s > 0) {
    dfs_status e = union_ffn_gather(P, S, l, st);
    if (e) return e;
    DFS_LAUNCH(DFS_K_GEMM_UP, dfs::launch_gemm(S.g_up, P->num_sms, st));
    dfs::GemmArgs g = S.g_down;
    g.out = out;
    g.gate = gate_f;
    DFS_LAUNCH(DFS_K_GEMM_DOWN, dfs::launch_gemm(g, P->num_sms, st));
  } else {
    DFS_LAUNCH(DFS_K_OTHER, dfs::launch_bias_residual(out, 0, P->x1, 1, gate_f, C.bdown, N, d, st));
  }
  return DFS_OK;
}

dfs_status check_forward_args(dfs_plan* P, int step, int layer, const void* x, const void* t_emb, void* out,
                              bool device = true) {
  if (!P) return fail(DFS_EINVAL, "plan is NULL");
  if (!x || !t_emb || !out) return fail(DFS_EINVAL, "NULL x, t_emb or out");
  if (x == out) return fail(DFS_EINVAL, "x and out must not alias");
  if (device && (!aligned16(x) || !aligned16(t_emb) || !aligned16(out)))
    return fail(DFS_EINVAL, "x, t_emb and out must be 16-byte aligned");
  if (step < 0 || step >= P->T) return fail(DFS_EINVAL, "step %d out of range [0, %d)", step, P->T);
  if (layer < 0 || layer >= P->L) return fail(DFS_EINVAL, "layer %d out of range [0, %d)", layer, P->L);
  return DFS_OK;
}

dfs_status block_layer(dfs_plan* P, int step, int layer, const bf16* x, const bf16* t_emb, bf16* out,
                       cudaStream_t st) {
  const int d = P->cfg.dim;
  if (!P->block_gate[static_cast<size_t>(step) * P->L + layer]) {
    DFS_LAUNCH(DFS_K_OTHER, cudaMemcpyAsync(out, x, sizeof(bf16) * P->N * d, cudaMemcpyDeviceToDevice, st));
    return DFS_OK;
  }
  DFS_LAUNCH(DFS_K_MODULATION, dfs::launch_modulation(P->mod, P->w_t, P->b_t, P->lc[layer].emod, t_emb, 6 * d, d, st));
  return forward_impl(P, step, layer, x, out, st);
}

// Drops the cached device address of the allocation-free forward's static array for
// `device` (defined with the array below).
void noalloc_forget_device(int device);

}  // namespace

// ------------------------------------------------------------------ C ABI

extern "C" {

dfs_status dfs_plan_create(const dfs_config* cfg, const dfs_layer_weights* layers, const void* w_t,
                           const void* b_t, const dfs_masks* masks, const void* ctx, void* stream, dfs_plan** out) {
  g_last_error.clear();
  dfs_status e = validate(cfg, layers, w_t, b_t, masks, ctx, out);
  if (e) return e;
  dfs_plan* P = new (std::nothrow) dfs_plan();
  if (!P) return fail(DFS_ENOMEM, "host allocation failed");
  P->cfg = *cfg;
  P->uni = cfg->engine == DFS_ENGINE_UNION;
  P->T = cfg->n_steps;
  P->L = cfg->n_layers;
  P->N = cfg->grid_t * cfg->grid_h * cfg->grid_w;
  P->block_gate.assign(masks->block_gate, masks->block_gate + static_cast<size_t>(P->T) * P->L);
  if (const char* f = getenv("DFS_FAULT_ALLOC")) P->fault_alloc = atoi(f);
  if (const char* f = getenv("DFS_FAULT_LAUNCH")) P->fault_launch = atoll(f);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  e = create_impl(P, layers, w_t, b_t, masks, ctx, st);
  if (e) {
    cudaStreamSynchronize(st);
    (void)cudaGetLastError();
    free_plan(P);
    return e;
  }
  // A plan exists only in a context created after the device's last reset, so the next
  // allocation-free call looks the static array's address up again in this context.
  noalloc_forget_device(P->device);
  *out = P;
  return DFS_OK;
}

dfs_status dfs_block_forward_layer(dfs_plan* plan, int step, int layer, const void* x, const void* t_emb,
                                   void* out, void* stream) {
  dfs_status e = check_forward_args(plan, step, layer, x, t_emb, out);
  if (e) return e;
  return block_layer(plan, step, layer, static_cast<const bf16*>(x), static_cast<const bf16*>(t_emb),
                     static_cast<bf16*>(out), static_cast<cudaStream_t>(stream));
}

dfs_status dfs_block_forward(dfs_plan* plan, int step, const void* x, const void* t_emb, void* out, void* stream) {
  return dfs_block_forward_layer(plan, step, 0, x, t_emb, out, stream);
}

namespace {

// Makes `st` wait for every copy the staging ring has in flight.
dfs_status ring_join(dfs_plan* P, cudaStream_t st) {
  dfs_plan::HostRing& R = P->ring;
  if (!R.ready) return DFS_OK;
  for (int b = 0; b < 2; ++b) {
    DFS_CK(cudaStreamWaitEvent(st, R.loaded[b], 0));
    DFS_CK(cudaStreamWaitEvent(st, R.drained[b], 0));
  }
  return DFS_OK;
}

// First use of the ring: the second slot's device buffers, two copy streams, six events.
dfs_status ring_init(dfs_plan* P) {
  dfs_plan::HostRing& R = P->ring;
  if (R.ready) return DFS_OK;
  const long long n = static_cast<long long>(P->N) * P->cfg.dim;
  R.x[0] = P->stage_x;
  R.out[0] = P->stage_out;
  R.t[0] = P->stage_t;
  dfs_status e;
  if (!R.x[1] && ((e = alloc_n(P, &R.x[1], n)) || (e = alloc_n(P, &R.out[1], n)) ||
                  (e = alloc_n(P, &R.t[1], P->cfg.dim))))
    return e;
  if (!R.h2d) DFS_CK(cudaStreamCreateWithFlags(&R.h2d, cudaStreamNonBlocking));
  if (!R.d2h) DFS_CK(cudaStreamCreateWithFlags(&R.d2h, cudaStreamNonBlocking));
  for (int b = 0; b < 2; ++b)
    for (cudaEvent_t* ev : {&R.loaded[b], &R.computed[b], &R.drained[b]})
      if (!*ev) DFS_CK(cudaEventCreateWithFlags(ev, cudaEventDisableTiming));
  R.ready = true;
  return DFS_OK;
}

}  // namespace

dfs_status dfs_block_forward_host_async(dfs_plan* plan, int step, int layer, const void* x_host,
                                        const void* t_emb_host, void* out_host, void* stream) {
  dfs_status e = check_forward_args(plan, step, layer, x_host, t_emb_host, out_host, false);
  if (e) return e;
  if ((e = ring_init(plan))) return e;
  dfs_plan::HostRing& R = plan->ring;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int b = R.next;
  const size_t bytes = sizeof(bf16) * plan->N * plan->cfg.dim;
  // inputs: into slot b once the forward two calls back has finished reading it
  DFS_CK(cudaStreamWaitEvent(R.h2d, R.computed[b], 0));
  DFS_CK(cudaMemcpyAsync(R.x[b], x_host, bytes, cudaMemcpyHostToDevice, R.h2d));
  DFS_CK(cudaMemcpyAsync(R.t[b], t_emb_host, sizeof(bf16) * plan->cfg.dim, cudaMemcpyHostToDevice, R.h2d));
  DFS_CK(cudaEventRecord(R.loaded[b], R.h2d));
  // forward on the caller's stream once the inputs are in and slot b's last output is out
  DFS_CK(cudaStreamWaitEvent(st, R.loaded[b], 0));
  DFS_CK(cudaStreamWaitEvent(st, R.drained[b], 0));
  e = block_layer(plan, step, layer, R.x[b], R.t[b], R.out[b], st);
  // recorded even after a failed launch, so that the slot's next input copy waits for
  // whatever part of this forward did reach the stream (the slot is then reused next call)
  DFS_CK(cudaEventRecord(R.computed[b], st));
  if (e) return e;
  // output: back to the host while the caller's stream moves on
  DFS_CK(cudaStreamWaitEvent(R.d2h, R.computed[b], 0));
  DFS_CK(cudaMemcpyAsync(out_host, R.out[b], bytes, cudaMemcpyDeviceToHost, R.d2h));
  DFS_CK(cudaEventRecord(R.drained[b], R.d2h));
  R.next = b ^ 1;
  return DFS_OK;
}

dfs_status dfs_block_forward_host(dfs_plan* plan, int step, int layer, const void* x_host, const void* t_emb_host,
                                  void* out_host, void* stream) {
  dfs_status e = check_forward_args(plan, step, layer, x_host, t_emb_host, out_host, false);
  if (e) return e;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // slot 0 of the asynchronous ring may still be in use by earlier asynchronous calls
  if ((e = ring_join(plan, st))) return e;
  const size_t bytes = sizeof(bf16) * plan->N * plan->cfg.dim;
  DFS_CK(cudaMemcpyAsync(plan->stage_x, x_host, bytes, cudaMemcpyHostToDevice, st));
  DFS_CK(cudaMemcpyAsync(plan->stage_t, t_emb_host, sizeof(bf16) * plan->cfg.dim, cudaMemcpyHostToDevice, st));
  e = block_layer(plan, step, layer, plan->stage_x, plan->stage_t, plan->stage_out, st);
  if (e) return e;
  DFS_CK(cudaMemcpyAsync(out_host, plan->stage_out, bytes, cudaMemcpyDeviceToHost, st));
  DFS_CK(cudaStreamSynchronize(st));
  return DFS_OK;
}

dfs_status dfs_denoise(dfs_plan* P, void* latents, int n_steps, const void* t_embs, void* stream) {
  if (!P || !latents || !t_embs) return fail(DFS_EINVAL, "NULL plan, latents or t_embs");
  if (!aligned16(latents) || !aligned16(t_embs)) return fail(DFS_EINVAL, "latents and t_embs must be 16-byte aligned");
  if (n_steps < 1 || n_steps > P->T) return fail(DFS_EINVAL, "n_steps must be in 1..%d", P->T);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int d = P->cfg.dim;
  bf16* lat = static_cast<bf16*>(latents);
  const bf16* temb = static_cast<const bf16*>(t_embs);
  for (int s = 0; s < n_steps; ++s) {
    float* base = P->mod_base + 6LL * d * s;
    DFS_LAUNCH(DFS_K_MODULATION,
               dfs::launch_modulation(base, P->w_t, P->b_t, nullptr, temb + static_cast<long long>(s) * d, 6 * d, d, st));
    const bf16* cur = lat;
    int ping = 0;
    for (int l = 0; l < P->L; ++l) {
      if (!P->block_gate[static_cast<size_t>(s) * P->L + l]) continue;
      DFS_LAUNCH(DFS_K_MODULATION, dfs::launch_add_table(P->mod, base, P->lc[l].emod, 6 * d, st));
      bf16* dst = P->act[ping];
      dfs_status e = forward_impl(P, s, l, cur, dst, st);
      if (e) return e;
      cur = dst;
      ping ^= 1;
    }
    DFS_LAUNCH(DFS_K_OTHER, dfs::launch_euler(lat, cur, 1.f / P->cfg.n_steps, static_cast<long long>(P->N) * d, st));
  }
  return DFS_OK;
}

// ------------------------------------------------------------------ model around the blocks

}  // extern "C"

namespace {

// One pass of the model on `lat` at step s with host timestep t: the timestep MLP, patch
// embedding, every layer of step s, the head; leaves the velocity token rows in m_vtok.
dfs_status model_pass(dfs_plan* P, int s, const bf16* lat, float t, cudaStream_t st) {
  const dfs_config& c = P->cfg;
  const int d = c.dim, C = P->mC;
  DFS_LAUNCH(DFS_K_MODEL, dfs::launch_timestep_freq(P->m_freq, static_cast<double>(t), P->mD, st));
  DFS_LAUNCH(DFS_K_MODEL, dfs::launch_gemv(P->m_h1, nullptr, P->m_t_w1, P->m_t_b1, P->m_freq, d, P->mD, 0, st));
  DFS_LAUNCH(DFS_K_MODEL, dfs::launch_gemv(P->m_temb_f, P->m_temb, P->m_t_w2, P->m_t_b2, P->m_h1, d, d, 1, st));
  DFS_LAUNCH(DFS_K_MODEL, dfs::launch_patchify(P->m_tok, lat, C, c.grid_t, c.grid_h, c.grid_w, st));
  DFS_LAUNCH(DFS_K_MODEL, dfs::launch_gemm(P->g_embed, P->num_sms, st));
  float* base = P->mod_base + 6LL * d * s;
  DFS_LAUNCH(DFS_K_MODULATION, dfs::launch_modulation(base, P->w_t, P->b_t, nullptr, P->m_temb, 6 * d, d, st));
  const bf16* cur = P->m_x0;
  int ping = 0;
  for (int l = 0; l < P->L; ++l) {
    if (!P->block_gate[static_cast<size_t>(s) * P->L + l]) continue;
    DFS_LAUNCH(DFS_K_MODULATION, dfs::launch_add_table(P->mod, base, P->lc[l].emod, 6 * d, st));
    bf16* dst = P->act[ping];
    dfs_status e = forward_impl(P, s, l, cur, dst, st);
    if (e) return e;
    cur = dst;
    ping ^= 1;
  }
  // head: (shift, scale) = head_mod + t_emb; LN + modulate into xm; v tokens = xm head_w^T + b
  DFS_LAUNCH(DFS_K_MODEL, dfs::launch_add_table(P->m_hm, P->m_temb_f, P->m_head_mod, d, st));
  DFS_LAUNCH(DFS_K_MODEL, dfs::launch_add_table(P->m_hm + d, P->m_temb_f, P->m_head_mod + d, d, st));
  DFS_LAUNCH(DFS_K_MODEL, dfs::launch_row_norm(P->xm, cur, 0, P->N, d, P->m_hm + d, 1.f, P->m_hm, c.ln_eps, st));
  DFS_LAUNCH(DFS_K_MODEL, dfs::launch_gemm(P->g_head, P->num_sms, st));
  return DFS_OK;
}

}  // namespace

extern "C" {

dfs_status dfs_model_attach(dfs_plan* P, const dfs_model_weights* w, void* stream) {
  if (!P || !w) return fail(DFS_EINVAL, "NULL plan or weights");
  const void* req[] = {w->patch_w, w->patch_b, w->t_w1, w->t_b1, w->t_w2, w->t_b2, w->head_mod, w->head_w, w->head_b};
  for (const void* q : req) {
    if (!q) return fail(DFS_EINVAL, "NULL model weight pointer");
    if (!aligned16(q)) return fail(DFS_EINVAL, "model weight pointers must be 16-byte aligned");
  }
  if (w->in_channels < 2 || w->in_channels % 2 != 0 || w->in_channels > 1024)
    return fail(DFS_EINVAL, "in_channels must be even, 2..1024");
  if (w->freq_dim < 8 || w->freq_dim % 8 != 0 || w->freq_dim > 8192)
    return fail(DFS_EINVAL, "freq_dim must be a multiple of 8 in 8..8192");
  if (P->has_model) return fail(DFS_EUNSUPPORTED, "a model is already attached to this plan");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const long long d = P->cfg.dim, C = w->in_channels, D = w->freq_dim, N = P->N, p4 = 4 * C;
  P->mC = static_cast<int>(C);
  P->mD = static_cast<int>(D);
  dfs_status e;
  struct Cp { bf16** dst; const void* src; long long n; };
  const Cp cps[] = {{&P->m_patch_w, w->patch_w, d * p4}, {&P->m_patch_b, w->patch_b, d}, {&P->m_t_w1, w->t_w1, d * D},
                    {&P->m_t_b1, w->t_b1, d}, {&P->m_t_w2, w->t_w2, d * d}, {&P->m_t_b2, w->t_b2, d},
                    {&P->m_head_mod, w->head_mod, 2 * d}, {&P->m_head_w, w->head_w, p4 * d},
                    {&P->m_head_b, w->head_b, p4}};
  for (const Cp& q : cps) {
    if ((e = alloc_weights(P, q.dst, q.n))) return e;
    DFS_CK(cudaMemcpyAsync(*q.dst, q.src, 2 * q.n, cudaMemcpyDeviceToDevice, st));
  }
  if ((e = alloc_n(P, &P->m_tok, N * p4)) || (e = alloc_n(P, &P->m_x0, N * d)) || (e = alloc_n(P, &P->m_vtok, N * p4)) ||
      (e = alloc_n(P, &P->m_temb, d)) || (e = alloc_n(P, &P->m_freq, D)) || (e = alloc_n(P, &P->m_h1, d)) ||
      (e = alloc_n(P, &P->m_temb_f, d)) || (e = alloc_n(P, &P->m_hm, 2 * d)))
    return e;
  CUtensorMap ma, mb;
  if (!make_map(&ma, P->m_tok, p4, N, p4, 64, 128) || !make_map(&mb, P->m_patch_w, p4, d, p4, 64, dfs::kGemmBRows))
    return fail(DFS_ECUDA, "tensor map (patch embedding) failed");
  P->g_embed = gemm_args(P, ma, mb, static_cast<int>(N), static_cast<int>(d), static_cast<int>(p4), dfs::kEpiBias,
                         P->m_patch_b);
  P->g_embed.out = P->m_x0; P->g_embed.ldo = d;
  if (!make_map(&ma, P->xm, d, N, d, 64, 128) || !make_map(&mb, P->m_head_w, d, p4, d, 64, dfs::kGemmBRows))
    return fail(DFS_ECUDA, "tensor map (head) failed");
  P->g_head = gemm_args(P, ma, mb, static_cast<int>(N), static_cast<int>(p4), static_cast<int>(d), dfs::kEpiBias,
                        P->m_head_b);
  P->g_head.out = P->m_vtok; P->g_head.ldo = p4;
  DFS_CK(cudaStreamSynchronize(st));
  P->has_model = true;
  return DFS_OK;
}

dfs_status dfs_model_forward(dfs_plan* P, int step, const void* latent, float t, void* v_out, void* stream) {
  if (!P || !latent || !v_out) return fail(DFS_EINVAL, "NULL plan, latent or v_out");
  if (!aligned16(latent) || !aligned16(v_out)) return fail(DFS_EINVAL, "latent and v_out must be 16-byte aligned");
  if (!P->has_model) return fail(DFS_EINVAL, "no model attached (dfs_model_attach)");
  if (latent == v_out) return fail(DFS_EINVAL, "latent and v_out must not alias");
  if (step < 0 || step >= P->T) return fail(DFS_EINVAL, "step %d out of range [0, %d)", step, P->T);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  dfs_status e = model_pass(P, step, static_cast<const bf16*>(latent), t, st);
  if (e) return e;
  const dfs_config& c = P->cfg;
  DFS_LAUNCH(DFS_K_MODEL, dfs::launch_unpatchify(static_cast<bf16*>(v_out), nullptr, P->m_vtok, 1.f, P->mC, c.grid_t,
                                                 c.grid_h, c.grid_w, st));
  return DFS_OK;
}

dfs_status dfs_model_denoise(dfs_plan* P, void* latent, int n_steps, const float* timesteps, void* stream) {
  if (!P || !latent || !timesteps) return fail(DFS_EINVAL, "NULL plan, latent or timesteps");
  if (!aligned16(latent)) return fail(DFS_EINVAL, "latent must be 16-byte aligned");
  if (!P->has_model) return fail(DFS_EINVAL, "no model attached (dfs_model_attach)");
  if (n_steps < 1 || n_steps > P->T) return fail(DFS_EINVAL, "n_steps must be in 1..%d", P->T);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const dfs_config& c = P->cfg;
  bf16* lat = static_cast<bf16*>(latent);
  for (int s = 0; s < n_steps; ++s) {
    dfs_status e = model_pass(P, s, lat, timesteps[s], st);
    if (e) return e;
    DFS_LAUNCH(DFS_K_MODEL, dfs::launch_unpatchify(lat, lat, P->m_vtok, 1.f / c.n_steps, P->mC, c.grid_t, c.grid_h,
                                                   c.grid_w, st));
  }
  return DFS_OK;
}

dfs_status dfs_plan_indices(const dfs_plan* P, int step, int layer, int kind, int32_t* out, int* count) {
  if (!P || !count) return fail(DFS_EINVAL, "NULL plan or count");
  if (step < 0 || step >= P->T || layer < 0 || layer >= P->L) return fail(DFS_EINVAL, "step/layer out of range");
  const StepLayer& S = P->sl[step * P->L + layer];
  const LayerUnion& U = P->lu[layer];
  // kinds 0..2 the step's ids, 3..5 the union's ids, 6..8 the step's positions in the union
  const std::vector<int>* lists[9] = {&S.heads,     &S.chunks,     &S.xheads,     &U.heads,     &U.chunks,
                                      &U.xheads,    &S.pos_heads,  &S.pos_chunks, &S.pos_xheads};
  if (kind < 0 || kind > 8) return fail(DFS_EINVAL, "kind must be in 0..8");
  const std::vector<int>* v = lists[kind];
  *count = static_cast<int>(v->size());
  if (out)
    for (size_t i = 0; i < v->size(); ++i) out[i] = (*v)[i];
  return DFS_OK;
}

dfs_status dfs_plan_panel(const dfs_plan* P, int step, int layer, int which, const void** dev, int64_t* rows,
                          int64_t* cols, int64_t* ld) {
  if (!P || !dev || !rows || !cols || !ld) return fail(DFS_EINVAL, "NULL argument");
  if (step < 0 || step >= P->T || layer < 0 || layer >= P->L) return fail(DFS_EINVAL, "step/layer out of range");
  if (which < 0 || which > 14 || (which > 7 && !P->cfg.has_cross)) return fail(DFS_EINVAL, "bad panel id");
  const Panel& p = P->sl[step * P->L + layer].P[which];
  *dev = p.p; *rows = p.rows; *cols = p.cols; *ld = p.ld;
  return DFS_OK;
}

dfs_status dfs_plan_union_panel(const dfs_plan* P, int layer, int which, const void** dev, int64_t* rows,
                                int64_t* cols, int64_t* ld) {
  if (!P || !dev || !rows || !cols || !ld) return fail(DFS_EINVAL, "NULL argument");
  if (layer < 0 || layer >= P->L) return fail(DFS_EINVAL, "layer out of range");
  if (which < 0 || which > 5 || (which > 3 && !P->cfg.has_cross)) return fail(DFS_EINVAL, "bad union panel id");
  if (!P->uni) return fail(DFS_EUNSUPPORTED, "the plan does not use DFS_ENGINE_UNION");
  const LayerUnion& U = P->lu[layer];
  const Panel* ps[6] = {&U.wqkv, &U.wo, &U.wup, &U.wdown, &U.cwq, &U.cwo};
  const Panel& p = *ps[which];
  *dev = p.p; *rows = p.rows; *cols = p.cols; *ld = p.ld;
  return DFS_OK;
}

dfs_status dfs_plan_memory(const dfs_plan* P, int64_t* weight_bytes, int64_t* device_bytes) {
  if (!P || !weight_bytes || !device_bytes) return fail(DFS_EINVAL, "NULL argument");
  *weight_bytes = P->bytes_weights;
  *device_bytes = P->bytes_total;
  return DFS_OK;
}

dfs_status dfs_plan_flops(const dfs_plan* P, int step, int layer, double* flops) {
  if (!P || !flops) return fail(DFS_EINVAL, "NULL argument");
  if (step < 0 || step >= P->T || layer < 0 || layer >= P->L) return fail(DFS_EINVAL, "step/layer out of range");
  *flops = P->block_gate[static_cast<size_t>(step) * P->L + layer] ? P->sl[step * P->L + layer].flops : 0.0;
  return DFS_OK;
}

dfs_status dfs_plan_workspace(const dfs_plan* P, int which, void** dev, int64_t* rows, int64_t* cols, int64_t* ld,
                              int* dtype) {
  if (!P || !dev || !rows || !cols || !ld || !dtype) return fail(DFS_EINVAL, "NULL argument");
  const int s = P->last_step < 0 ? 0 : P->last_step, l = P->last_layer < 0 ? 0 : P->last_layer;
  const StepLayer& S = P->sl[s * P->L + l];
  const long long N = P->N, d = P->cfg.dim, hd = static_cast<long long>(S.h_s) * P->cfg.head_dim;
  *dtype = 0;
  switch (which) {
    case 0: *dev = P->xm; *rows = N; *cols = d; *ld = d; break;
    case 1: *dev = P->qk; *rows = N; *cols = 2 * hd; *ld = 2 * hd; break;
    case 2: *dev = P->vt; *rows = hd; *cols = N; *ld = P->vt_ld; break;
    case 3: *dev = P->attn; *rows = N; *cols = hd; *ld = hd; break;
    case 4: *dev = P->x1; *rows = N; *cols = d; *ld = d; *dtype = 1; break;
    case 5: *dev = P->h; *rows = N; *cols = S.f_s; *ld = round_up(S.f_s, 64); break;
    case 6: *dev = P->mod; *rows = 6; *cols = d; *ld = d; *dtype = 1; break;
    default: return fail(DFS_EINVAL, "bad workspace id");
  }
  return DFS_OK;
}

dfs_status dfs_plan_sync(dfs_plan* P, void* stream) {
  if (!P) return fail(DFS_EINVAL, "plan is NULL");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  dfs_status e = ring_join(P, st);
  if (e) return e;
  DFS_CK(cudaStreamSynchronize(st));
  int herr = 0;
  DFS_CK(cudaMemcpy(&herr, P->err, sizeof(int), cudaMemcpyDeviceToHost));
  if (herr) {
    DFS_CK(cudaMemset(P->err, 0, sizeof(int)));
    return fail(DFS_ETIMEOUT, "a kernel gave up on a bounded wait (error word %d)", herr);
  }
  return DFS_OK;
}

dfs_status dfs_selftest_wait_timeout(dfs_plan* P, void* stream) {
  if (!P) return fail(DFS_EINVAL, "plan is NULL");
  DFS_CK(dfs::launch_wait_selftest(P->err, static_cast<cudaStream_t>(stream)));
  return DFS_OK;
}

dfs_status dfs_plan_profile(dfs_plan* P, int enable) {
  if (!P) return fail(DFS_EINVAL, "plan is NULL");
  if (enable) {
    P->ev_used = 0;
    for (long long& n : P->launches) n = 0;
  }
  P->prof_on = enable != 0;
  return DFS_OK;
}

dfs_status dfs_plan_profile_read(dfs_plan* P, int kind, double* total_ms, int64_t* launches) {
  if (!P || !total_ms || !launches) return fail(DFS_EINVAL, "NULL argument");
  if (kind < 0 || kind >= DFS_K_COUNT) return fail(DFS_EINVAL, "bad kernel kind");
  double t = 0.0;
  for (size_t i = 0; i < P->ev_used; ++i) {
    if (P->ev_kind[i] != kind) continue;
    DFS_CK(cudaEventSynchronize(P->ev[2 * i + 1]));
    float ms = 0.f;
    DFS_CK(cudaEventElapsedTime(&ms, P->ev[2 * i], P->ev[2 * i + 1]));
    t += ms;
  }
  *total_ms = t;
  *launches = P->launches[kind];
  return DFS_OK;
}

dfs_status dfs_gates_from_soft_masks(int kind, int n_rows, int n_units, int unit_size, const float* m, uint8_t* g) {
  if (!m || !g) return fail(DFS_EINVAL, "NULL m or g");
  if (n_rows < 0 || n_units < 0 || unit_size < 1) return fail(DFS_EINVAL, "bad sizes");
  if (kind != 1 && unit_size != 1) return fail(DFS_EINVAL, "unit_size must be 1 for block and FFN gates");
  if (kind < 0 || kind > 2) return fail(DFS_EINVAL, "kind must be 0, 1 or 2");
  for (long long r = 0; r < n_rows; ++r)
    for (long long u = 0; u < n_units; ++u) {
      const float* p = m + (r * n_units + u) * unit_size;
      double sum = 0.0;
      for (int i = 0; i < unit_size; ++i) sum += static_cast<double>(p[i]);
      g[r * n_units + u] = (sum / unit_size > 0.0) ? 1 : 0;
    }
  return DFS_OK;
}

void dfs_plan_destroy(dfs_plan* plan) {
  if (!plan) return;
  cudaDeviceSynchronize();
  free_plan(plan);
}

const char* dfs_last_error(void) { return g_last_error.c_str(); }

}  // extern "C"

// ------------------------------------------------------------------ forward without allocation
//
// dfs_block_forward_noalloc runs the same kernels as dfs_block_forward, but its
// activation workspace (modulation vector, normalised activations, q/k, V^T, attention
// output, fp32 residual, FFN hidden) lives in one file-scope device array instead of
// memory the plan allocated.  It is meant for callers that must not allocate device
// memory at forward time: for example a host application that owns all device memory
// through its own pool and budget (a cudaMalloc behind its back breaks the budget and
// fragments the pool), or a latency-critical serving loop where cudaMalloc / cudaFree
// would add their implicit device synchronisation and unbounded latency.  The plan (its
// compacted weights) must still have been created beforehand.

namespace {

constexpr size_t kNoAllocScratchBytes = 16u << 20;  // 16 MiB, held by every GPU that loads the library

__device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_noalloc_mu;
std::map<int, unsigned char*> g_noalloc_addr;  // device ordinal -> device address of the array

void noalloc_forget_device(int device) {
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  g_noalloc_addr.erase(device);
}

// Looks up (once per device, with that device current) the device address of the
// scratch array; host code cannot use the symbol itself as a device pointer.  The cached
// address is dropped whenever a plan is created on the device (dfs_plan_create), because
// a device reset (cudaDeviceReset) reloads the module, possibly at another address, and
// invalidates every plan made before it: any plan a later call can use was created after
// the reset, and its creation cleared the entry.
dfs_status noalloc_scratch(int device, unsigned char** out) {
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  auto it = g_noalloc_addr.find(device);
  if (it != g_noalloc_addr.end()) {
    *out = it->second;
    return DFS_OK;
  }
  void* p = nullptr;
  cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (e != cudaSuccess || p == nullptr)
    return fail(DFS_ECUDA, "cudaGetSymbolAddress(scratch) failed: %s", cudaGetErrorString(e));
  g_noalloc_addr[device] = static_cast<unsigned char*>(p);
  *out = static_cast<unsigned char*>(p);
  return DFS_OK;
}

dfs_status noalloc_forward(dfs_plan* P, int s, int l, const bf16* x, const bf16* t_emb, bf16* out,
                           cudaStream_t st) {
  const dfs_config& c = P->cfg;
  const int d = c.dim, dh = c.head_dim, N = P->N;
  StepLayer& S = P->sl[s * P->L + l];
  const LayerConst& C = P->lc[l];
  if (!P->block_gate[static_cast<size_t>(s) * P->L + l]) {
    DFS_CK(cudaMemcpyAsync(out, x, sizeof(bf16) * N * d, cudaMemcpyDeviceToDevice, st));
    return DFS_OK;
  }
  const long long hd = static_cast<long long>(S.h_s) * dh, hcd = static_cast<long long>(S.hc) * dh;
  const long long fs = S.f_s, vt_ld = round_up(N, 64);
  // carve the scratch array (256-byte aligned pieces)
  long long off = 0;
  auto take = [&](long long bytes) {
    const long long at = off;
    off += round_up(bytes, 256);
    return at;
  };
  const long long o_mod = take(6LL * d * 4), o_xm = take(2LL * N * d), o_qk = take(2LL * N * 2 * hd),
                  o_vt = take(2LL * hd * vt_ld), o_attn = take(2LL * N * std::max(hd, hcd)),
                  o_x1 = take(4LL * N * d), o_h = take(2LL * N * round_up(fs, 64)), o_qc = take(2LL * N * hcd);
  if (off > static_cast<long long>(kNoAllocScratchBytes))
    return fail(DFS_EUNSUPPORTED,
                "this (step, layer) needs %lld bytes of scratch; the allocation-free forward has %zu",
                off, kNoAllocScratchBytes);
  int dev = 0;
  DFS_CK(cudaGetDevice(&dev));
  if (dev != P->device)
    return fail(DFS_EINVAL, "the current device (%d) is not the plan's device (%d)", dev, P->device);
  unsigned char* base = nullptr;
  dfs_status e = noalloc_scratch(dev, &base);
  if (e) return e;
  float* mod = reinterpret_cast<float*>(base + o_mod);
  bf16* xm = reinterpret_cast<bf16*>(base + o_xm);
  bf16* qk = reinterpret_cast<bf16*>(base + o_qk);
  bf16* vt = reinterpret_cast<bf16*>(base + o_vt);
  bf16* attn = reinterpret_cast<bf16*>(base + o_attn);
  float* x1 = reinterpret_cast<float*>(base + o_x1);
  bf16* h = reinterpret_cast<bf16*>(base + o_h);
  bf16* qc = reinterpret_cast<bf16*>(base + o_qc);
  // Every scratch element a kernel reads is written earlier in this call, so nothing
  // has to be cleared between calls.

  DFS_CK(dfs::launch_modulation(mod, P->w_t, P->b_t, C.emod, t_emb, 6 * d, d, st));
  DFS_CK(dfs::launch_row_norm(xm, x, 0, N, d, mod + d, 1.f, mod, c.ln_eps, st));
  if (hd > 0) {
    dfs::GemmArgs g = S.g_qkv;
    if (!make_map(&g.tma_a, xm, d, N, d, 64, 128)) return fail(DFS_ECUDA, "tensor map (QKV) failed");
    g.out = qk; g.out_t = vt; g.ldt = vt_ld;
    DFS_CK(dfs::launch_gemm(g, P->num_sms, st));
    DFS_CK(dfs::launch_qk_norm_rope(qk, 2 * hd, N, static_cast<int>(hd), static_cast<int>(hd), S.P[2].p,
                                    S.P[3].p, dh, c.qk_norm_mode, c.ln_eps, &P->rope, st));
    dfs::AttnArgs a = S.a_self;
    if (!make_map(&a.tma_q, qk, 2 * hd, N, 2 * hd, 64, 128) || !make_map(&a.tma_k, qk, 2 * hd, N, 2 * hd, 64, 64) ||
        !make_map(&a.tma_vt, vt, N, hd, vt_ld, 64, dh / 2))
      return fail(DFS_ECUDA, "tensor map (attention) failed");
    a.out = attn;
    DFS_CK(dfs::launch_attention(a, dh, st));
    dfs::GemmArgs o = S.g_o;
    if (!make_map(&o.tma_a, attn, hd, N, hd, 64, 128)) return fail(DFS_ECUDA, "tensor map (O) failed");
    o.out = x1; o.res = x; o.gate = mod + 2 * d; o.out_tma = 0;
    DFS_CK(dfs::launch_gemm(o, P->num_sms, st));
  } else {
    DFS_CK(dfs::launch_bias_residual(x1, 1, x, 0, mod + 2 * d, C.bo, N, d, st));
  }
  if (c.has_cross) {
    DFS_CK(dfs::launch_row_norm(xm, x1, 1, N, d, C.cln_w, 0.f, C.cln_b, c.ln_eps, st));
    if (hcd > 0) {
      dfs::GemmArgs q = S.g_cq;
      if (!make_map(&q.tma_a, xm, d, N, d, 64, 128)) return fail(DFS_ECUDA, "tensor map (cross q) failed");
      q.out = qc;
      DFS_CK(dfs::launch_gemm(q, P->num_sms, st));
      DFS_CK(dfs::launch_qk_norm_rope(qc, hcd, N, static_cast<int>(hcd), 0, S.P[12].p, nullptr, dh,
                                      c.qk_norm_mode, c.ln_eps, nullptr, st));
      dfs::AttnArgs a = S.a_cross;
      if (!make_map(&a.tma_q, qc, hcd, N, hcd, 64, 128)) return fail(DFS_ECUDA, "tensor map (cross attn) failed");
      a.out = attn;
      DFS_CK(dfs::launch_attention(a, dh, st));
      dfs::GemmArgs o = S.g_co;
      if (!make_map(&o.tma_a, attn, hcd, N, hcd, 64, 128)) return fail(DFS_ECUDA, "tensor map (cross o) failed");
      o.out = x1; o.res = x1; o.out_tma = 0;
      DFS_CK(dfs::launch_gemm(o, P->num_sms, st));
    } else {
      DFS_CK(dfs::launch_bias_residual(x1, 1, x1, 1, nullptr, C.cbo, N, d, st));
    }
  }
  DFS_CK(dfs::launch_row_norm(xm, x1, 1, N, d, mod + 4 * d, 1.f, mod + 3 * d, c.ln_eps, st));
  if (fs > 0) {
    // union engine: FFN panels into the plan's scratch (allocated with the plan)
    dfs_status eg = union_ffn_gather(P, S, l, st, false);
    if (eg) return eg;
    dfs::GemmArgs u = S.g_up;
    if (!make_map(&u.tma_a, xm, d, N, d, 64, 128)) return fail(DFS_ECUDA, "tensor map (up) failed");
    u.out = h;
    DFS_CK(dfs::launch_gemm(u, P->num_sms, st));
    dfs::GemmArgs dn = S.g_down;
    if (!make_map(&dn.tma_a, h, fs, N, round_up(fs, 64), 64, 128)) return fail(DFS_ECUDA, "tensor map (down) failed");
    dn.out = out; dn.res = x1; dn.gate = mod + 5 * d;
    DFS_CK(dfs::launch_gemm(dn, P->num_sms, st));
  } else {
    DFS_CK(dfs::launch_bias_residual(out, 0, x1, 1, mod + 5 * d, C.bdown, N, d, st));
  }
  return DFS_OK;
}

}  // namespace

extern "C" dfs_status dfs_block_forward_noalloc(dfs_plan* plan, int step, int layer, const void* x,
                                                const void* t_emb, void* out, void* stream) {
  dfs_status e = check_forward_args(plan, step, layer, x, t_emb, out);
  if (e) return e;
  return noalloc_forward(plan, step, layer, static_cast<const bf16*>(x), static_cast<const bf16*>(t_emb),
                         static_cast<bf16*>(out), static_cast<cudaStream_t>(stream));
}
