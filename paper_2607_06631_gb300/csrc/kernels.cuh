// Argument structs and host launchers of every kernel of the library.  Launchers
// enqueue on the given stream and return the launch's cudaError_t.
#pragma once

#include "common.cuh"

namespace dfs {

// ------------------------------------------------------------------------ K4 GEMM
// D[M, N] = A[M, K] * B[N, K]^T with bf16 operands (both K-major), fp32 accumulation
// in TMEM, and one of three fused epilogues.
enum EpiMode : int {
  kEpiBias = 0,      // out = acc + bias (bf16); columns >= split go transposed to out_t
  kEpiBiasGelu = 1,  // out = GELU_tanh(acc + bias) (bf16)
  kEpiGatedRes = 2,  // out = res + gate * (acc + bias) (res / out bf16 or fp32)
};

// A CTA pair computes a kGemmTileM x kGemmBN output tile; each CTA stages kGemmBM rows of A
// and kGemmBRows rows of B per K block.
constexpr int kGemmBM = 128, kGemmTileM = 256, kGemmBN = 256, kGemmBRows = 128, kGemmBK = 64, kGemmStages = 6;
constexpr int kGemmThreads = 384;  // warpgroup 0: TMA, MMA, 2 idle warps; warpgroups 1-2: epilogue
// Register split (setmaxnreg) between warpgroup 0 and the two epilogue warpgroups; launch
// 384 x 168 registers; 128 x kGemmRegsControl + 256 x kGemmRegsEpilogue must not exceed it.
constexpr int kGemmRegsLaunch = 168, kGemmRegsControl = 72, kGemmRegsEpilogue = 216;
static_assert(128 * kGemmRegsControl + 256 * kGemmRegsEpilogue <= kGemmThreads * kGemmRegsLaunch, "GEMM register split exceeds the launch");
static_assert((kGemmRegsControl + 2 * kGemmRegsEpilogue) * 32 <= 16384, "GEMM register split exceeds a sub-partition");
constexpr int kGemmABytes = kGemmBM * kGemmBK * 2;
constexpr int kGemmBBytes = kGemmBRows * kGemmBK * 2;
constexpr int kGemmStageBytes = kGemmABytes + kGemmBBytes;
constexpr int kGemmStageOut = 32 * 32 * 4;  // one epilogue warp's 32 x 32 fp32 output chunk (TMA store)
constexpr int kGemmSmem = kGemmStages * kGemmStageBytes + 8 * kGemmStageOut + 1024 + 256;
static_assert(kGemmSmem <= 227 * 1024, "GEMM shared memory exceeds a CTA's maximum");

// How the B operand reaches shared memory.  kGatherNone reads B [N, K] as stored; the other
// modes read a union weight matrix (the parameters retained at any step, Sec. 4.3) through
// a per-step index map, one whole attention head at a time, so that the step's weights never
// exist as a separate copy:
//   kGatherRows    B rows (output features) in groups of b_group = head_dim rows (64 or 128):
//                  group g of the step is union row b_idx[g] * b_group of [N_union, K].
//   kGatherKCols   K block k (64 columns) of the step is union column b_idx[k] * 64 of
//                  [N, K_union] (head_dim a multiple of 64, so K has no tail).
// The map travels in the kernel parameters: indexed by tile / K-block counters it is read
// with uniform constant loads, so the TMA coordinates need no per-copy conversion from a
// per-thread register.  kGatherRows maps are padded (repeating the last entry) to
// n_tiles * 256 / b_group entries, so that every group a CTA stages, including groups past
// N, reads a valid row; those rows land in output columns that are never stored.
enum GatherMode : int { kGatherNone = 0, kGatherRows = 1, kGatherKCols = 2 };
constexpr int kGemmMapMax = 512;  // entries: 3 * 8192 / 64 row groups, 8192 / 64 K blocks

struct GemmArgs {
  CUtensorMap tma_a;  // A [M, K], box {64, 128}, 128 B swizzle
  CUtensorMap tma_b;  // B [N, K], box {64, 128}, 128 B swizzle (see GatherMode for the others)
  CUtensorMap tma_out;  // out_tma: fp32 output [M, ldo], box {32, 32}, 128 B swizzle
  int M, N, K;
  int mode;
  const bf16* bias;  // [N] or null
  void* out;
  long long ldo;
  int out_f32;
  int split;         // kEpiBias: first column written transposed (multiple of 32); N = none
  bf16* out_t;
  long long ldt;
  const void* res;   // kEpiGatedRes residual [M, ldr]
  long long ldr;
  int res_f32;
  const float* gate;  // [N] or null (gate = 1)
  int out_tma;        // kEpiGatedRes, fp32 output: full tiles stored by TMA from shared memory
  int epi_warps;      // epilogue warps per CTA: 8 (two per TMEM lane quarter, 128 columns each) or 4
  int group;          // M tiles per raster group (tiles of one group sweep N together; odd groups
                      // sweep N backwards, so a group starts on the B bands the previous one ended on)
  int b_gather;       // GatherMode
  int b_group;        // kGatherRows: rows per group (64 or 128)
  unsigned short b_idx[kGemmMapMax];  // index map of the gather (see GatherMode)
  int* err;
};

cudaError_t launch_gemm(const GemmArgs& a, int num_sms, cudaStream_t s);
// M tiles per raster group for a reduction length K: 16 up to K = 6144, 8 beyond.  A group's
// A bands (256 rows x K each) stay in L2 while its tiles sweep N; with the long reductions of
// the FFN down projection (K = f_s up to 13824, 7 MB per band) 16 bands crowd out the B bands
// that the concurrent tiles share.  Measured on the Wan-14B-shaped down projections (GB300,
// serpentine order): groups of 8 ran 4% faster than 16 at 75600 tokens and 1.5% at 32760;
// 4, 6, 12 and 24 were slower; for K = 5120 (QKV, FFN up) 16 was fastest.
inline int gemm_group(int K) { return K > 6144 ? 8 : 16; }
// Epilogue warps per CTA for a reduction length K: with short reductions (K <= 2048, e.g. the
// Wan-1.3B-shaped projections at K = 1536) a tile's main loop is shorter than its epilogue,
// which 8 warps run in about half the time; with long ones 4 warps leave more of the memory
// system to the main loop.
inline int gemm_epilogue_warps(int K) { return K <= 2048 ? 8 : 4; }
cudaError_t gemm_prepare();  // opts the kernel into its shared-memory size

// ------------------------------------------------------------------------ K5 attention
// O[q, h*DH : (h+1)*DH] = softmax(Q_h K_h^T / sqrt(DH)) V_h for the retained heads.
struct AttnArgs {
  CUtensorMap tma_q;   // over the Q source, box {64, 128}
  CUtensorMap tma_k;   // over the K source, box {64, 64} (one CTA's half of a 128-key tile)
  CUtensorMap tma_vt;  // over V^T [heads*DH, n_kv], box {64, DH/2} (one CTA's half)
  int n_q, n_kv, n_heads;
  int q_col0, k_col0;  // column of head 0 in the Q / K sources
  bf16* out;           // [n_q, ldo]
  long long ldo;
  float scale_log2;    // log2(e) / sqrt(DH)
  int* err;
};

cudaError_t launch_attention(const AttnArgs& a, int head_dim, cudaStream_t s);
cudaError_t attention_prepare();

// ------------------------------------------------------------------------ memory-bound kernels

// Streaming multiprocessors of the current device (queried once per device, then cached).
int current_device_sms();

// K1: dst[i, :] = src[rows[i], :] for i < n_rows (cols elements, multiple of 8).
cudaError_t launch_gather_rows(bf16* dst, long long ld_dst, const bf16* src, long long ld_src,
                               const int* rows, int n_rows, int cols, cudaStream_t s);
// K1: dst[r, 8j : 8j+8] = src[r, 8*seg[j] : 8*seg[j]+8] for r < n_rows, j < n_seg.
cudaError_t launch_gather_segs(bf16* dst, long long ld_dst, const bf16* src, long long ld_src,
                               const int* seg, int n_seg, int n_rows, cudaStream_t s);

// K6: out[r] = sum_c W[r, c] t[c] + b[r] (+ e[r]) for r < rows; W bf16 [rows, cols].
cudaError_t launch_modulation(float* out, const bf16* W, const bf16* b, const bf16* e,
                              const bf16* t, int rows, int cols, cudaStream_t s);
// out[i] = base[i] + e[i] (e bf16), i < n.
cudaError_t launch_add_table(float* out, const float* base, const bf16* e, int n, cudaStream_t s);

// K2 / K7: y = (x - mean) * rstd * (mul_bias + mul[c]) + add[c], per row of `cols`;
// x bf16 or fp32, y bf16.  mul / add fp32.
cudaError_t launch_row_norm(bf16* y, const void* x, int x_f32, int rows, int cols, const float* mul,
                            float mul_bias, const float* add, float eps, cudaStream_t s);

// K3: in-place QK RMSNorm (+ 3D RoPE) on a row-major bf16 buffer: per row, channels
// [0, nq) use gamma_q and [nq, nq + nk) use gamma_k; each part normalised on its own
// (mode 0) or per head (mode 1); RoPE when rope_cos != null.
struct RopeTables {
  const float* cos_t; const float* sin_t;  // [G_t][p_t]
  const float* cos_h; const float* sin_h;  // [G_h][p_h]
  const float* cos_w; const float* sin_w;  // [G_w][p_w]
  int grid_h, grid_w, p_t, p_h, p_w;
};
cudaError_t launch_qk_norm_rope(bf16* buf, long long ld, int rows, int nq, int nk, const bf16* gamma_q,
                                const bf16* gamma_k, int head_dim, int mode, float eps,
                                const RopeTables* rope, cudaStream_t s);

// out[r, c] = res[r, c] + (gate ? gate[c] : 1) * bias[c]; res / out bf16 or fp32 (may alias).
cudaError_t launch_bias_residual(void* out, int out_f32, const void* res, int res_f32, const float* gate,
                                 const bf16* bias, int rows, int cols, cudaStream_t s);

// out[i] = float(in[i]), i < n.
cudaError_t launch_to_f32(float* out, const bf16* in, int n, cudaStream_t s);

// Waits (bounded) on an mbarrier that nothing completes; sets *err to kErrTimeout.
cudaError_t launch_wait_selftest(int* err, cudaStream_t s);

// Model around the blocks (model.cu).
// e[i] = cos(t w_i), e[dim/2 + i] = sin(t w_i), w_i = 10000^(-i / (dim/2)); e fp32 [dim].
cudaError_t launch_timestep_freq(float* e, double t, int dim, cudaStream_t s);
// out[r] = sum_c W[r, c] f(in[c]) + b[r] for r < rows, f = SiLU when silu_in, else identity;
// W bf16 [rows, cols] (cols % 8 == 0), in fp32 [cols]; out_f32 / out_bf16 may be null.
cudaError_t launch_gemv(float* out_f32, bf16* out_bf16, const bf16* W, const bf16* b, const float* in, int rows,
                        int cols, int silu_in, cudaStream_t s);
// tok[n, 4c + 2dy + dx] = lat[c, f, 2y + dy, 2x + dx], n = (f gh + y) gw + x; lat [C, F, 2gh, 2gw].
cudaError_t launch_patchify(bf16* tok, const bf16* lat, int C, int F, int gh, int gw, cudaStream_t s);
// out[c, f, 2y + dy, 2x + dx] = (base ? base[same] : 0) + dt * tok[n, 4c + 2dy + dx] (out may alias base).
cudaError_t launch_unpatchify(bf16* out, const bf16* base, const bf16* tok, float dt, int C, int F, int gh, int gw,
                              cudaStream_t s);

// K8: x = x + dt * v (bf16, n elements, n % 8 == 0).
cudaError_t launch_euler(bf16* x, const bf16* v, float dt, long long n, cudaStream_t s);

}  // namespace dfs
