/*
 * block_forward.c - one pruned-block forward through the C ABI (include/dfs.h) from plain C,
 * with no Python or torch: device memory comes from the CUDA runtime, the plan and the
 * forward from libdfs.so.
 *
 * Usage: block_forward <dir> <step>
 *   <dir>/config.txt   dim n_heads head_dim ffn_dim n_layers(=1) n_steps grid_t grid_h grid_w
 *   <dir>/<name>.bin   raw bf16 bits (uint16, row-major) of w_t, b_t, x, t_emb ([n_steps, dim])
 *                      and of the 15 layer-0 tensors wq .. e_mod (dfs_layer_weights order)
 *   <dir>/block_gate.bin, head_gate.bin, ffn_gate.bin   uint8 gates (dfs_masks layouts)
 * Writes <dir>/out.bin: the block output [N, dim] (bf16 bits) at MoM step <step>.
 * Build: nvcc -O2 -I include block_forward.c -L <lib dir> -ldfs -lcudart -o block_forward
 */
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime_api.h>

#include "dfs.h"

static void* read_file(const char* dir, const char* name, size_t* bytes) {
  char path[4096];
  snprintf(path, sizeof(path), "%s/%s.bin", dir, name);
  FILE* f = fopen(path, "rb");
  if (!f) return NULL;
  fseek(f, 0, SEEK_END);
  long n = ftell(f);
  fseek(f, 0, SEEK_SET);
  void* buf = malloc(n > 0 ? (size_t)n : 1);
  if (buf && n > 0 && fread(buf, 1, (size_t)n, f) != (size_t)n) {
    free(buf);
    buf = NULL;
  }
  fclose(f);
  *bytes = (size_t)n;
  return buf;
}

/* A device copy of <dir>/<name>.bin (cudaMalloc'd, so 256-byte aligned). */
static void* upload(const char* dir, const char* name, size_t* bytes) {
  size_t n = 0;
  void* host = read_file(dir, name, &n);
  void* dev = NULL;
  if (!host) {
    fprintf(stderr, "cannot read %s/%s.bin\n", dir, name);
    return NULL;
  }
  if (cudaMalloc(&dev, n) != cudaSuccess || cudaMemcpy(dev, host, n, cudaMemcpyHostToDevice) != cudaSuccess) {
    fprintf(stderr, "device copy of %s failed\n", name);
    dev = NULL;
  }
  free(host);
  if (bytes) *bytes = n;
  return dev;
}

int main(int argc, char** argv) {
  if (argc != 3) {
    fprintf(stderr, "usage: %s <dir> <step>\n", argv[0]);
    return 2;
  }
  const char* dir = argv[1];
  const int step = atoi(argv[2]);
  char path[4096];
  snprintf(path, sizeof(path), "%s/config.txt", dir);
  FILE* f = fopen(path, "r");
  dfs_config c;
  memset(&c, 0, sizeof(c));
  if (!f || fscanf(f, "%d %d %d %d %d %d %d %d %d", &c.dim, &c.n_heads, &c.head_dim, &c.ffn_dim, &c.n_layers,
                   &c.n_steps, &c.grid_t, &c.grid_h, &c.grid_w) != 9) {
    fprintf(stderr, "cannot read %s\n", path);
    return 2;
  }
  fclose(f);
  c.ffn_chunk = 8;
  c.ln_eps = 1e-6f;
  c.rope_theta = 1e4f;
  c.qk_norm_mode = 0;
  c.engine = DFS_ENGINE_COMPACTED;

  static const char* names[15] = {"wq", "bq", "wk", "bk", "wv", "bv", "wo", "bo", "gq", "gk",
                                  "w_up", "b_up", "w_down", "b_down", "e_mod"};
  const void* dev[15];
  for (int i = 0; i < 15; ++i)
    if (!(dev[i] = upload(dir, names[i], NULL))) return 1;
  dfs_layer_weights lw;
  memset(&lw, 0, sizeof(lw));
  lw.wq = dev[0]; lw.bq = dev[1]; lw.wk = dev[2]; lw.bk = dev[3]; lw.wv = dev[4]; lw.bv = dev[5];
  lw.wo = dev[6]; lw.bo = dev[7]; lw.gq = dev[8]; lw.gk = dev[9]; lw.w_up = dev[10]; lw.b_up = dev[11];
  lw.w_down = dev[12]; lw.b_down = dev[13]; lw.e_mod = dev[14];
  void* w_t = upload(dir, "w_t", NULL);
  void* b_t = upload(dir, "b_t", NULL);
  size_t xbytes = 0;
  void* x = upload(dir, "x", &xbytes);
  void* t_emb = upload(dir, "t_emb", NULL);
  if (!w_t || !b_t || !x || !t_emb) return 1;

  size_t nb = 0;
  dfs_masks m;
  m.block_gate = (const uint8_t*)read_file(dir, "block_gate", &nb);
  m.head_gate = (const uint8_t*)read_file(dir, "head_gate", &nb);
  m.ffn_gate = (const uint8_t*)read_file(dir, "ffn_gate", &nb);
  m.xhead_gate = NULL;
  if (!m.block_gate || !m.head_gate || !m.ffn_gate) {
    fprintf(stderr, "cannot read the gates\n");
    return 1;
  }

  dfs_plan* plan = NULL;
  if (dfs_plan_create(&c, &lw, w_t, b_t, &m, NULL, NULL, &plan) != DFS_OK) {
    fprintf(stderr, "dfs_plan_create: %s\n", dfs_last_error());
    return 1;
  }
  void* out = NULL;
  if (cudaMalloc(&out, xbytes) != cudaSuccess) return 1;
  const char* temb_s = (const char*)t_emb + (size_t)step * (size_t)c.dim * 2;
  if (dfs_block_forward(plan, step, x, temb_s, out, NULL) != DFS_OK || dfs_plan_sync(plan, NULL) != DFS_OK) {
    fprintf(stderr, "forward: %s\n", dfs_last_error());
    return 1;
  }
  void* host = malloc(xbytes);
  if (!host || cudaMemcpy(host, out, xbytes, cudaMemcpyDeviceToHost) != cudaSuccess) return 1;
  snprintf(path, sizeof(path), "%s/out.bin", dir);
  f = fopen(path, "wb");
  if (!f || fwrite(host, 1, xbytes, f) != xbytes) return 1;
  fclose(f);
  printf("block_forward ok: step %d, %zu bytes written\n", step, xbytes);
  dfs_plan_destroy(plan);
  return 0;
}
