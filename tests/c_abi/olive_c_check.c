/*
 * A C11 program that uses libolive.so through include/olive.h alone.
 *
 *   olive_c_check            host-side entry points: ABI version, status
 *                            strings, workspace sizes, argument validation
 *                            (no CUDA work is launched)
 *   olive_c_check splice     reads a batch from stdin (S V T_cap, then the
 *                            prefix offsets, prefix ids, continuation offsets
 *                            and continuation ids), runs olive_splice_pack on
 *                            the current CUDA device and prints n_rows, rows,
 *                            targets and the loss mask
 *   olive_c_check step IN OUT
 *                            one training step: reads a batch, the hidden
 *                            rows and W (bf16 bit patterns) from IN, runs
 *                            olive_splice_pack and olive_token_loss_fwd_bwd
 *                            (fp32 gradients, a workspace sized by
 *                            olive_workspace_size) and writes the status
 *                            word, logp [T], lse [T], the loss, d_hidden
 *                            [T, d] and d_W [V, d] to OUT
 */
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime.h>

#include "olive.h"

static int fails = 0;
#define CHECK(cond)                                              \
  do {                                                           \
    if (!(cond)) {                                               \
      fprintf(stderr, "check failed (line %d): %s\n", __LINE__, #cond); \
      ++fails;                                                   \
    }                                                            \
  } while (0)

static int host_checks(void) {
  CHECK(olive_abi_version() == OLIVE_ABI_VERSION);
  CHECK(strcmp(olive_status_string(OLIVE_OK), "ok") == 0);
  CHECK(strcmp(olive_status_string((olive_status)42), "unknown status") == 0);
  const size_t fwd = olive_workspace_size(OLIVE_OP_LOGPROB_FWD, 32768, 4096, 0, 151936, 0, 0);
  CHECK(fwd >= (size_t)2 * 32768 * 4096 && fwd % 256 == 0);
  CHECK(olive_workspace_size(OLIVE_OP_LOGPROB_FWD, 32768, 4095, 0, 151936, 0, 0) == 0);
  CHECK(olive_workspace_size(OLIVE_OP_LOSS_FWD_BWD, 32768, 4096, 0, 151936, 1, OLIVE_DTYPE_BF16) >
        olive_workspace_size(OLIVE_OP_LOSS_BWD, 32768, 4096, 0, 151936, 1, OLIVE_DTYPE_BF16) / 2);
  /* rejected before any CUDA call */
  CHECK(olive_token_logprob_fwd(NULL, NULL, NULL, NULL, NULL, 64, 64, 100, 1.0f, OLIVE_REDUCE_SUM,
                                NULL, NULL, NULL, NULL, 0, NULL, NULL) == OLIVE_ERR_INVALID_ARG);
  static unsigned char buf[4096] __attribute__((aligned(256)));
  void* p = buf;
  CHECK(olive_token_logprob_fwd(p, p, p, p, p, 64, 60, 100, 1.0f, OLIVE_REDUCE_SUM, p, p, p, p,
                                sizeof buf, p, NULL) == OLIVE_ERR_ALIGNMENT);
  CHECK(olive_token_divergence(p, p, 64, p, p, 64, p, p, 64, 100, 1.0f, 7, p, NULL, NULL, 0, p,
                               sizeof buf, p, NULL) == OLIVE_ERR_INVALID_ARG);
  CHECK(olive_splice_pack(p, p, p, p, 0, 10, 10, p, p, p, p, p, p, p, p, NULL) == OLIVE_ERR_SHAPE);
  printf("%s\n", fails ? "FAIL" : "ok");
  return fails ? 1 : 0;
}

static int* read_ints(int n) {
  int* a = (int*)malloc(sizeof(int) * (n > 0 ? n : 1));
  for (int i = 0; i < n; ++i)
    if (scanf("%d", &a[i]) != 1) exit(3);
  return a;
}

static void* dev_copy(const void* h, size_t bytes) {
  void* d = NULL;
  if (cudaMalloc(&d, bytes > 0 ? bytes : 4) != cudaSuccess) exit(4);
  if (bytes > 0 && cudaMemcpy(d, h, bytes, cudaMemcpyHostToDevice) != cudaSuccess) exit(4);
  return d;
}

static int splice(void) {
  int S, V, T_cap;
  if (scanf("%d %d %d", &S, &V, &T_cap) != 3) return 3;
  int* poff = read_ints(S + 1);
  int* pids = read_ints(poff[S]);
  int* coff = read_ints(S + 1);
  int* cids = read_ints(coff[S]);
  int32_t *ids, *targets, *cu, *cut, *rows, *n_rows, *st;
  uint8_t* mask;
  cudaMalloc((void**)&ids, 4 * T_cap);
  cudaMalloc((void**)&targets, 4 * T_cap);
  cudaMalloc((void**)&mask, T_cap);
  cudaMalloc((void**)&cu, 4 * (S + 1));
  cudaMalloc((void**)&cut, 4 * S);
  cudaMalloc((void**)&rows, 4 * T_cap);
  cudaMalloc((void**)&n_rows, 4);
  cudaMalloc((void**)&st, 4);
  cudaMemset(st, 0, 4);
  const olive_status s = olive_splice_pack(
      dev_copy(pids, 4 * (size_t)poff[S]), dev_copy(poff, 4 * (size_t)(S + 1)),
      dev_copy(cids, 4 * (size_t)coff[S]), dev_copy(coff, 4 * (size_t)(S + 1)), S, V, T_cap, ids,
      targets, mask, cu, cut, rows, n_rows, st, NULL);
  if (s != OLIVE_OK) {
    fprintf(stderr, "olive_splice_pack: %s\n", olive_status_string(s));
    return 5;
  }
  int n = 0, dst = 0;
  int* h_rows = (int*)malloc(4 * (size_t)T_cap);
  int* h_tg = (int*)malloc(4 * (size_t)T_cap);
  unsigned char* h_mask = (unsigned char*)malloc((size_t)T_cap);
  cudaMemcpy(&n, n_rows, 4, cudaMemcpyDeviceToHost);
  cudaMemcpy(&dst, st, 4, cudaMemcpyDeviceToHost);
  cudaMemcpy(h_rows, rows, 4 * (size_t)T_cap, cudaMemcpyDeviceToHost);
  cudaMemcpy(h_tg, targets, 4 * (size_t)T_cap, cudaMemcpyDeviceToHost);
  if (cudaMemcpy(h_mask, mask, (size_t)T_cap, cudaMemcpyDeviceToHost) != cudaSuccess) return 4;
  const int T = poff[S] + coff[S];
  printf("status %d\nn_rows %d\nrows", dst, n);
  for (int i = 0; i < n; ++i) printf(" %d", h_rows[i]);
  printf("\ntargets");
  for (int i = 0; i < T; ++i) printf(" %d", h_tg[i]);
  printf("\nmask");
  for (int i = 0; i < T; ++i) printf(" %d", h_mask[i]);
  printf("\n");
  return 0;
}

static int read_exact(FILE* f, void* dst, size_t bytes) {
  return fread(dst, 1, bytes, f) == bytes ? 0 : 1;
}

/* IN: int32 S, V, T, d; int32 prefix_off[S+1], cont_off[S+1]; int32
   prefix_ids, cont_ids; uint16 hidden[T*d], W[V*d] (bf16 bits). */
static int step(const char* in_path, const char* out_path) {
  FILE* f = fopen(in_path, "rb");
  if (!f) return 3;
  int32_t hdr[4];
  if (read_exact(f, hdr, sizeof hdr)) return 3;
  const int S = hdr[0], V = hdr[1], T = hdr[2], d = hdr[3];
  int32_t* poff = (int32_t*)malloc(4 * (size_t)(S + 1));
  int32_t* coff = (int32_t*)malloc(4 * (size_t)(S + 1));
  if (read_exact(f, poff, 4 * (size_t)(S + 1)) || read_exact(f, coff, 4 * (size_t)(S + 1))) return 3;
  int32_t* pids = (int32_t*)malloc(4 * (size_t)(poff[S] + 1));
  int32_t* cids = (int32_t*)malloc(4 * (size_t)(coff[S] + 1));
  if (read_exact(f, pids, 4 * (size_t)poff[S]) || read_exact(f, cids, 4 * (size_t)coff[S])) return 3;
  const size_t hb = 2 * (size_t)T * d, wb = 2 * (size_t)V * d;
  void* h_hidden = malloc(hb);
  void* h_W = malloc(wb);
  if (read_exact(f, h_hidden, hb) || read_exact(f, h_W, wb)) return 3;
  fclose(f);

  int32_t *ids, *targets, *cu, *cut, *rows, *n_rows, *st;
  uint8_t* mask;
  float *logp, *lse, *loss, *gl, *dh, *dw;
  void* ws;
  cudaMalloc((void**)&ids, 4 * (size_t)T);
  cudaMalloc((void**)&targets, 4 * (size_t)T);
  cudaMalloc((void**)&mask, (size_t)T);
  cudaMalloc((void**)&cu, 4 * (size_t)(S + 1));
  cudaMalloc((void**)&cut, 4 * (size_t)S);
  cudaMalloc((void**)&rows, 4 * (size_t)T);
  cudaMalloc((void**)&n_rows, 4);
  cudaMalloc((void**)&st, 4);
  cudaMemset(st, 0, 4);
  cudaMalloc((void**)&logp, 4 * (size_t)T);
  cudaMalloc((void**)&lse, 4 * (size_t)T);
  cudaMalloc((void**)&loss, 4);
  cudaMalloc((void**)&dh, 4 * (size_t)T * d);
  cudaMalloc((void**)&dw, 4 * (size_t)V * d);
  const float one = 1.0f;
  gl = (float*)dev_copy(&one, 4);
  const size_t ws_bytes = olive_workspace_size(OLIVE_OP_LOSS_FWD_BWD, T, d, 0, V, 1, OLIVE_DTYPE_F32);
  if (ws_bytes == 0 || cudaMalloc(&ws, ws_bytes) != cudaSuccess) return 4;
  void* d_hidden = dev_copy(h_hidden, hb);
  void* d_W = dev_copy(h_W, wb);

  olive_status s = olive_splice_pack(dev_copy(pids, 4 * (size_t)poff[S]), dev_copy(poff, 4 * (size_t)(S + 1)),
                                     dev_copy(cids, 4 * (size_t)coff[S]), dev_copy(coff, 4 * (size_t)(S + 1)),
                                     S, V, T, ids, targets, mask, cu, cut, rows, n_rows, st, NULL);
  if (s != OLIVE_OK) {
    fprintf(stderr, "olive_splice_pack: %s\n", olive_status_string(s));
    return 5;
  }
  s = olive_token_loss_fwd_bwd(d_hidden, d_W, targets, rows, n_rows, T, d, V, 1.0f, OLIVE_REDUCE_SUM, gl,
                               logp, lse, loss, dh, dw, OLIVE_DTYPE_F32, ws, ws_bytes, st, NULL);
  if (s != OLIVE_OK) {
    fprintf(stderr, "olive_token_loss_fwd_bwd: %s\n", olive_status_string(s));
    return 5;
  }
  if (cudaDeviceSynchronize() != cudaSuccess) return 4;

  int32_t dst = 0;
  float h_loss = 0.f;
  float* h_logp = (float*)malloc(4 * (size_t)T);
  float* h_lse = (float*)malloc(4 * (size_t)T);
  float* h_dh = (float*)malloc(4 * (size_t)T * d);
  float* h_dw = (float*)malloc(4 * (size_t)V * d);
  cudaMemcpy(&dst, st, 4, cudaMemcpyDeviceToHost);
  cudaMemcpy(&h_loss, loss, 4, cudaMemcpyDeviceToHost);
  cudaMemcpy(h_logp, logp, 4 * (size_t)T, cudaMemcpyDeviceToHost);
  cudaMemcpy(h_lse, lse, 4 * (size_t)T, cudaMemcpyDeviceToHost);
  cudaMemcpy(h_dh, dh, 4 * (size_t)T * d, cudaMemcpyDeviceToHost);
  if (cudaMemcpy(h_dw, dw, 4 * (size_t)V * d, cudaMemcpyDeviceToHost) != cudaSuccess) return 4;
  FILE* o = fopen(out_path, "wb");
  if (!o) return 3;
  fwrite(&dst, 4, 1, o);
  fwrite(h_logp, 4, (size_t)T, o);
  fwrite(h_lse, 4, (size_t)T, o);
  fwrite(&h_loss, 4, 1, o);
  fwrite(h_dh, 4, (size_t)T * d, o);
  fwrite(h_dw, 4, (size_t)V * d, o);
  fclose(o);
  return 0;
}

int main(int argc, char** argv) {
  if (argc > 1 && strcmp(argv[1], "splice") == 0) return splice();
  if (argc > 3 && strcmp(argv[1], "step") == 0) return step(argv[2], argv[3]);
  return host_checks();
}
