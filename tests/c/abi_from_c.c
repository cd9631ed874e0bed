/* Calls libhdl through its C ABI from plain C (no Python, no torch): a small
 * re-scoring + selection problem with cudaMalloc'd buffers.  Inputs are read
 * from a binary file written by the test (bf16 bits of H_orig, H_hind, W,
 * int32 targets, int64 root offsets); outputs are written to another file.
 *   abi_from_c <in.bin> <out.bin> N d V R k
 * Exit status 0 on success; the test compares the outputs with the Python
 * binding's. */
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>

#include "hdl.h"

#define CHECK(x)                                                       \
  do {                                                                 \
    if ((x) != cudaSuccess) {                                          \
      fprintf(stderr, "CUDA error at %s:%d\n", __FILE__, __LINE__);    \
      return 2;                                                        \
    }                                                                  \
  } while (0)

static void* upload(FILE* f, size_t bytes) {
  void* host = malloc(bytes ? bytes : 1);
  void* dev = NULL;
  if (!host || fread(host, 1, bytes, f) != bytes) return NULL;
  if (cudaMalloc(&dev, bytes ? bytes : 1) != cudaSuccess) return NULL;
  if (cudaMemcpy(dev, host, bytes, cudaMemcpyHostToDevice) != cudaSuccess) return NULL;
  free(host);
  return dev;
}

int main(int argc, char** argv) {
  if (argc != 8) return 1;
  const int64_t N = atoll(argv[3]);
  const int32_t d = atoi(argv[4]), V = atoi(argv[5]), R = atoi(argv[6]), k = atoi(argv[7]);
  if (hdl_abi_version() != HDL_ABI_VERSION) return 3;
  FILE* in = fopen(argv[1], "rb");
  if (!in) return 1;
  void* h0 = upload(in, (size_t)N * d * 2);
  void* h1 = upload(in, (size_t)N * d * 2);
  void* w = upload(in, (size_t)V * d * 2);
  int32_t* y = (int32_t*)upload(in, (size_t)N * 4);
  int64_t* offs = (int64_t*)upload(in, (size_t)(R + 1) * 8);
  fclose(in);
  if (!h0 || !h1 || !w || !y || !offs) return 4;

  float *lp0, *lp1, *delta, *bd;
  int32_t *bp, *ns;
  void* ws;
  const size_t ws_bytes = hdl_rescore_workspace_bytes(N, d, V, HDL_BF16);
  CHECK(cudaMalloc((void**)&lp0, N * 4));
  CHECK(cudaMalloc((void**)&lp1, N * 4));
  CHECK(cudaMalloc((void**)&delta, N * 4));
  CHECK(cudaMalloc((void**)&bp, (size_t)R * k * 4));
  CHECK(cudaMalloc((void**)&ns, (size_t)R * 4));
  CHECK(cudaMalloc((void**)&bd, (size_t)R * k * 4));
  CHECK(cudaMalloc(&ws, ws_bytes));
  cudaStream_t st;
  CHECK(cudaStreamCreate(&st));

  /* an argument error is reported before anything runs */
  if (hdl_rescore(h0, h1, w, HDL_BF16, y, N, d + 1, V, lp0, lp1, delta, ws, ws_bytes, st) !=
      HDL_ERR_UNSUPPORTED)
    return 5;
  if (hdl_rescore(h0, h1, w, HDL_BF16, y, N, d, V, lp0, lp1, delta, ws, ws_bytes - 256, st) !=
      HDL_ERR_WORKSPACE)
    return 6;

  hdl_status s = hdl_rescore(h0, h1, w, HDL_BF16, y, N, d, V, lp0, lp1, delta, ws, ws_bytes, st);
  if (s != HDL_OK) return 10 + (int)s;
  s = hdl_select_branches(delta, NULL, N, offs, R, k, NULL, bp, ns, bd, st);
  if (s != HDL_OK) return 20 + (int)s;
  uint32_t raw = 0;
  s = hdl_device_status(ws, ws_bytes, st, &raw);
  if (s != HDL_OK) return 30 + (int)s;

  float* hl = (float*)malloc(N * 8);
  int32_t* hb = (int32_t*)malloc((size_t)R * k * 4);
  CHECK(cudaMemcpy(hl, lp0, N * 4, cudaMemcpyDeviceToHost));
  CHECK(cudaMemcpy(hl + N, lp1, N * 4, cudaMemcpyDeviceToHost));
  CHECK(cudaMemcpy(hb, bp, (size_t)R * k * 4, cudaMemcpyDeviceToHost));
  FILE* out = fopen(argv[2], "wb");
  if (!out) return 1;
  fwrite(hl, 4, (size_t)2 * N, out);
  fwrite(hb, 4, (size_t)R * k, out);
  fclose(out);
  printf("ok %s\n", hdl_status_string(s));
  return 0;
}
