/* A minimal NVTX tool for tests/test_nvtx_ranges.py: loaded by the NVTX v3 headers of a process whose
 * NVTX_INJECTION64_PATH names this library, it writes one line per range push ("push <name>") and pop ("pop")
 * to the file named by MIKV_NVTX_LOG. Written against the injection interface declared in the CUDA toolkit's
 * nvtx3 headers (callbacks export table, core module). Test infrastructure only. */
#define NVTX_NO_IMPL
#include <nvtx3/nvToolsExt.h>
#include <stdio.h>
#include <stdlib.h>

static FILE* out;

static int push_a(const char* name) {
  fprintf(out, "push %s\n", name);
  fflush(out);
  return 0;
}

static int pop(void) {
  fprintf(out, "pop\n");
  fflush(out);
  return 0;
}

int InitializeInjectionNvtx2(NvtxGetExportTableFunc_t get) {
  const NvtxExportTableCallbacks* cb = (const NvtxExportTableCallbacks*)get(NVTX_ETID_CALLBACKS);
  NvtxFunctionTable table = 0;
  unsigned int n = 0;
  const char* path = getenv("MIKV_NVTX_LOG");
  if (!cb || !path || !cb->GetModuleFunctionTable(NVTX_CB_MODULE_CORE, &table, &n) || n <= NVTX_CBID_CORE_RangePop)
    return 0;
  out = fopen(path, "w");
  if (!out) return 0;
  *table[NVTX_CBID_CORE_RangePushA] = (NvtxFunctionPointer)push_a;
  *table[NVTX_CBID_CORE_RangePop] = (NvtxFunctionPointer)pop;
  return 1;
}
