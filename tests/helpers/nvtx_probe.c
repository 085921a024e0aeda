/* nvtx_probe.c -- an NVTX injection library for the tests: NVTX loads it
 * through NVTX_INJECTION64_PATH and calls InitializeInjectionNvtx2, which
 * puts this file's handlers into the core-2 (domain) callback slots.  The
 * handlers record every domain created and every range pushed and popped;
 * the test reads the record through nvtx_probe_* (the same library, loaded
 * again by path, shares its state).  Host code only. */
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include <nvtx3/nvToolsExt.h>

#define MAX_EVENTS 4096

static char g_names[MAX_EVENTS][64];      /* "+name" on push, "-" on pop, "@domain" on create */
static int g_n = 0;
static int g_depth = 0, g_max_depth = 0;
static char g_domain[64];

static void record(char kind, const char *s) {
  if (g_n >= MAX_EVENTS) return;
  g_names[g_n][0] = kind;
  snprintf(g_names[g_n] + 1, 63, "%s", s ? s : "");
  ++g_n;
}

static nvtxDomainHandle_t probe_domain_create(const char *name) {
  snprintf(g_domain, sizeof g_domain, "%s", name ? name : "");
  record('@', name);
  return (nvtxDomainHandle_t)(uintptr_t)0x1000;
}

static int probe_push(nvtxDomainHandle_t d, const nvtxEventAttributes_t *a) {
  (void)d;
  record('+', (a && a->messageType == NVTX_MESSAGE_TYPE_ASCII) ? a->message.ascii : "?");
  if (++g_depth > g_max_depth) g_max_depth = g_depth;
  return g_depth - 1;
}

static int probe_pop(nvtxDomainHandle_t d) {
  (void)d;
  record('-', "");
  return --g_depth;
}

int InitializeInjectionNvtx2(NvtxGetExportTableFunc_t get_table) {
  const NvtxExportTableCallbacks *cb = (const NvtxExportTableCallbacks *)get_table(NVTX_ETID_CALLBACKS);
  if (!cb || !cb->GetModuleFunctionTable) return 0;
  NvtxFunctionTable table = 0;
  unsigned int size = 0;
  if (!cb->GetModuleFunctionTable(NVTX_CB_MODULE_CORE2, &table, &size) || !table) return 0;
  if (size <= NVTX_CBID_CORE2_DomainCreateA) return 0;
  *table[NVTX_CBID_CORE2_DomainRangePushEx] = (NvtxFunctionPointer)probe_push;
  *table[NVTX_CBID_CORE2_DomainRangePop] = (NvtxFunctionPointer)probe_pop;
  *table[NVTX_CBID_CORE2_DomainCreateA] = (NvtxFunctionPointer)probe_domain_create;
  return 1;
}

int nvtx_probe_count(void) { return g_n; }
int nvtx_probe_depth(void) { return g_depth; }
int nvtx_probe_max_depth(void) { return g_max_depth; }
const char *nvtx_probe_event(int i) { return (i >= 0 && i < g_n) ? g_names[i] : ""; }
const char *nvtx_probe_domain(void) { return g_domain; }
